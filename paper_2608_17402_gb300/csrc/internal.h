// internal.h -- host-side launch interface between the kernel files and api.cu.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace mv {

// Counts kernel launches made by this library (read by moevie_launch_count).
void count_launches(int n);

// Launches kern<<<grid, block, smem, s>>>(args...) with programmatic stream
// serialization, so that its launch overlaps the end of the previous kernel on s
// (every kernel of this library calls pdl_wait() before reading its inputs).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                       Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[1];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = at;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}
// The same for a cooperative launch (all CTAs co-resident; grid-wide barriers).
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl_coop(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem,
                            cudaStream_t s, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute at[2];
    at[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    at[0].val.programmaticStreamSerializationAllowed = 1;
    at[1].id = cudaLaunchAttributeCooperative;
    at[1].val.cooperative = 1;
    cfg.attrs = at;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<KArgs>(args)...);
}

// ----------------------------------------------------------------- router

// Error model of the fast logits used to decide when a token's selection must be
// re-decided with exact logits.  The fast logits are x . (hi + mid), two bf16 pieces of
// W_r = hi + mid + lo (lo, the last 8 significand bits, is left out), on the tensor
// cores with fp32 accumulation:
//   |s_fast[t, e] - s[t, e]| <= |x_t| (ROUTE_TAU_C 2^-24 (|W_r[:, e]| + |lo_e|) + |lo_e|).
// The |x_t| |lo_e| term bounds the left-out piece (Cauchy-Schwarz, rigorous); the first
// term is the accumulation error, whose constant is fixed by measurement (the tensor
// cores' accumulation order is undocumented).
constexpr float ROUTE_TAU_C = 128.0f;
// Extra allowance, in key units, for the fp32 evaluation of sigmoid(s) + b.
constexpr float ROUTE_KEY_SLACK = 2e-6f;

// Columns of the router logit buffer: E rounded up to 16 (rows stay 16-byte aligned).
inline int route_epad(int E) { return (E + 31) / 32 * 32; }
// Rows of each W_r piece: d rounded up to 64 (zero rows), so that no 64-wide K block
// of the router GEMM straddles two pieces.
inline int route_dpad(int d) { return (d + 63) / 64 * 64; }
// The router GEMM's B holds the two bf16 pieces hi, mid of W_r side by side along N
// ([d_pad][2 E_pad]: x is read once, the epilogue sums the pieces) when they fit one
// n-tile; otherwise one after another along K ([2][d_pad][E_pad], x read per piece).
inline bool route_concat(int E) { return 2 * route_epad(E) <= 256; }   // 256: largest MMA N

// W_r fp32 [d, E] -> the bf16 pieces hi = bf16(w), mid = bf16(w - hi) (W_r = hi + mid +
// lo exactly, lo = w - hi - mid; zero in the padding rows and columns), the transposed
// fp32 copy wrt [E][d_pad] (zero rows past d), and per-CTA partial sums of squares of
// W_r's columns and of lo's columns (wpart: two sets of route_split_parts(d) x E_pad
// floats; |W_r[:, e]| and |lo_e| are the square roots of their sums over the parts).
// It also writes each CTA's largest exponent field of each column (wexp:
// route_split_parts(d) x E_pad ints, at least 1), which sets the exact re-decision's
// accumulator window.  Also clears the fallback counter in st (may be NULL).
int route_split_parts(int d);
cudaError_t launch_route_split(const float* Wr, int d, int E, __nv_bfloat16* Wsplit, float* wrt,
                               float* wpart, int32_t* wexp, DevStatus* st, cudaStream_t s);

// Splits of K for the router GEMM: enough CTA-pair work items for about
// ROUTE_SPLIT_TARGET items (ROUTE_SPLIT_TARGET_CONCAT with the pieces side by side),
// at most ROUTE_MAX_KSPLIT, at least three K blocks each.
// Depends on the sizes only (the workspace size uses it).
constexpr int ROUTE_SPLIT_TARGET = 76;
constexpr int ROUTE_SPLIT_TARGET_CONCAT = 64;   // the same with the pieces side by side (E <= 128)
constexpr int ROUTE_MAX_KSPLIT = 16;
int route_ksplit(int64_t T, int d, int E);
// Rows of partial-logit storage: an upper bound of route_ksplit(T) * T that is
// monotone in T (ROUTE_MAX_KSPLIT T, and (ROUTE_SPLIT_TARGET + m-tiles x n-tiles) x 256).
int64_t route_logits_rows(int64_t T, int d, int E);

// out = the sum over the nparts partial logit arrays (n floats each, part_stride apart).
cudaError_t launch_route_sum_parts(const float* logits, int64_t part_stride, int nparts, int64_t n,
                                   float* out, cudaStream_t s);

// Keys, warp top-k with a certificate, gates; uncertified tokens are listed in
// fb_tokens and re-decided by a second kernel with exact logits (integer long
// accumulator) of the experts near their boundary.  wnorm: |W_r[:, e]| [E] then |lo_e|
// [E] (the error model above); wexp: the split kernel's largest exponent fields.  The
// top-k kernel also clears zero[0, zero_n) (16-byte aligned, zero_n % 4 == 0; NULL:
// nothing).  logits: nparts partial arrays [T][ld] (part_stride floats apart); part 0 is
// overwritten with the sum for uncertified tokens.
cudaError_t launch_route_select(const __nv_bfloat16* x, const float* wrt, const float* b,
                                float* logits, int ld, int nparts, int64_t part_stride,
                                const float* wnorm, const int32_t* wexp, int T, int d, int E, int k,
                                int32_t* idx, float* gate, int32_t* fb_tokens, float* xnorm,
                                DevStatus* st, int num_sms, cudaStream_t s, float* zero = nullptr,
                                int64_t zero_n = 0);

// ---------------------------------------------------------------- permute

constexpr int PERM_CHUNK_MAX = 4096;   // flat slots per CTA of the histogram / scatter

// Slots per CTA for n flat slots on num_sms SMs (multiple of 256, <= PERM_CHUNK_MAX).
int perm_chunk(int64_t n, int num_sms);

// Always-on groups appended to the permuted rows: S groups E .. E + S - 1 of T rows
// each (row n_slots + c T + t: token t, gate lambda).
struct SharedRows {
    int S;
    int64_t T;
    float lambda;
};

// Stable expert-major order; also writes the m-tile table of the grouped GEMMs
// (tiles[i] = {expert, first row, rows, 0}, *n_tiles = their number), followed by the
// tiles and rows of the always-on groups `sh` describes (none when sh is null).
cudaError_t launch_permute(const int32_t* idx, int64_t n_slots, int k, int E, int bm, int chunk,
                           const float* gate_flat, int32_t* hist, int32_t* counts,
                           int32_t* offsets, int4* tiles, int32_t* n_tiles, int32_t* perm,
                           int32_t* inv, int32_t* row_tok, float* row_gate, DevStatus* st,
                           cudaStream_t s, const SharedRows* sh = nullptr);

// m-tile table of `bm`-row tiles from given segment offsets [G + 1].
cudaError_t launch_tile_table(const int32_t* offsets, int G, int bm, int4* tiles,
                              int32_t* n_tiles, cudaStream_t s);

// Band-ordered work items for the down-projection (see item_order_kernel).
constexpr int ITEM_MAX_BANDS = 16;
constexpr int ITEM_MAX_TILES = 24576;   // m-tiles one ordering pass holds in shared memory
cudaError_t launch_item_order(const int4* tiles, const int32_t* n_tiles, const int32_t* row_tok,
                              int64_t T, int nb, int n_ntiles, int gsz, int BN, int max_tiles,
                              int4* items, int32_t* n_items, cudaStream_t s);

// ----------------------------------------------------------- grouped GEMM

constexpr int GM_BM = 256;        // rows per m-tile: one CTA pair, 128 rows per CTA
constexpr int GM_HALF = 128;      // rows per CTA (tcgen05 M = 256 across the pair)
constexpr int GM_BK = 64;         // K per stage: 64 bf16 = one 128-byte swizzle row
constexpr int GM_STAGES_MAX = 7;   // operand ring depth (6 when the reduction staging is needed)
constexpr int GM_MAXBN = 256;     // largest N of one tcgen05.mma
constexpr int GM_EPI_WARPS = 8;   // two warps per TMEM lane quadrant, alternate 32-column chunks
constexpr int GM_WARP_MMA = GM_EPI_WARPS;        // TMEM allocation + tcgen05.mma issue
constexpr int GM_WARP_LOAD = GM_EPI_WARPS + 1;   // TMA loads of B (and of contiguous A)
constexpr int GM_GATHER_WARPS = 8;               // token-gather warps
constexpr int GM_WARP_GATHER = GM_EPI_WARPS + 2; // first token-gather warp
constexpr int GM_WARP_FWD = GM_WARP_GATHER + GM_GATHER_WARPS;   // publishes gathered stages
constexpr int GM_THREADS = (GM_WARP_FWD + 1) * 32;
// Each gather thread copies one 16-byte chunk of GM_GATHER_ROWS rows per stage, rows
// GM_GATHER_RSTEP apart (8 threads cover a row's 128 bytes).
constexpr int GM_GATHER_RSTEP = GM_GATHER_WARPS * 32 / 8;
constexpr int GM_GATHER_ROWS = 128 / GM_GATHER_RSTEP;
constexpr int GM_A_BYTES = GM_HALF * GM_BK * 2;           // one CTA's A rows per stage
constexpr int GM_B_BYTES = GM_BK * (GM_MAXBN / 2) * 2;    // one CTA's half of B per stage
constexpr int GM_STG_ROWS = 32;    // rows per warp in the reduction staging buffer (at most)
constexpr int GM_STG_LD = 36;      // floats per staged row: 32 values, the row's y offset, pad
constexpr int GM_OVERHEAD_BYTES = 1024 + 512;   // alignment, barriers / TMEM slot / flags / sink
// The y-accumulator epilogue (epi 2, EPI_ADD_F32) stages stg_rows (32 or 16) rows per warp
// and gives up operand stages for them: 32 rows -> 5 stages, 16 rows -> 6.  Other
// epilogues run 7 stages.
__host__ __device__ constexpr int gm_stg_bytes(int epi, int stg_rows) {
    return epi == 2 ? GM_EPI_WARPS * stg_rows * GM_STG_LD * 4 : 0;
}
__host__ __device__ constexpr int gm_stages(int epi, int stg_rows) {
    return epi == 2 ? (stg_rows > 16 ? 5 : 6) : 7;
}
__host__ __device__ constexpr int gm_smem_bytes(int epi, int stg_rows) {
    return gm_stages(epi, stg_rows) * (GM_A_BYTES + GM_B_BYTES) + gm_stg_bytes(epi, stg_rows) +
           GM_OVERHEAD_BYTES;
}
constexpr int GM_SMEM_BYTES_MAX = GM_STAGES_MAX * (GM_A_BYTES + GM_B_BYTES) + GM_OVERHEAD_BYTES;
static_assert(GM_SMEM_BYTES_MAX <= 232448 && gm_smem_bytes(2, 32) <= 232448 &&
                  gm_smem_bytes(2, 16) <= 232448,
              "shared memory of one CTA");
static_assert(3 * GM_STAGES_MAX + 5 <= 32, "barriers fit before the signal sink at +256 bytes");

inline int64_t max_mtiles(int64_t rows, int64_t groups) { return (rows + GM_BM - 1) / GM_BM + groups; }

enum Epilogue : int {
    EPI_GELU_BF16 = 0,   // out[r, n] = bf16(GELU(acc))
    EPI_STORE_BF16 = 1,  // out[r, n] = bf16(acc)
    EPI_ADD_F32 = 2,     // yacc[tok(r), n] += scale(r) * acc   (vector atomics)
    EPI_STORE_F32 = 3,   // yacc[tok(r), n]  = scale(r) * acc
    EPI_SWIGLU_BF16 = 5, // out[r, n] = bf16(SiLU(acc[gate n]) * acc[up n]): accumulator columns
                         //   0..127 from W1 (gate, the pair's first CTA's B half), 128..255 from
                         //   W3 (up, the second CTA's); 128 output columns per n-tile
    EPI_SUM2_F32 = 4,    // yacc[tok(r), n]  = scale(r) * (acc[n] + acc[n + N/2]), n < N/2
                         //   (two column groups summed; one n-tile)
    EPI_GELU2_BF16 = 6,  // out[r, n] = bf16(GELU(acc)), out2[r, n] = bf16(acc) (the pre-activation)
    EPI_DGELU_BF16 = 7,  // out[r, n] = bf16(scale(r) acc GELU'(u[r, n])), and the row dot
                         //   sum_n acc a[r, n] (a = GELU(u)) in partials dg_part[2 nt + half][r]
    EPI_DSWIGLU_BF16 = 8,// SwiGLU a = SiLU(u) v: out = du = bf16(scale acc v SiLU'(u)), out2 = dv =
                         //   bf16(scale acc SiLU(u)), and the row dot sum_n acc a as for EPI_DGELU_BF16
};
static_assert(EPI_ADD_F32 == 2, "gm_stages / gm_smem_bytes test the reduction epilogue by value");
// Epilogue classes of the grouped GEMM's kernel instances: bf16 outputs (GELU, SwiGLU,
// plain), fp32 stores (plain, two-group sums), fp32 reductions into the accumulator.
enum { ECLS_BF16 = 0, ECLS_F32 = 1, ECLS_ADD = 2 };

struct GemmArgs {
    CUtensorMap tmB;            // B = weights [G][K][N] bf16 (N contiguous), 3-D map {N, K, G}
    CUtensorMap tmB2;           // groups g >= g_split: B from this map, group g - g_split
    CUtensorMap tmB3;           // swiglu with groups g >= g_split: their gate (CTA rank 0) and
    CUtensorMap tmB4;           //   up (rank 1) weights, group g - g_split
    CUtensorMap tmA;            // A = rows [a_nrows][K_A] bf16, 2-D map {K_A, a_nrows}, box
                                // {64, 128}; used when A rows are contiguous (a_rows == nullptr)
    const __nv_bfloat16* A;     // A rows, for the token gather
    int64_t lda;
    const int32_t* a_rows;      // A row of GEMM row r: a_rows ? a_rows[r] / a_div : r (gather)
    int a_div;
    int a_kperiod;              // 0, or a multiple of 64: column of K index kk in A is kk % a_kperiod
    int64_t a_nrows;            // rows of A; a gathered row outside [0, a_nrows) is a device error
    int64_t m_total;            // GEMM rows that may be written
    const int4* tiles;          // m-tile table {g, row0, nrows, 0}; nullptr: one dense group;
                                // with item_table: work items {g, row0, nrows, n0}
    int item_table;             // tiles lists (m-tile, n-tile) items; *n_tiles_dev counts items
    int a_ident;                // gathered path with A row r = r (contiguous rows through cp.async)
    int stg_rows;               // EPI_ADD_F32: rows staged per warp and phase (32 or 16)
    const int32_t* n_tiles_dev; // number of entries of `tiles`
    int64_t max_mtiles;         // host bound on *n_tiles_dev
    int G, K, N, BN, n_ntiles, num_kb, nbox;
    int g_split;                // first group read through tmB2 (G when there is none)
    int swiglu;                 // EPI_SWIGLU_BF16: B half of CTA rank 1 from tmB2 (W3), same columns;
                                // groups g >= g_split from tmB3 (rank 0) and tmB4 (rank 1)
    int n_step;                 // output columns per n-tile (BN; BN / 2 with swiglu)
    int ksplit;                 // K is split into this many parts (work items), >= 1
    int64_t y_split_stride;     // fp32 outputs: split ks writes yacc + ks * y_split_stride
    int epi;
    __nv_bfloat16* out;         // EPI_*_BF16
    int64_t ldo;
    float* yacc;                // EPI_*_F32
    int64_t ldy;
    int64_t o_nrows;            // rows of yacc; tokens outside are a device error
    const int32_t* o_rows;      // output token of row r: o_rows ? o_rows[r] / o_div : r
    int o_div;
    const float* row_scale;     // scale(r) = row_scale ? row_scale[r] : scale
    float scale;
    float4* zero;               // dense A only: the otherwise idle gather warps clear zero[0, zero_n)
    int64_t zero_n;             //   (float4 elements), alongside the GEMM
    const __nv_bfloat16* nrm_x; // dense A only: the idle gather warps also write, for the rows of
    int64_t nrm_ld;             //   every n-tile-0 item, nrm_out[r] = |nrm_x[r, 0:nrm_cols]|
    int nrm_cols;               //   (nrm_cols % 8 == 0)
    float* nrm_out;
    const float* wn_part;       // dense A only: the idle gather warps also write, for each set
    int wn_nparts, wn_E, wn_Ep; //   q < wn_sets and e < wn_E, wn_out[q wn_E + e] =
    int wn_sets;                //   sqrt(sum_p wn_part[(q wn_nparts + p) wn_Ep + e])
    float* wn_out;              //   (the router's |W_r[:, e]| and |lo_e| from per-CTA partial sums)
    // Operand layouts and work items of the training path (all 0 on the forward):
    int b_kmajor;               // B stored K-major, W[G][N][K] (K contiguous): tmB is the 3-D map
                                //   {K, N, G} with box {64, BN/2, 1}; the shared tile holds BN/2
                                //   rows of 128 bytes like A's
    int a_mn;                   // A stored M-major, A[K][M] (M contiguous): tmA is the 3-D map
                                //   {M, K, 1} with box {64, 64, 1}, two boxes per CTA and stage
    int wg_M;                   // item_table == 2: weight-gradient items {g, m0 | n0 << 16, kb0,
                                //   kb1} (absolute k-blocks of the rows both operands share);
                                //   output row of (g, m) is g wg_M + m, B's map has one group
    int a_neg_zero;             // gathered rows with a negative table entry are zero rows (padding)
    int o_neg_skip;             // fp32 outputs: rows with a negative output token are padding, skipped
    __nv_bfloat16* out2;        // EPI_GELU2_BF16: the pre-activation, laid out as out; with
    __nv_bfloat16* out3;        //   EPI_SWIGLU_BF16 (training instances): u in out2, v in out3;
                                //   EPI_DSWIGLU_BF16: dv in out2
    const __nv_bfloat16* epi_u; // EPI_DGELU_BF16 / EPI_DSWIGLU_BF16: pre-activations u (and v)
    const __nv_bfloat16* epi_v; //   and activations a of the GEMM rows, [m_total][ldo] bf16
    const __nv_bfloat16* epi_a;
    float* dg_part;             // EPI_D*_BF16: per-row partial dots, [2 n_ntiles][m_total] fp32 (or NULL: none)
    DevStatus* status;
    uint64_t limit_ns;
};

// Encodes the 3-D weight tensor map {N, K, G} for W[G][K][N] bf16.
bool make_weight_tmap(CUtensorMap* tm, const void* base, int64_t N, int64_t K, int64_t G);
// The same for a strided view: element (g, kk, n) at base + g * g_ld + kk * k_ld + n
// (strides in elements, multiples of 8).
bool make_weight_tmap_strided(CUtensorMap* tm, const void* base, int64_t N, int64_t K, int64_t G,
                              int64_t k_ld, int64_t g_ld);
// Encodes the 2-D row tensor map {cols, rows} of A[rows][cols] bf16 (row stride ld
// elements), box {64, GM_HALF}.
bool make_rows_tmap(CUtensorMap* tm, const void* base, int64_t cols, int64_t rows, int64_t ld);
// The 3-D map {K, N, G} of a K-major operand W[G][N][K] bf16 (row stride k_ld, group
// stride g_ld elements, multiples of 8), box {64, box_n, 1}.
bool make_kmajor_tmap(CUtensorMap* tm, const void* base, int64_t K, int64_t N, int64_t G, int64_t k_ld,
                      int64_t g_ld, int box_n);
// Picks BN (multiple of 32, <= 256) and the number of N tiles for width N.
void choose_bn(int N, int* BN, int* n_ntiles);
cudaError_t launch_grouped_gemm(const GemmArgs& a, int grid, cudaStream_t s);

// ------------------------------------------------------- training path

// k-blocks (of 64 rows) per weight-gradient work item at most.
constexpr int64_t BWD_KCH = 64;
// Set in a weight-gradient item's end k-block when its group has one chunk of K: the item
// is the only one writing its output tile, so the GEMM stores instead of adding.
constexpr int BWD_STORE_BIT = 1 << 30;
// Per token: sig[t k + j] = sigmoid(x_t . W_r[:, idx[t k + j]]) (fp32, from the transposed
// copy wrt [E][dp]) and gate = sig / sum_j sig (k <= 32).
cudaError_t launch_bwd_gates(const __nv_bfloat16* x, const float* wrt, int dp, const int32_t* idx, int64_t T,
                             int d, int E, int k, float* sig, float* gate, DevStatus* st, cudaStream_t s);
// poff[E + 1]: exclusive prefix of counts rounded up to multiples of 64 (E <= 1024).
cudaError_t launch_bwd_pad(const int32_t* counts, int E, int32_t* poff, cudaStream_t s);
// Padded rows: ptok / pgate of every padded row (-1 / 0 for padding) and the padded row
// of every routing slot (from the stable expert-major rows inv and offsets).
cudaError_t launch_bwd_rows(const int32_t* idx, const int32_t* inv, const int32_t* counts,
                            const int32_t* offsets, const int32_t* poff, const float* gate, int64_t n_slots,
                            int k, int E, int32_t* ptok, float* pgate, int32_t* slot_prow, cudaStream_t s);
// Weight-gradient work items (see bwd_items_kernel) and a bound on their number for
// groups holding `rows` rows in total.
int64_t bwd_max_items(int64_t rows, int G, int M, int N, int BN);
cudaError_t launch_bwd_items(const int32_t* koff, int G, int64_t K_rows, int M, int N, int BN,
                             int max_items, int4* items, int32_t* n_items, int32_t* gclear, DevStatus* st,
                             cudaStream_t s);
// Clears what the weight-gradient items will not write of out [G][M][ld] (fp32): the
// groups with gclear[g] set (no rows, or several chunks adding up), and the pad columns
// [N, ld) of the others.
cudaError_t launch_bwd_zero(const int32_t* gclear, int G, int M, int N, int64_t ld, float* out, int num_sms,
                            cudaStream_t s);
// xp[r] = x[ptok[r]], gdy[r] = pgate[r] dy[ptok[r]] over the poff[E] padded rows.
cudaError_t launch_bwd_gather(const __nv_bfloat16* x, const __nv_bfloat16* dy, const int32_t* ptok,
                              const float* pgate, const int32_t* poff, int E, int d, int64_t max_rows,
                              __nv_bfloat16* xp, __nv_bfloat16* gdy, cudaStream_t s);
// Router backward per token (Eqs. 4-5): ds, dx += ds W_r^T, ds into [T][Ep] bf16.
cudaError_t launch_bwd_router(const int32_t* idx, const float* sig, const float* gate, const int32_t* slot_prow,
                              const float* dg_part, int nparts, int64_t part_stride, const float* wrt, int dp,
                              int64_t T, int d, int E, int k, int Ep, float* dx, __nv_bfloat16* ds,
                              cudaStream_t s);
cudaError_t launch_bwd_copy(const float* src, int64_t ld_src, float* dst, int64_t rows, int64_t cols,
                            cudaStream_t s);

// ---------------------------------------- permute without a caller workspace

// moevie_permute_static keeps its scratch in one fixed device array (in permute.cu):
//   [0, 256)                 DevStatus (cleared by every call)
//   [256, 260)               number of m-tiles
//   [PERM_STATIC_HIST_OFF)   chunk histograms, <= PERM_STATIC_MAX_CHUNKS x 1024 int32
//   [PERM_STATIC_TILES_OFF)  m-tile table, <= max_mtiles(PERM_STATIC_MAX_SLOTS, 1024) int4
constexpr int64_t PERM_STATIC_MAX_SLOTS = int64_t(1) << 20;   // largest T * k
constexpr int PERM_STATIC_MAX_CHUNKS = 512;
constexpr size_t PERM_STATIC_NTILES_OFF = 256;
constexpr size_t PERM_STATIC_HIST_OFF = 512;
constexpr size_t PERM_STATIC_TILES_OFF =
    PERM_STATIC_HIST_OFF + size_t(4) * PERM_STATIC_MAX_CHUNKS * 1024;
constexpr size_t PERM_STATIC_SCRATCH_BYTES =
    PERM_STATIC_TILES_OFF + size_t(16) * ((PERM_STATIC_MAX_SLOTS + GM_BM - 1) / GM_BM + 1024);

static_assert((PERM_STATIC_MAX_SLOTS + PERM_STATIC_MAX_CHUNKS - 1) / PERM_STATIC_MAX_CHUNKS <=
                  PERM_CHUNK_MAX,
              "the largest permute must fit PERM_STATIC_MAX_CHUNKS chunks");

// Device address of that array on the current device.  The first call on a device
// looks the symbol up (cudaGetSymbolAddress, which may load the module); later calls
// return the cached address while the device's context is the one it was looked up in
// (after a device reset the next call looks it up again).  Thread-safe.
cudaError_t perm_static_scratch(unsigned char** out);
// The calling thread's current CUDA context (an opaque handle; nullptr when it cannot be
// read), for per-context caches of device-side objects.
void* current_context();

// ------------------------------------------------------------------- misc

cudaError_t launch_zero_f32(float* p, int64_t n, cudaStream_t s);
cudaError_t launch_f32_to_bf16(const float* src, __nv_bfloat16* dst, int64_t n, cudaStream_t s);
// Loss-free bias update (Eq. 9 z-score, rule 0; Eq. 8 sign, rule 1) from counts[E], E <= 1024.
cudaError_t launch_update_bias(const int32_t* counts, int E, float alpha, int rule, float* b,
                               DevStatus* st, cudaStream_t s);
// Rows of the shared expert folded into the grouped GEMMs as S always-on groups
// E .. E + S - 1 of T rows each, at rows base + c T + t (token t, gate lambda), and
// their m-tiles appended to the tile table (after the *n_tiles routed ones).
cudaError_t launch_shared_rows(int64_t T, int64_t base, int S, int E, float lambda,
                               int32_t* row_tok, float* row_gate, int4* tiles, int32_t* n_tiles,
                               int64_t max_routed, DevStatus* st, cudaStream_t s);
cudaError_t launch_combine(const __nv_bfloat16* rows, const int32_t* inv, const float* gate,
                           const __nv_bfloat16* shared, float lambda, int64_t T, int k, int d,
                           __nv_bfloat16* y, cudaStream_t s);
cudaError_t launch_wait_probe(DevStatus* st, uint64_t limit_ns, cudaStream_t s);

}  // namespace mv
