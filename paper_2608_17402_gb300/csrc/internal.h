// internal.h -- host-side launch interface between the kernel files and api.cu.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <stdint.h>

#include "common.cuh"

namespace mv {

// Counts kernel launches made by this library (read by moevie_launch_count).
void count_launches(int n);

// ----------------------------------------------------------------- router

// Relative bound on the fp32 logit error used to decide when a token's selection
// must be re-decided with exact logits: |s_fast - s| <= TAU_C * 2^-24 * |x_t| * max_e |W_r[:, e]|.
constexpr float ROUTE_TAU_C = 64.0f;
// Extra allowance, in key units, for the fp32 evaluation of sigmoid(s) + b.
constexpr float ROUTE_KEY_SLACK = 2e-6f;

struct RouteBufs {
    float* logits;      // [T, E]
    float* xnorm2;      // [T]
    float* wnorm2;      // [E]
    int32_t* fb_tokens; // [T]
};

cudaError_t launch_route_logits(const __nv_bfloat16* x, const float* Wr, int T, int d, int E,
                                const RouteBufs& rb, DevStatus* st, cudaStream_t s);
cudaError_t launch_route_select(const __nv_bfloat16* x, const float* Wr, const float* b, int T,
                                int d, int E, int k, int32_t* idx, float* gate,
                                const RouteBufs& rb, DevStatus* st, int num_sms, cudaStream_t s);

// ---------------------------------------------------------------- permute

constexpr int PERM_CHUNK = 4096;   // flat slots per CTA of the histogram / scatter

cudaError_t launch_permute(const int32_t* idx, int64_t n_slots, int k, int E, int bm,
                           const float* gate_flat, int32_t* hist, int32_t* counts,
                           int32_t* offsets, int32_t* tile_off, int32_t* perm, int32_t* inv,
                           int32_t* row_tok, float* row_gate, DevStatus* st, cudaStream_t s);

// One group of T rows: offsets = {0, T}, tile_off = {0, ceil(T / bm)}.
cudaError_t launch_single_group(int32_t* offsets, int32_t* tile_off, int T, int bm, cudaStream_t s);

// Tiles of `bm` rows per group from given offsets: tile_off[g] = sum_{g'<g} ceil(cnt/bm).
cudaError_t launch_tile_prefix(const int32_t* offsets, int G, int bm, int32_t* tile_off,
                               cudaStream_t s);

// ----------------------------------------------------------- grouped GEMM

constexpr int GM_BM = 128;        // rows per tile (tcgen05 M)
constexpr int GM_BK = 64;         // K per stage: 64 bf16 = one 128-byte swizzle row
constexpr int GM_STAGES = 4;
constexpr int GM_MAXBN = 256;     // largest N of one tcgen05.mma with M = 128
constexpr int GM_THREADS = 320;   // 4 epilogue warps, MMA warp, TMA warp, 4 gather warps
constexpr int GM_A_BYTES = GM_BM * GM_BK * 2;
constexpr int GM_B_BYTES = GM_BK * GM_MAXBN * 2;
constexpr int GM_SMEM_BYTES = GM_STAGES * (GM_A_BYTES + GM_B_BYTES) + 1024 + 256;

enum Epilogue : int {
    EPI_GELU_BF16 = 0,   // out[r, n] = bf16(GELU(acc))
    EPI_STORE_BF16 = 1,  // out[r, n] = bf16(acc)
    EPI_ADD_F32 = 2,     // yacc[tok(r), n] += scale(r) * acc   (vector atomics)
    EPI_STORE_F32 = 3,   // yacc[tok(r), n]  = scale(r) * acc
};

struct GemmArgs {
    CUtensorMap tmB;            // B = weights [G][K][N] bf16 (N contiguous), 3-D map {N, K, G}
    const __nv_bfloat16* A;     // A rows [*, lda] bf16
    int64_t lda;
    const int32_t* a_rows;      // A row of GEMM row r: a_rows ? a_rows[r] / a_div : r
    int a_div;
    int64_t a_nrows;            // rows of A; a gathered row outside [0, a_nrows) is a device error
    int64_t m_total;            // GEMM rows that may be written; tiles past it are a device error
    int64_t max_mtiles;         // host bound on tile_off[G]
    int64_t o_nrows;            // rows of yacc (EPI_*_F32); tokens outside are a device error
    const int32_t* offsets;     // [G + 1] GEMM-row segment of each group
    const int32_t* tile_off;    // [G + 1] m-tile prefix; tile_off[G] = number of m-tiles
    int G, K, N, BN, n_ntiles, num_kb, nbox;
    int epi;
    __nv_bfloat16* out;         // EPI_*_BF16
    int64_t ldo;
    float* yacc;                // EPI_*_F32
    int64_t ldy;
    const int32_t* o_rows;      // output token of row r: o_rows ? o_rows[r] / o_div : r
    int o_div;
    const float* row_scale;     // scale(r) = row_scale ? row_scale[r] : scale
    float scale;
    DevStatus* status;
    uint64_t limit_ns;
};

// Encodes the 3-D weight tensor map {N, K, G} for W[G][K][N] bf16.
bool make_weight_tmap(CUtensorMap* tm, const void* base, int64_t N, int64_t K, int64_t G);
// Picks BN (multiple of 16, <= 256) and the number of N tiles for width N.
void choose_bn(int N, int* BN, int* n_ntiles);
cudaError_t launch_grouped_gemm(const GemmArgs& a, int grid, cudaStream_t s);

// ------------------------------------------------------------------- misc

cudaError_t launch_zero_f32(float* p, int64_t n, cudaStream_t s);
cudaError_t launch_f32_to_bf16(const float* src, __nv_bfloat16* dst, int64_t n, cudaStream_t s);
cudaError_t launch_combine(const __nv_bfloat16* rows, const int32_t* inv, const float* gate,
                           const __nv_bfloat16* shared, float lambda, int64_t T, int k, int d,
                           __nv_bfloat16* y, cudaStream_t s);
cudaError_t launch_wait_probe(DevStatus* st, uint64_t limit_ns, cudaStream_t s);

}  // namespace mv
