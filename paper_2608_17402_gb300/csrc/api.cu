// api.cu -- extern "C" entry points of the MoE-ViE layer library (moevie.h,
// moevie_testing.h): argument checks, workspace carving and launch order.
// Nothing here allocates, frees or synchronises on the layer path.
#include <stdint.h>
#include <string.h>

#include <algorithm>
#include <atomic>
#include <mutex>

#include "internal.h"
#include "moevie_testing.h"

using namespace mv;

namespace {
std::atomic<uint64_t> g_launches{0};
}  // namespace

void mv::count_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

namespace {

constexpr uint64_t WAIT_LIMIT_NS = 2000000000ull;   // 2 s per pipeline wait

inline size_t up256(size_t v) { return (v + 255) & ~static_cast<size_t>(255); }
inline bool a16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
// Row stride (elements) of a bf16 matrix whose rows hold h values: W1, W3, Ws1, Ws3
// and the hidden activations.  Rows start 16 bytes apart, as a TMA stride must; the
// tensor maps cover the first h columns only, so the pad is never read.
inline int64_t row_ld(int64_t h) { return (h + 7) / 8 * 8; }

// Workspace carve-up.  Every buffer size is monotone in every size argument and
// the order is fixed, so a workspace sized for the whole layer also serves each
// stage (which passes 0 for the sizes it does not use).
struct Layout {
    size_t status, xnorm, wnorm, wpart, wexp, wsplit, wrt, logits, fb_tokens;
    size_t idx, gate, hist, counts, offsets, tiles, n_tiles, items, n_items, perm, inv, row_tok,
        row_gate;
    size_t H, Hs, yacc;
    size_t total;
};

struct BandPlan {   // token bands and n-tiles per column group of the down-projection
    int nb, gsz;
};
// Work order of the down-projection.  Its epilogue adds every routed row into the
// fp32 y accumulator [T, d]; when that is larger than ITEM_BAND_MIN_BYTES (it would
// not stay in L2 next to the streamed operands) the items run in nb token bands x
// column groups of gsz n-tiles (item_order_kernel), so that the accumulator block
// being reduced into (at most ITEM_BLOCK_BYTES) stays in L2.  Each extra band re-reads
// the weights W2 of the experts with m-tiles in it, each extra column group the rows
// of H.  Measured on GB300 (stress layer T = 65536, d = 1664, E = 256: 16 bands x 2
// column groups 955 us, 8 x 2 990 us, 5 x 4 1016 us, 16 x 1 984 us; video layer T =
// 32768, d = 1536, E = 128: every plan 408-411 us): the most bands, then the fewest
// column groups whose block fits, is the best plan on both.  Skewed loads keep the W2
// re-reads far below one per band per expert: an expert's rows span few bands unless
// it is large, and a large one is re-read from L2 within a band.
constexpr double ITEM_BAND_MIN_BYTES = 64.0 * (1 << 20);
constexpr double ITEM_BLOCK_BYTES = 24.0 * (1 << 20);
BandPlan choose_bands(int64_t T, int64_t d, int64_t E, int64_t k, int64_t h) {
    (void)h;
    int BN = 0, nnt = 0;
    choose_bn((int)d, &BN, &nnt);
    const double yacc = 4.0 * T * d;
    if (yacc <= ITEM_BAND_MIN_BYTES || max_mtiles(T * k, E) > ITEM_MAX_TILES) return {1, nnt};
    const int nb = ITEM_MAX_BANDS;
    for (int groups = 1; groups <= nnt; ++groups) {
        const int gsz = (nnt + groups - 1) / groups;
        const int g = (nnt + gsz - 1) / gsz;   // groups that gsz actually gives
        if (yacc / ((double)nb * g) <= ITEM_BLOCK_BYTES) return {nb, gsz};
    }
    return {nb, 1};
}

// The shared expert runs inside the grouped GEMMs as S = h_s / h always-on groups
// E .. E + S - 1 (its hidden units in chunks of h: GELU, like SiLU(gate) * up, acts
// unit by unit, so the chunks' down-projections add up to the shared expert's output),
// every token with gate lambda, when h divides h_s and the down-projection is not
// band-ordered.
// 0: the shared expert runs as its own dense GEMMs.
constexpr int64_t SHARED_MAX_CHUNKS = 16;
// Always-on groups the shapes allow (h divides h_s); the workspace reserves room for
// them whatever the band decision, so that its size stays monotone in T.
// Chunk c starts at column c h of Ws1 (and Ws3), h columns of a TMA stride apart: with
// more than one chunk, h must be a multiple of 8.
int64_t shared_chunks_max(int64_t h, int64_t hs) {
    if (hs <= 0 || h <= 0 || hs % h != 0 || hs / h > SHARED_MAX_CHUNKS) return 0;
    if (hs / h > 1 && h % 8 != 0) return 0;
    return hs / h;
}
int64_t shared_chunks(int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t hs) {
    if (shared_chunks_max(h, hs) == 0 || d <= 0 || T < 0) return 0;
    if (T * (k + hs / h) >= (int64_t(1) << 31)) return 0;
    int BN = 0, nnt = 0;
    choose_bn((int)d, &BN, &nnt);
    const BandPlan bp = choose_bands(T, d, E, k, h);
    if (bp.nb > 1 || bp.gsz < nnt) return 0;
    return hs / h;
}

Layout make_layout(int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t hs) {
    Layout L;
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o += up256(bytes);
        return at;
    };
    const int64_t n = T * k;
    const int64_t Ep = route_epad((int)E);
    const int64_t nchunks_max = (n + 255) / 256;   // chunks are at least 256 slots
    L.status = take(sizeof(DevStatus));
    L.xnorm = take(4 * T);
    L.wnorm = take(4 * 2 * E);                                        // |W_r[:, e]|, |lo_e|
    L.wpart = take(4 * 2 * (int64_t)route_split_parts((int)d) * Ep);
    L.wexp = take(4 * (int64_t)route_split_parts((int)d) * Ep);
    L.wsplit = take(2 * 2 * (int64_t)route_dpad((int)d) * Ep);
    L.wrt = take(4 * E * (int64_t)route_dpad((int)d));
    L.logits = take(4 * route_logits_rows(T, (int)d, (int)E) * Ep);
    L.fb_tokens = take(4 * T);
    L.idx = take(4 * n);
    L.gate = take(4 * n);
    L.hist = take(4 * nchunks_max * E);
    L.counts = take(4 * E);
    L.offsets = take(4 * (E + 1));
    // GEMM rows: routed, then the shared expert's always-on groups (room for them
    // whenever h divides h_s, folded or not, so that the size is monotone in T)
    const int64_t S = shared_chunks_max(h, hs);
    const int64_t n2 = n + S * T;
    L.tiles = take(16 * (max_mtiles(n, E) + S * ((T + GM_BM - 1) / GM_BM)));
    int BN = 0, n_nt = 0;
    choose_bn((int)(d > 0 ? d : 1), &BN, &n_nt);
    L.items = take(16 * max_mtiles(n, E) * n_nt);   // band-ordered down-projection items
    L.n_items = take(4);
    L.n_tiles = take(4);
    L.perm = take(4 * n);
    L.inv = take(4 * n);
    L.row_tok = take(4 * n2);
    L.row_gate = take(4 * n2);
    L.H = take(2 * n2 * row_ld(h));
    // the shared expert's own hidden [T, h_s]: with room for always-on groups it is the
    // tail of H (those S T rows of width h, the same bytes), used by one path or the other
    L.Hs = S > 0 ? L.H + (size_t)(2 * n * row_ld(h)) : take(2 * T * row_ld(hs));
    L.yacc = take(4 * T * d);
    L.total = o;
    return L;
}

template <typename P>
P* at(void* ws, size_t off) {
    return reinterpret_cast<P*>(static_cast<uint8_t*>(ws) + off);
}

moevie_status check_sizes(int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t hs) {
    if (T < 0 || d <= 0 || E <= 0 || k <= 0 || h < 0 || hs < 0) return MOEVIE_ERR_INVALID_ARG;
    if (d % 8 != 0) return MOEVIE_ERR_UNSUPPORTED;
    if (k > E || E > 1024) return MOEVIE_ERR_UNSUPPORTED;
    if (T * k >= (int64_t(1) << 31) || T * route_epad((int)E) >= (int64_t(1) << 40) ||
        d >= (int64_t(1) << 24) || h >= (int64_t(1) << 24) || hs >= (int64_t(1) << 24))
        return MOEVIE_ERR_UNSUPPORTED;
    return MOEVIE_OK;
}

// SM count of the current device (GB300: 152), cached per device; safe to call from
// several host threads at once.
int num_sms() {
    static std::atomic<int> cache[64];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 152;
    int n = cache[dev].load(std::memory_order_relaxed);
    if (n == 0) {
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 152;
        cache[dev].store(n, std::memory_order_relaxed);
    }
    return n;
}

inline moevie_status cuda_status(cudaError_t e) { return e == cudaSuccess ? MOEVIE_OK : MOEVIE_ERR_CUDA; }

#define MV_TRY(expr)                                     \
    do {                                                 \
        cudaError_t _e = (expr);                         \
        if (_e != cudaSuccess) return MOEVIE_ERR_CUDA;   \
    } while (0)

// One grouped GEMM launch: D = A[rows] . W[g], W bf16 [G][K][N] (row stride N_ld).
// The weight tensor maps cover N columns and K rows: tiles past either edge read zeros.
struct GemmSpec {
    const void* A;
    int64_t lda;
    int64_t a_cols;       // valid columns of an A row (0 = K)
    const int32_t* a_rows;
    int a_div;
    int a_kperiod;
    int64_t a_nrows;      // rows of A
    int64_t m_total;      // GEMM rows
    const int4* tiles;    // nullptr: one dense group of m_total rows
    const int32_t* n_tiles;
    int G;
    const void* W;
    int K, N;
    int64_t N_ld;         // inner extent of W (>= N), 0 = N
    int epi;
    void* out;
    int64_t ldo;
    float* yacc;
    int64_t ldy;
    int64_t o_nrows;      // rows of yacc
    const int32_t* o_rows;
    int o_div;
    const float* row_scale;
    float scale;
    int ksplit;              // 0 or 1: no split of K; fp32 outputs only otherwise
    int64_t y_split_stride;  // floats between the outputs of consecutive splits
    int item_table;          // tiles / n_tiles hold (m-tile, n-tile) work items
    float* zero;             // dense A: also clear zero[0, zero_n) (zero_n % 4 == 0)
    int64_t zero_n;
    float* nrm_out;          // dense A: also nrm_out[r] = |A[r, 0:K_A]| (K_A = a_cols or K)
    const float* wn_part;    // dense A: also wn_out[e] = sqrt(sum_p wn_part[p wn_Ep + e])
    int wn_nparts, wn_E, wn_Ep, wn_sets;
    float* wn_out;
    const void* W2nd;        // groups g >= g_split: weights at W2nd + (g - g_split) w2_g_ld +
    int64_t w2_k_ld;         //   kk w2_k_ld + n (elements); W then holds g_split groups
    int64_t w2_g_ld;
    int g_split;
    const void* W3;          // EPI_SWIGLU_BF16: the up projection W3 [G][K][N] beside W1 = W (gate)
    const void* W3_2nd;      // EPI_SWIGLU_BF16 with W2nd: the up projection of groups >= g_split
                             //   (strides as W2nd, which then holds their gate)
    int a_ident;             // A rows contiguous but loaded by the gather warps (A row r = r)
    // training path (see GemmArgs): K-major B W[G][N][K] with row stride b_k_ld and group
    // stride b_g_ld; M-major A [a_nrows][a_cols] (row stride lda) for weight-gradient items
    int b_kmajor;
    int64_t b_k_ld, b_g_ld;
    int a_mn;
    int wg_M;                // item_table == 2: output rows per group
    int64_t b_rows;          // item_table == 2: rows of B (one group, the K rows all items share)
    int64_t max_items;       // item_table == 2: host bound on the number of items
    int a_neg_zero, o_neg_skip;
    void* out2;
    void* out3;
    const void* epi_u;
    const void* epi_v;
    const void* epi_a;
    float* dg_part;
};

moevie_status run_gemm(const GemmSpec& g, DevStatus* st, cudaStream_t s) {
    GemmArgs a;
    memset(&a, 0, sizeof a);
    const int64_t n_ld = g.N_ld > 0 ? g.N_ld : g.N;
    if (n_ld < g.N || n_ld % 8 != 0) return MOEVIE_ERR_UNSUPPORTED;
    const bool swiglu = g.epi == EPI_SWIGLU_BF16;
    if (g.b_kmajor) {   // box: the CTA's half of an n-tile's columns
        int bn = 0, nnt = 0;
        choose_bn(g.N, &bn, &nnt);
        if (swiglu || g.W2nd || g.b_k_ld % 8 != 0 || g.b_g_ld % 8 != 0 || g.b_k_ld < g.K)
            return MOEVIE_ERR_UNSUPPORTED;
        if (!make_kmajor_tmap(&a.tmB, g.W, g.K, g.N, g.G, g.b_k_ld, g.b_g_ld, bn / 2)) return MOEVIE_ERR_CUDA;
    } else if (g.item_table == 2) {   // weight gradients: B [b_rows][N] as one group
        if (!make_weight_tmap_strided(&a.tmB, g.W, g.N, g.b_rows, 1, n_ld, n_ld * g.b_rows)) return MOEVIE_ERR_CUDA;
    } else if (!make_weight_tmap_strided(&a.tmB, g.W, g.N, g.K, g.W2nd ? g.g_split : g.G, n_ld, n_ld * g.K)) {
        return MOEVIE_ERR_CUDA;
    }
    if (g.W2nd) {   // groups >= g_split (swiglu: their gate in tmB3, their up projection in tmB4)
        if (g.g_split <= 0 || g.g_split >= g.G || !a16(g.W2nd) || g.w2_k_ld % 8 != 0 ||
            g.w2_g_ld % 8 != 0 || g.w2_k_ld < g.N)
            return MOEVIE_ERR_UNSUPPORTED;
        if (!make_weight_tmap_strided(swiglu ? &a.tmB3 : &a.tmB2, g.W2nd, g.N, g.K, g.G - g.g_split,
                                      g.w2_k_ld, g.w2_g_ld))
            return MOEVIE_ERR_CUDA;
        if (swiglu) {
            if (!g.W3_2nd || !a16(g.W3_2nd)) return MOEVIE_ERR_UNSUPPORTED;
            if (!make_weight_tmap_strided(&a.tmB4, g.W3_2nd, g.N, g.K, g.G - g.g_split, g.w2_k_ld,
                                          g.w2_g_ld))
                return MOEVIE_ERR_CUDA;
        }
    }
    if (g.a_mn) {   // A [a_nrows = K rows][a_cols = M] as the 3-D map {M, K, 1}, box {64, 64, 1}
        if (g.a_rows || g.lda % 8 != 0 || g.item_table != 2) return MOEVIE_ERR_UNSUPPORTED;
        if (!make_weight_tmap_strided(&a.tmA, g.A, g.a_cols, g.a_nrows, 1, g.lda, g.lda * g.a_nrows))
            return MOEVIE_ERR_CUDA;
    } else if (!g.a_rows && !make_rows_tmap(&a.tmA, g.A, g.a_cols > 0 ? g.a_cols : g.K, g.a_nrows, g.lda)) {
        return MOEVIE_ERR_CUDA;
    }
    a.b_kmajor = g.b_kmajor ? 1 : 0;
    a.a_mn = g.a_mn ? 1 : 0;
    a.wg_M = g.wg_M;
    a.a_neg_zero = g.a_neg_zero;
    a.o_neg_skip = g.o_neg_skip;
    a.out2 = static_cast<__nv_bfloat16*>(g.out2);
    a.out3 = static_cast<__nv_bfloat16*>(g.out3);
    a.epi_u = static_cast<const __nv_bfloat16*>(g.epi_u);
    a.epi_v = static_cast<const __nv_bfloat16*>(g.epi_v);
    a.epi_a = static_cast<const __nv_bfloat16*>(g.epi_a);
    a.dg_part = g.dg_part;
    a.A = static_cast<const __nv_bfloat16*>(g.A);
    a.lda = g.lda;
    a.a_rows = g.a_rows;
    a.a_div = g.a_div > 0 ? g.a_div : 1;
    a.a_kperiod = g.a_kperiod;
    a.a_nrows = g.a_nrows;
    a.m_total = g.m_total;
    a.tiles = g.tiles;
    a.n_tiles_dev = g.n_tiles;
    a.max_mtiles = g.tiles ? max_mtiles(g.m_total, g.G) : (g.m_total + GM_BM - 1) / GM_BM;
    a.item_table = g.item_table;
    a.a_ident = (g.a_ident && !g.a_rows) ? 1 : 0;
    // reduction staging: a full-warp buffer (5 stages) unless the work is band-ordered
    // (accumulator beyond L2, DRAM-bound: the sixth stage pays more)
    a.stg_rows = g.item_table ? 16 : 32;
    if (g.zero && (g.a_rows || g.zero_n % 4 != 0 || !a16(g.zero))) return MOEVIE_ERR_UNSUPPORTED;
    a.zero = reinterpret_cast<float4*>(g.zero);
    a.zero_n = g.zero ? g.zero_n / 4 : 0;
    if (g.nrm_out) {
        const int64_t cols = g.a_cols > 0 ? g.a_cols : g.K;
        if (g.a_rows || cols % 8 != 0 || g.lda % 8 != 0) return MOEVIE_ERR_UNSUPPORTED;
        a.nrm_x = static_cast<const __nv_bfloat16*>(g.A);
        a.nrm_ld = g.lda;
        a.nrm_cols = (int)cols;
        a.nrm_out = g.nrm_out;
    }
    if (g.wn_out) {
        if (g.a_rows || g.wn_E <= 0 || g.wn_Ep < g.wn_E || g.wn_nparts < 1 || g.wn_sets < 1)
            return MOEVIE_ERR_UNSUPPORTED;
        a.wn_part = g.wn_part;
        a.wn_nparts = g.wn_nparts;
        a.wn_E = g.wn_E;
        a.wn_Ep = g.wn_Ep;
        a.wn_sets = g.wn_sets;
        a.wn_out = g.wn_out;
    }
    a.G = g.G;
    a.g_split = g.W2nd ? g.g_split : g.G;
    a.swiglu = swiglu ? 1 : 0;
    if (a.swiglu) {   // gate (W1) and up (W3) tiles of 128 columns side by side: one N = 256 MMA
        if (!g.W3 || !a16(g.W3) || g.ksplit > 1) return MOEVIE_ERR_UNSUPPORTED;
        if (!make_weight_tmap_strided(&a.tmB2, g.W3, g.N, g.K, g.G, n_ld, n_ld * g.K))
            return MOEVIE_ERR_CUDA;
    }
    a.K = g.K;
    a.N = g.N;
    choose_bn(g.N, &a.BN, &a.n_ntiles);
    a.n_step = a.BN;
    if (a.swiglu) {
        a.BN = GM_MAXBN;
        a.n_step = GM_MAXBN / 2;
        a.n_ntiles = (g.N + a.n_step - 1) / a.n_step;
    }
    a.num_kb = (g.K + GM_BK - 1) / GM_BK;
    a.nbox = (a.BN + 63) / 64;
    a.epi = g.epi;
    a.out = static_cast<__nv_bfloat16*>(g.out);
    a.ldo = g.ldo;
    a.yacc = g.yacc;
    a.ldy = g.ldy;
    a.o_nrows = g.o_nrows;
    a.o_rows = g.o_rows;
    a.o_div = g.o_div > 0 ? g.o_div : 1;
    a.row_scale = g.row_scale;
    a.scale = g.scale;
    a.ksplit = g.ksplit > 1 ? g.ksplit : 1;
    if (a.ksplit > a.num_kb) return MOEVIE_ERR_UNSUPPORTED;
    if (a.ksplit > 1 && g.epi != EPI_STORE_F32 && g.epi != EPI_ADD_F32 && g.epi != EPI_SUM2_F32)
        return MOEVIE_ERR_UNSUPPORTED;
    if (g.epi == EPI_SUM2_F32 && (g.N % 64 != 0 || g.N > GM_MAXBN)) return MOEVIE_ERR_UNSUPPORTED;
    a.y_split_stride = g.y_split_stride;
    a.status = st;
    a.limit_ns = WAIT_LIMIT_NS;
    if (a.item_table == 2) {
        if (!g.tiles || a.ksplit != 1 || g.wg_M <= 0 || g.wg_M > 65535 || g.N > 65535) return MOEVIE_ERR_UNSUPPORTED;
        a.max_mtiles = g.max_items;
    } else if (a.item_table) {
        if (!g.tiles || a.ksplit != 1) return MOEVIE_ERR_UNSUPPORTED;
        a.max_mtiles *= a.n_ntiles;   // bound on the item count
    }
    const int64_t work = a.item_table ? a.max_mtiles : a.max_mtiles * a.n_ntiles * a.ksplit;   // one CTA pair per item at most
    if (work >= (int64_t(1) << 31)) return MOEVIE_ERR_UNSUPPORTED;   // item indices are 32-bit in the kernel
    const int sms = num_sms() & ~1;
    const int grid = (int)(2 * work < sms ? (work > 0 ? 2 * work : 2) : sms);
    return cuda_status(launch_grouped_gemm(a, grid, s));
}

// Router (Eqs. 1, 7, 4-5): bf16 pieces hi, mid of W_r, tensor-core logits x . (hi +
// mid), certified top-k with exact re-decision of near ties.
moevie_status route_impl(const void* x, const float* W_r, const float* b, int64_t T, int64_t d,
                         int64_t E, int64_t k, int32_t* idx, float* gate, const Layout& L,
                         void* ws, cudaStream_t s, bool logits_only = false,
                         float* logits_out = nullptr, float* zero_acc = nullptr) {
    DevStatus* st = at<DevStatus>(ws, L.status);
    const int Ep = route_epad((int)E);
    __nv_bfloat16* wsplit = at<__nv_bfloat16>(ws, L.wsplit);
    float* wrt = at<float>(ws, L.wrt);
    float* wnorm = at<float>(ws, L.wnorm);
    const int ksplit = route_ksplit(T, (int)d, (int)E);
    // partial logits: ksplit arrays [T][Ep]; straight into logits_out when unsplit
    float* logits = (logits_out && ksplit == 1) ? logits_out : at<float>(ws, L.logits);
    const int64_t part_stride = T * Ep;
    MV_TRY(launch_route_split(W_r, (int)d, (int)E, wsplit, wrt, at<float>(ws, L.wpart),
                              at<int32_t>(ws, L.wexp), st, s));
    const int64_t dp = route_dpad((int)d);
    const bool cc = route_concat((int)E);
    GemmSpec g{};
    g.A = x;
    g.lda = d;
    g.a_cols = d;
    g.a_nrows = T;
    g.m_total = T;
    g.G = 1;
    g.W = wsplit;
    if (cc) {   // B [dp][2 Ep]: the two pieces side by side, summed by the epilogue
        g.K = (int)dp;
        g.N = 2 * Ep;
        g.N_ld = 2 * Ep;
        g.epi = EPI_SUM2_F32;
    } else {    // B [2][dp][Ep]: K = 2 dp, x read twice, once per piece
        g.a_kperiod = (int)dp;
        g.K = (int)(2 * dp);
        g.N = (int)E;
        g.N_ld = Ep;
        g.epi = EPI_STORE_F32;
    }
    g.yacc = logits;
    g.ldy = Ep;
    g.o_nrows = T;
    g.scale = 1.0f;
    g.ksplit = ksplit;
    g.y_split_stride = part_stride;
    g.nrm_out = logits_only ? nullptr : at<float>(ws, L.xnorm);   // |x_t| for the certificate
    if (!logits_only) {   // |W_r[:, e]| and |lo_e| for the certificate, from the split's partial sums
        g.wn_part = at<float>(ws, L.wpart);
        g.wn_nparts = route_split_parts((int)d);
        g.wn_E = (int)E;
        g.wn_Ep = Ep;
        g.wn_sets = 2;
        g.wn_out = wnorm;
    }
    moevie_status c = run_gemm(g, st, s);
    if (c != MOEVIE_OK) return c;
    if (logits_only) {
        if (logits_out && ksplit > 1)
            MV_TRY(launch_route_sum_parts(logits, part_stride, ksplit, part_stride, logits_out, s));
        return MOEVIE_OK;
    }
    MV_TRY(launch_route_select(static_cast<const __nv_bfloat16*>(x), wrt, b, logits, Ep, ksplit,
                               part_stride, wnorm, at<int32_t>(ws, L.wexp), (int)T, (int)d, (int)E,
                               (int)k, idx, gate, at<int32_t>(ws, L.fb_tokens), at<float>(ws, L.xnorm),
                               st, num_sms(), s, zero_acc, T * d));   // top-k also clears y's accumulator
    return MOEVIE_OK;
}

moevie_status expert_up(const void* x, const int32_t* a_rows, int a_div, const int4* tiles,
                        const int32_t* n_tiles, const void* W1, int64_t T, int64_t d, int64_t h,
                        int64_t E, int64_t k, void* hidden, DevStatus* st, cudaStream_t s) {
    GemmSpec g{};
    g.A = x;
    g.lda = d;
    g.a_rows = a_rows;
    g.a_div = a_div;
    g.a_nrows = T;
    g.m_total = T * k;
    g.tiles = tiles;
    g.n_tiles = n_tiles;
    g.G = (int)E;
    g.W = W1;
    g.K = (int)d;
    g.N = (int)h;
    g.N_ld = row_ld(h);
    g.epi = EPI_GELU_BF16;
    g.out = hidden;
    g.ldo = row_ld(h);
    return run_gemm(g, st, s);
}

// Shared expert as one dense group of all T rows.  Writes either a bf16 output
// (out != NULL) or lambda * S(x) as the first value of the fp32 y accumulator.
moevie_status shared_expert(const void* x, const void* Ws1, const void* Ws2, int64_t T, int64_t d,
                            int64_t hs, void* out, float* yacc, float lambda, const Layout& L,
                            void* ws, DevStatus* st, cudaStream_t s, const void* Ws3 = nullptr) {
    void* Hs = at<void>(ws, L.Hs);
    GemmSpec g{};
    g.A = x;
    g.lda = d;
    g.a_nrows = T;
    g.m_total = T;
    g.G = 1;
    g.W = Ws1;
    g.K = (int)d;
    g.N = (int)hs;
    g.N_ld = row_ld(hs);
    g.epi = EPI_GELU_BF16;
    if (Ws3) {   // SwiGLU shared expert: gate Ws1, up Ws3 (the SwiGLU epilogue runs with gathered A)
        g.epi = EPI_SWIGLU_BF16;
        g.W3 = Ws3;
        g.a_ident = 1;
    }
    g.out = Hs;
    g.ldo = row_ld(hs);
    moevie_status c = run_gemm(g, st, s);
    if (c != MOEVIE_OK) return c;
    GemmSpec g2{};
    g2.A = Hs;
    g2.lda = row_ld(hs);
    g2.a_nrows = T;
    g2.m_total = T;
    g2.G = 1;
    g2.W = Ws2;
    g2.K = (int)hs;
    g2.N = (int)d;
    if (out) {
        g2.epi = EPI_STORE_BF16;
        g2.out = out;
        g2.ldo = d;
    } else {
        g2.epi = EPI_STORE_F32;
        g2.yacc = yacc;
        g2.ldy = d;
        g2.o_nrows = T;
        g2.scale = lambda;
    }
    return run_gemm(g2, st, s);
}

}  // namespace

extern "C" {

const char* moevie_status_string(moevie_status s) {
    switch (s) {
        case MOEVIE_OK: return "MOEVIE_OK";
        case MOEVIE_ERR_INVALID_ARG: return "MOEVIE_ERR_INVALID_ARG";
        case MOEVIE_ERR_UNSUPPORTED: return "MOEVIE_ERR_UNSUPPORTED";
        case MOEVIE_ERR_WORKSPACE: return "MOEVIE_ERR_WORKSPACE";
        case MOEVIE_ERR_CUDA: return "MOEVIE_ERR_CUDA";
        case MOEVIE_ERR_TIMEOUT: return "MOEVIE_ERR_TIMEOUT";
        case MOEVIE_ERR_DEVICE: return "MOEVIE_ERR_DEVICE";
        default: return "MOEVIE_ERR_UNKNOWN";
    }
}

int moevie_version(void) { return 200; }

uint64_t moevie_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

moevie_status moevie_update_bias(const int32_t* counts, int64_t E, float alpha, int rule, float* b,
                                 void* ws, size_t ws_bytes, void* stream) {
    if (E < 1 || E > 1024 || (rule != 0 && rule != 1)) return MOEVIE_ERR_INVALID_ARG;
    if (!counts || !b || !ws || !a16(ws)) return MOEVIE_ERR_INVALID_ARG;
    if (ws_bytes < 256) return MOEVIE_ERR_WORKSPACE;
    return cuda_status(launch_update_bias(counts, (int)E, alpha, rule, b, static_cast<DevStatus*>(ws),
                                          static_cast<cudaStream_t>(stream)));
}

int64_t moevie_shared_groups(int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t h_s) {
    if (check_sizes(T, d, E, k, h, h_s) != MOEVIE_OK) return 0;
    return shared_chunks(T, d, E, k, h, h_s);
}

moevie_status moevie_workspace_size(int64_t T_max, int64_t d, int64_t E, int64_t k, int64_t h,
                                    int64_t h_s, size_t* bytes) {
    if (!bytes) return MOEVIE_ERR_INVALID_ARG;
    const moevie_status c = check_sizes(T_max, d, E, k, h, h_s);
    if (c != MOEVIE_OK) return c;
    *bytes = make_layout(T_max, d, E, k, h, h_s).total;
    return MOEVIE_OK;
}

moevie_status moevie_workspace_init(void* ws, size_t ws_bytes, void* stream) {
    if (!ws || ws_bytes < sizeof(DevStatus) || !a16(ws)) return MOEVIE_ERR_INVALID_ARG;
    return cuda_status(cudaMemsetAsync(ws, 0, sizeof(DevStatus), static_cast<cudaStream_t>(stream)));
}

moevie_status moevie_route(const void* x, const float* W_r, const float* b, int64_t T, int64_t d,
                           int64_t E, int64_t k, int32_t* idx, float* gate, void* ws,
                           size_t ws_bytes, void* stream) {
    moevie_status c = check_sizes(T, d, E, k, 0, 0);
    if (c != MOEVIE_OK) return c;
    if (T == 0) return MOEVIE_OK;
    if (!x || !W_r || !b || !idx || !gate || !ws) return MOEVIE_ERR_INVALID_ARG;
    if (!a16(x) || !a16(ws)) return MOEVIE_ERR_INVALID_ARG;
    const Layout L = make_layout(T, d, E, k, 0, 0);
    if (ws_bytes < L.total) return MOEVIE_ERR_WORKSPACE;
    return route_impl(x, W_r, b, T, d, E, k, idx, gate, L, ws, static_cast<cudaStream_t>(stream));
}

moevie_status moevie_permute(const int32_t* idx, int64_t T, int64_t k, int64_t E, int32_t* counts,
                             int32_t* offsets, int32_t* perm, int32_t* inv, void* ws,
                             size_t ws_bytes, void* stream) {
    moevie_status c = check_sizes(T, 8, E, k, 0, 0);
    if (c != MOEVIE_OK) return c;
    if (!counts || !offsets || !ws) return MOEVIE_ERR_INVALID_ARG;
    if (T > 0 && (!idx || !perm || !inv)) return MOEVIE_ERR_INVALID_ARG;
    if (!a16(ws) || (idx && !a16(idx))) return MOEVIE_ERR_INVALID_ARG;
    const Layout L = make_layout(T, 0, E, k, 0, 0);
    if (ws_bytes < L.total) return MOEVIE_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (T == 0) {   // all counts and offsets are zero
        MV_TRY(cudaMemsetAsync(counts, 0, 4 * E, s));
        MV_TRY(cudaMemsetAsync(offsets, 0, 4 * (E + 1), s));
        return MOEVIE_OK;
    }
    DevStatus* st = at<DevStatus>(ws, L.status);
    const int chunk = perm_chunk(T * k, num_sms());
    MV_TRY(launch_permute(idx, T * k, (int)k, (int)E, GM_BM, chunk, nullptr, at<int32_t>(ws, L.hist),
                          counts, offsets, at<int4>(ws, L.tiles), at<int32_t>(ws, L.n_tiles), perm,
                          inv, nullptr, nullptr, st, s));
    return MOEVIE_OK;
}

moevie_status moevie_permute_static(const int32_t* idx, int64_t T, int64_t k, int64_t E,
                                    int32_t* counts, int32_t* offsets, int32_t* perm,
                                    int32_t* inv, void* stream) {
    moevie_status c = check_sizes(T, 8, E, k, 0, 0);
    if (c != MOEVIE_OK) return c;
    if (T * k > PERM_STATIC_MAX_SLOTS) return MOEVIE_ERR_UNSUPPORTED;   // beyond the fixed scratch
    if (!counts || !offsets) return MOEVIE_ERR_INVALID_ARG;
    if (T > 0 && (!idx || !perm || !inv)) return MOEVIE_ERR_INVALID_ARG;
    if (idx && !a16(idx)) return MOEVIE_ERR_INVALID_ARG;
    unsigned char* scratch = nullptr;
    MV_TRY(perm_static_scratch(&scratch));   // the first call on a device looks it up
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (T == 0) {
        MV_TRY(cudaMemsetAsync(counts, 0, 4 * E, s));
        MV_TRY(cudaMemsetAsync(offsets, 0, 4 * (E + 1), s));
        return MOEVIE_OK;
    }
    // The status block must start at zero (a report only lands in a clear block);
    // the histograms, tile table and tile count are fully rewritten by the kernels.
    DevStatus* st = reinterpret_cast<DevStatus*>(scratch);
    MV_TRY(cudaMemsetAsync(st, 0, sizeof(DevStatus), s));
    const int64_t n = T * k;
    int64_t chunk = perm_chunk(n, num_sms());
    const int64_t min_chunk = ((n + PERM_STATIC_MAX_CHUNKS - 1) / PERM_STATIC_MAX_CHUNKS + 255) / 256 * 256;
    if (chunk < min_chunk) chunk = min_chunk;   // at most PERM_STATIC_MAX_CHUNKS histograms
    MV_TRY(launch_permute(idx, n, (int)k, (int)E, GM_BM, (int)chunk, nullptr,
                          reinterpret_cast<int32_t*>(scratch + PERM_STATIC_HIST_OFF), counts, offsets,
                          reinterpret_cast<int4*>(scratch + PERM_STATIC_TILES_OFF),
                          reinterpret_cast<int32_t*>(scratch + PERM_STATIC_NTILES_OFF), perm, inv,
                          nullptr, nullptr, st, s));
    return MOEVIE_OK;
}

moevie_status moevie_expert_ffn(const void* x, const int32_t* perm, const int32_t* offsets,
                                const void* W1, const void* W2, int64_t T, int64_t d, int64_t h,
                                int64_t E, int64_t k, void* out_rows, void* ws, size_t ws_bytes,
                                void* stream) {
    moevie_status c = check_sizes(T, d, E, k, h, 0);
    if (c != MOEVIE_OK) return c;
    if (h == 0) return MOEVIE_ERR_UNSUPPORTED;
    if (T == 0) return MOEVIE_OK;
    if (!x || !perm || !offsets || !W1 || !W2 || !out_rows || !ws) return MOEVIE_ERR_INVALID_ARG;
    if (!a16(x) || !a16(W1) || !a16(W2) || !a16(out_rows) || !a16(ws)) return MOEVIE_ERR_INVALID_ARG;
    const Layout L = make_layout(T, 0, E, k, h, 0);
    if (ws_bytes < L.total) return MOEVIE_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DevStatus* st = at<DevStatus>(ws, L.status);
    int4* tiles = at<int4>(ws, L.tiles);
    int32_t* n_tiles = at<int32_t>(ws, L.n_tiles);
    void* H = at<void>(ws, L.H);
    MV_TRY(launch_tile_table(offsets, (int)E, GM_BM, tiles, n_tiles, s));
    c = expert_up(x, perm, (int)k, tiles, n_tiles, W1, T, d, h, E, k, H, st, s);
    if (c != MOEVIE_OK) return c;
    GemmSpec g{};
    g.A = H;
    g.lda = row_ld(h);
    g.a_nrows = T * k;
    g.m_total = T * k;
    g.tiles = tiles;
    g.n_tiles = n_tiles;
    g.G = (int)E;
    g.W = W2;
    g.K = (int)h;
    g.N = (int)d;
    g.epi = EPI_STORE_BF16;
    g.out = out_rows;
    g.ldo = d;
    return run_gemm(g, st, s);
}

moevie_status moevie_shared_expert(const void* x, const void* Ws1, const void* Ws2, int64_t T,
                                   int64_t d, int64_t h_s, void* out, void* ws, size_t ws_bytes,
                                   void* stream) {
    moevie_status c = check_sizes(T, d, 1, 1, 0, h_s);
    if (c != MOEVIE_OK) return c;
    if (h_s == 0) return MOEVIE_ERR_UNSUPPORTED;
    if (T == 0) return MOEVIE_OK;
    if (!x || !Ws1 || !Ws2 || !out || !ws) return MOEVIE_ERR_INVALID_ARG;
    if (!a16(x) || !a16(Ws1) || !a16(Ws2) || !a16(out) || !a16(ws)) return MOEVIE_ERR_INVALID_ARG;
    const Layout L = make_layout(T, 0, 1, 1, 0, h_s);
    if (ws_bytes < L.total) return MOEVIE_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    return shared_expert(x, Ws1, Ws2, T, d, h_s, out, nullptr, 0.f, L, ws,
                         at<DevStatus>(ws, L.status), s);
}

moevie_status moevie_combine(const void* out_rows, const int32_t* inv, const float* gate,
                             const void* shared_out, float lambda, int64_t T, int64_t k, int64_t d,
                             void* y, void* stream) {
    moevie_status c = check_sizes(T, d, k, k, 0, 0);
    if (c != MOEVIE_OK) return c;
    if (T == 0) return MOEVIE_OK;
    if (!out_rows || !inv || !gate || !y) return MOEVIE_ERR_INVALID_ARG;
    if (!a16(out_rows) || !a16(y) || (shared_out && !a16(shared_out))) return MOEVIE_ERR_INVALID_ARG;
    return cuda_status(launch_combine(static_cast<const __nv_bfloat16*>(out_rows), inv, gate,
                                      static_cast<const __nv_bfloat16*>(shared_out), lambda, T,
                                      (int)k, (int)d, static_cast<__nv_bfloat16*>(y),
                                      static_cast<cudaStream_t>(stream)));
}

static moevie_status forward_impl(const moevie_layer* Lr, const void* x, int64_t T, void* y,
                                  const moevie_routing* routing, void* ws, size_t ws_bytes,
                                  void* stream, void* const* events, int n_events) {
    if (!Lr) return MOEVIE_ERR_INVALID_ARG;
    if (events && n_events != 7) return MOEVIE_ERR_INVALID_ARG;
    const int64_t d = Lr->d, E = Lr->E, k = Lr->k, h = Lr->h, hs = Lr->h_s;
    moevie_status c = check_sizes(T, d, E, k, h, hs);
    if (c != MOEVIE_OK) return c;
    if (h == 0) return MOEVIE_ERR_UNSUPPORTED;
    if (T == 0) return MOEVIE_OK;
    if (!x || !y || !ws || !Lr->W_r || !Lr->b || !Lr->W1 || !Lr->W2) return MOEVIE_ERR_INVALID_ARG;
    if (hs > 0 && (!Lr->Ws1 || !Lr->Ws2)) return MOEVIE_ERR_INVALID_ARG;
    if (Lr->W3 && hs > 0 && !Lr->Ws3) return MOEVIE_ERR_INVALID_ARG;   // SwiGLU shared expert needs Ws3
    if (!a16(x) || !a16(y) || !a16(ws) || !a16(Lr->W1) || !a16(Lr->W2)) return MOEVIE_ERR_INVALID_ARG;
    if (Lr->W3 && !a16(Lr->W3)) return MOEVIE_ERR_INVALID_ARG;
    if (Lr->W3 && hs > 0 && !a16(Lr->Ws3)) return MOEVIE_ERR_INVALID_ARG;
    if (hs > 0 && (!a16(Lr->Ws1) || !a16(Lr->Ws2))) return MOEVIE_ERR_INVALID_ARG;
    const Layout L = make_layout(T, d, E, k, h, hs);
    if (ws_bytes < L.total) return MOEVIE_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DevStatus* st = at<DevStatus>(ws, L.status);
    moevie_routing r{};
    if (routing) r = *routing;
    int32_t* idx = r.idx ? r.idx : at<int32_t>(ws, L.idx);
    float* gate = r.gate ? r.gate : at<float>(ws, L.gate);
    int32_t* counts = r.counts ? r.counts : at<int32_t>(ws, L.counts);
    int32_t* offsets = r.offsets ? r.offsets : at<int32_t>(ws, L.offsets);
    int32_t* perm = r.perm ? r.perm : at<int32_t>(ws, L.perm);
    int32_t* inv = r.inv ? r.inv : at<int32_t>(ws, L.inv);
    if (!a16(idx)) return MOEVIE_ERR_INVALID_ARG;
    int4* tiles = at<int4>(ws, L.tiles);
    int32_t* n_tiles = at<int32_t>(ws, L.n_tiles);
    int32_t* row_tok = at<int32_t>(ws, L.row_tok);
    float* row_gate = at<float>(ws, L.row_gate);
    float* yacc = at<float>(ws, L.yacc);
    auto mark = [&](int i) -> cudaError_t {
        return events ? cudaEventRecord(static_cast<cudaEvent_t>(events[i]), s) : cudaSuccess;
    };

    // shared expert inside the grouped GEMMs (GELU or SwiGLU: both act unit by unit)
    const int64_t S = shared_chunks(T, d, E, k, h, hs);
    const int64_t n2 = T * k + S * T;
    MV_TRY(mark(0));
    // 1. router (Eqs. 1, 7, 4-5)
    // unless a separate shared-expert GEMM writes it first, the router's top-k kernel
    // also clears the y accumulator (it leaves HBM mostly idle)
    if ((c = route_impl(x, Lr->W_r, Lr->b, T, d, E, k, idx, gate, L, ws, s, false, nullptr,
                        (hs > 0 && S == 0) ? nullptr : yacc)) != MOEVIE_OK)
        return c;
    MV_TRY(mark(1));
    // 2. expert-major order (Algorithm 1, phase 1), per-row token and gate, m-tile table
    const int chunk = perm_chunk(T * k, num_sms());
    // (with the shared expert's always-on groups appended: rows, gates lambda, m-tiles)
    const SharedRows sh{(int)S, T, Lr->lambda};
    MV_TRY(launch_permute(idx, T * k, (int)k, (int)E, GM_BM, chunk, gate, at<int32_t>(ws, L.hist),
                          counts, offsets, tiles, n_tiles, perm, inv, row_tok, row_gate, st, s,
                          S > 0 ? &sh : nullptr));
    int dBN = 0, dnt = 0;
    choose_bn((int)d, &dBN, &dnt);
    const BandPlan bp = choose_bands(T, d, E, k, h);
    const bool banded = bp.nb > 1 || bp.gsz < dnt;
    if (banded)
        MV_TRY(launch_item_order(tiles, n_tiles, row_tok, T, bp.nb, dnt, bp.gsz, dBN,
                                 (int)max_mtiles(T * k, E), at<int4>(ws, L.items),
                                 at<int32_t>(ws, L.n_items), s));
    MV_TRY(mark(2));
    // 3. shared expert (Eq. 3): S always-on groups of the grouped GEMMs (appended by the
    // permute step); otherwise its own GEMMs write lambda * shared expert as the first
    // value of the y accumulator
    if (S == 0 && hs > 0) {
        c = shared_expert(x, Lr->Ws1, Lr->Ws2, T, d, hs, nullptr, yacc, Lr->lambda, L, ws, st, s,
                          Lr->W3 ? Lr->Ws3 : nullptr);
        if (c != MOEVIE_OK) return c;
    }
    MV_TRY(mark(3));
    // 4. grouped up-projection, token gather in the operand load, GELU epilogue
    {
        GemmSpec up{};
        up.A = x;
        up.lda = d;
        up.a_rows = row_tok;
        up.a_div = 1;
        up.a_nrows = T;
        up.m_total = n2;
        up.tiles = tiles;
        up.n_tiles = n_tiles;
        up.G = (int)(E + S);
        up.W = Lr->W1;
        up.K = (int)d;
        up.N = (int)h;
        up.N_ld = row_ld(h);
        up.epi = Lr->W3 ? EPI_SWIGLU_BF16 : EPI_GELU_BF16;
        up.W3 = Lr->W3;   // SwiGLU: W1 the gate, W3 the up projection
        up.out = at<void>(ws, L.H);
        up.ldo = row_ld(h);
        if (S > 0) {   // chunk c of Ws1 [d, h_s] (and of Ws3): columns c h .. c h + h - 1
            up.W2nd = Lr->Ws1;
            up.W3_2nd = Lr->W3 ? Lr->Ws3 : nullptr;
            up.w2_k_ld = row_ld(hs);
            up.w2_g_ld = S > 1 ? h : row_ld(hs) * d;   // one chunk: any stride of 16-byte multiples
            up.g_split = (int)E;
        }
        if ((c = run_gemm(up, st, s)) != MOEVIE_OK) return c;
    }
    MV_TRY(mark(4));
    // 5. grouped down-projection, epilogue: gate * row added into y (scatter-add)
    GemmSpec dn{};
    dn.A = at<void>(ws, L.H);
    dn.lda = row_ld(h);
    dn.a_nrows = n2;
    dn.m_total = n2;
    dn.tiles = banded ? at<int4>(ws, L.items) : tiles;
    dn.n_tiles = banded ? at<int32_t>(ws, L.n_items) : n_tiles;
    dn.item_table = banded ? 1 : 0;
    dn.G = (int)(E + S);
    dn.W = Lr->W2;
    if (S > 0) {   // chunk c of Ws2 [h_s, d]: rows c h .. c h + h - 1
        dn.W2nd = Lr->Ws2;
        dn.w2_k_ld = d;
        dn.w2_g_ld = h * d;
        dn.g_split = (int)E;
    }
    dn.K = (int)h;
    dn.N = (int)d;
    dn.epi = EPI_ADD_F32;
    dn.yacc = yacc;
    dn.ldy = d;
    dn.o_nrows = T;
    dn.o_rows = row_tok;
    dn.o_div = 1;
    dn.row_scale = row_gate;
    if ((c = run_gemm(dn, st, s)) != MOEVIE_OK) return c;
    MV_TRY(mark(5));
    // 6. y = bf16(accumulator)
    MV_TRY(launch_f32_to_bf16(yacc, static_cast<__nv_bfloat16*>(y), T * d, s));
    MV_TRY(mark(6));
    return MOEVIE_OK;
}

moevie_status moevie_moe_forward(const moevie_layer* layer, const void* x, int64_t T, void* y,
                                 const moevie_routing* routing, void* ws, size_t ws_bytes,
                                 void* stream) {
    return forward_impl(layer, x, T, y, routing, ws, ws_bytes, stream, nullptr, 0);
}

}  // extern "C"

namespace {

// Copy streams and events of moevie_moe_forward_host, one set per device, created by the
// first call in a context (and again in a new context after a device reset).
struct HostPipe {
    void* ctx = nullptr;
    cudaStream_t in = nullptr, out = nullptr;
    cudaEvent_t start = nullptr, done = nullptr;
    cudaEvent_t ev_in[MOEVIE_HOST_MAX_CHUNKS + 1] = {}, ev_out[MOEVIE_HOST_MAX_CHUNKS + 1] = {};   // per piece
};

cudaError_t host_pipe(HostPipe** out) {
    constexpr int kMaxDevices = 64;
    static std::mutex mu;
    static HostPipe pipes[kMaxDevices];
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    std::lock_guard<std::mutex> lock(mu);
    HostPipe& p = pipes[dev];
    void* cur = current_context();
    if (!p.in || cur == nullptr || cur != p.ctx) {
        HostPipe n;
        const unsigned ef = cudaEventDisableTiming;
        if ((e = cudaStreamCreateWithFlags(&n.in, cudaStreamNonBlocking)) != cudaSuccess ||
            (e = cudaStreamCreateWithFlags(&n.out, cudaStreamNonBlocking)) != cudaSuccess ||
            (e = cudaEventCreateWithFlags(&n.start, ef)) != cudaSuccess ||
            (e = cudaEventCreateWithFlags(&n.done, ef)) != cudaSuccess)
            return e;
        for (int c = 0; c <= MOEVIE_HOST_MAX_CHUNKS; ++c)
            if ((e = cudaEventCreateWithFlags(&n.ev_in[c], ef)) != cudaSuccess ||
                (e = cudaEventCreateWithFlags(&n.ev_out[c], ef)) != cudaSuccess)
                return e;
        n.ctx = current_context();
        p = n;
    }
    *out = &p;
    return cudaSuccess;
}

}  // namespace

extern "C" {

moevie_status moevie_moe_forward_host(const moevie_layer* layer, const void* x_host, int64_t T, void* y_host,
                                      void* x_dev, void* y_dev, int64_t chunks, void* ws, size_t ws_bytes,
                                      void* stream) {
    if (!layer) return MOEVIE_ERR_INVALID_ARG;
    const int64_t d = layer->d;
    moevie_status c = check_sizes(T, d, layer->E, layer->k, layer->h, layer->h_s);
    if (c != MOEVIE_OK) return c;
    if (chunks < 1 || chunks > MOEVIE_HOST_MAX_CHUNKS) return MOEVIE_ERR_UNSUPPORTED;
    if (T == 0) return MOEVIE_OK;
    if (!x_host || !y_host || !x_dev || !y_dev || !ws || !a16(x_dev) || !a16(y_dev)) return MOEVIE_ERR_INVALID_ARG;
    const int64_t Tc = (T + chunks - 1) / chunks;   // tokens per chunk
    if (ws_bytes < make_layout(Tc, d, layer->E, layer->k, layer->h, layer->h_s).total) return MOEVIE_ERR_WORKSPACE;
    // the pieces the layer runs on: with several chunks a half chunk first, whole chunks,
    // and what is left last (another half chunk when Tc divides T), so that the first
    // copy in and the last copy out, the two no layer hides, are half as long
    int64_t bnd[MOEVIE_HOST_MAX_CHUNKS + 2];
    int64_t n_chunks = 0;
    bnd[0] = 0;
    if (chunks == 1) {
        bnd[++n_chunks] = T;
    } else {
        int64_t t = std::min(T, (Tc + 1) / 2);
        bnd[++n_chunks] = t;
        while (t < T) {
            t = std::min(T, t + Tc);
            bnd[++n_chunks] = t;
        }
    }
    HostPipe* p = nullptr;
    MV_TRY(host_pipe(&p));
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const size_t row_bytes = 2 * (size_t)d;
    const uint8_t* xh = static_cast<const uint8_t*>(x_host);
    uint8_t* yh = static_cast<uint8_t*>(y_host);
    uint8_t* xd = static_cast<uint8_t*>(x_dev);
    uint8_t* yd = static_cast<uint8_t*>(y_dev);
    // the copies into x_dev wait for the work already on `stream` (an earlier call's chunks
    // still reading x_dev); every chunk's rows are copied in, back to back
    MV_TRY(cudaEventRecord(p->start, s));
    MV_TRY(cudaStreamWaitEvent(p->in, p->start, 0));
    for (int64_t i = 0; i < n_chunks; ++i) {
        const int64_t t0 = bnd[i], n = bnd[i + 1] - bnd[i];
        MV_TRY(cudaMemcpyAsync(xd + t0 * row_bytes, xh + t0 * row_bytes, n * row_bytes, cudaMemcpyHostToDevice,
                               p->in));
        MV_TRY(cudaEventRecord(p->ev_in[i], p->in));
    }
    // each chunk's layer once its rows are in, its rows of y out once it is done
    for (int64_t i = 0; i < n_chunks; ++i) {
        const int64_t t0 = bnd[i], n = bnd[i + 1] - bnd[i];
        MV_TRY(cudaStreamWaitEvent(s, p->ev_in[i], 0));
        if ((c = forward_impl(layer, xd + t0 * row_bytes, n, yd + t0 * row_bytes, nullptr, ws, ws_bytes, stream,
                              nullptr, 0)) != MOEVIE_OK)
            return c;
        MV_TRY(cudaEventRecord(p->ev_out[i], s));
        MV_TRY(cudaStreamWaitEvent(p->out, p->ev_out[i], 0));
        MV_TRY(cudaMemcpyAsync(yh + t0 * row_bytes, yd + t0 * row_bytes, n * row_bytes, cudaMemcpyDeviceToHost,
                               p->out));
    }
    // `stream` completes after the last copy out
    MV_TRY(cudaEventRecord(p->done, p->out));
    MV_TRY(cudaStreamWaitEvent(s, p->done, 0));
    return MOEVIE_OK;
}

moevie_status moevie_get_device_status(const void* ws, void* stream, moevie_status* out,
                                       int32_t* detail) {
    if (!ws || !out) return MOEVIE_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return MOEVIE_ERR_CUDA;
    int32_t v[4];
    if (cudaMemcpy(v, ws, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return MOEVIE_ERR_CUDA;
    *out = v[0];
    if (detail) memcpy(detail, v, sizeof v);
    return MOEVIE_OK;
}

// ------------------------------------------------------------ training path

}  // extern "C"

namespace {

// Workspace of moevie_moe_backward.  Expert segments are padded to multiples of 64 rows
// (rows_max = T k + 63 E bounds the padded total), so that the weight-gradient GEMMs'
// K blocks never straddle two experts.
struct BwdLayout {
    size_t status, wsplit, wrt, wpart, wexp, sig, gate, hist, counts, offsets, tiles, n_tiles, perm,
        inv, poff, ptok, pgate, slot_prow, ptiles, n_ptiles, dx_items, n_dx_items, it2, n_it2, it1, n_it1,
        itr, n_itr, H, U, DU, V, DV, Gm, Xp, dgp, DS, dwr, its2, n_its2, its1, n_its1, Hs, Us, DUs, Vs, DVs,
        gc2, gc1, gcr, gcs2, gcs1;   // per group of each item set: 1 = its gradient is cleared first
    int64_t rows_max, max_it2, max_it1, max_itr, max_its2, max_its1;
    int nt_h;
    size_t total;
};

BwdLayout make_bwd_layout(int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t hs, bool swiglu) {
    BwdLayout L;
    size_t o = 0;
    auto take = [&](size_t bytes) {
        const size_t at = o;
        o += up256(bytes);
        return at;
    };
    const int64_t n = T * k, Ep = route_epad((int)E), dp = route_dpad((int)d), hp = row_ld(h);
    L.rows_max = n + 63 * E;
    int bn_d = 0, nt_d = 0, bn_h = 0, bn_e = 0, nt_e = 0;
    choose_bn((int)d, &bn_d, &nt_d);
    choose_bn((int)h, &bn_h, &L.nt_h);
    choose_bn((int)Ep, &bn_e, &nt_e);
    L.max_it2 = bwd_max_items(L.rows_max, (int)E, (int)h, (int)d, bn_d);
    L.max_it1 = bwd_max_items(L.rows_max, (int)E, (int)d, (int)h, bn_h);
    L.max_itr = bwd_max_items(T, 1, (int)d, (int)Ep, bn_e);
    int bn_s = 0, nt_s = 0;
    if (hs > 0) choose_bn((int)hs, &bn_s, &nt_s);
    L.max_its2 = hs > 0 ? bwd_max_items(T, 1, (int)hs, (int)d, bn_d) : 0;   // dWs2 [h_s, d]
    L.max_its1 = hs > 0 ? bwd_max_items(T, 1, (int)d, (int)hs, bn_s) : 0;   // dWs1 [d, h_s]
    L.status = take(sizeof(DevStatus));
    L.wsplit = take(2 * 2 * dp * Ep);
    L.wrt = take(4 * E * dp);
    L.wpart = take(4 * 2 * (int64_t)route_split_parts((int)d) * Ep);
    L.wexp = take(4 * (int64_t)route_split_parts((int)d) * Ep);
    L.sig = take(4 * n);
    L.gate = take(4 * n);
    L.hist = take(4 * ((n + 255) / 256) * E);
    L.counts = take(4 * E);
    L.offsets = take(4 * (E + 1));
    L.tiles = take(16 * max_mtiles(n, E));
    L.n_tiles = take(4);
    L.perm = take(4 * n);
    L.inv = take(4 * n);
    L.poff = take(4 * (E + 1));
    L.ptok = take(4 * L.rows_max);
    L.pgate = take(4 * L.rows_max);
    L.slot_prow = take(4 * n);
    L.ptiles = take(16 * max_mtiles(L.rows_max, E));
    L.n_ptiles = take(4);
    L.dx_items = take(16 * max_mtiles(L.rows_max, E) * nt_d);   // band-ordered dx GEMM items
    L.n_dx_items = take(4);
    L.it2 = take(16 * L.max_it2);
    L.n_it2 = take(4);
    L.it1 = take(16 * L.max_it1);
    L.n_it1 = take(4);
    L.itr = take(16 * L.max_itr);
    L.n_itr = take(4);
    L.gc2 = take(4 * E);
    L.gc1 = take(4 * E);
    L.gcr = take(4);
    L.gcs2 = take(4);
    L.gcs1 = take(4);
    L.H = take(2 * L.rows_max * hp);
    L.U = take(2 * L.rows_max * hp);
    L.DU = take(2 * L.rows_max * hp);
    L.V = swiglu ? take(2 * L.rows_max * hp) : 0;    // SwiGLU: the up projection's pre-activation
    L.DV = swiglu ? take(2 * L.rows_max * hp) : 0;   //   and its gradient
    L.Gm = take(2 * L.rows_max * d);
    L.Xp = take(2 * L.rows_max * d);
    L.dgp = take(4 * 2 * (int64_t)L.nt_h * L.rows_max);
    L.DS = take(2 * T * Ep);
    L.dwr = take(4 * d * Ep);
    if (hs > 0) {   // the shared expert: every token, one dense group of h_s hidden units
        const int64_t hsp = row_ld(hs);
        L.its2 = take(16 * L.max_its2);
        L.n_its2 = take(4);
        L.its1 = take(16 * L.max_its1);
        L.n_its1 = take(4);
        L.Hs = take(2 * T * hsp);
        L.Us = take(2 * T * hsp);
        L.DUs = take(2 * T * hsp);
        L.Vs = swiglu ? take(2 * T * hsp) : 0;
        L.DVs = swiglu ? take(2 * T * hsp) : 0;
    }
    L.total = o;
    return L;
}

moevie_status check_bwd_sizes(int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t hs) {
    moevie_status c = check_sizes(T, d, E, k, h, hs);
    if (c != MOEVIE_OK) return c;
    if (h <= 0 || k > 32 || d > 65535 || h > 65535 || hs > 65535 || T * k + 63 * E >= (int64_t(1) << 31))
        return MOEVIE_ERR_UNSUPPORTED;
    return MOEVIE_OK;
}

}  // namespace

extern "C" {

moevie_status moevie_backward_workspace_size(int64_t T_max, int64_t d, int64_t E, int64_t k, int64_t h,
                                             int64_t h_s, int swiglu, size_t* bytes) {
    if (!bytes) return MOEVIE_ERR_INVALID_ARG;
    const moevie_status c = check_bwd_sizes(T_max, d, E, k, h, h_s);
    if (c != MOEVIE_OK) return c;
    *bytes = make_bwd_layout(T_max, d, E, k, h, h_s, swiglu != 0).total;
    return MOEVIE_OK;
}

moevie_status moevie_moe_backward(const moevie_layer* Lr, const void* x, const void* dy, int64_t T,
                                  const int32_t* idx, float* dx, float* dW_r, float* dW1, float* dW2,
                                  float* dW3, float* dWs1, float* dWs2, float* dWs3, void* ws, size_t ws_bytes,
                                  void* stream) {
    if (!Lr) return MOEVIE_ERR_INVALID_ARG;
    const int64_t d = Lr->d, E = Lr->E, k = Lr->k, h = Lr->h, hs = Lr->h_s;
    moevie_status c = check_bwd_sizes(T, d, E, k, h, hs);
    if (c != MOEVIE_OK) return c;
    const bool swiglu = Lr->W3 != nullptr;
    const bool shared = hs > 0;
    if (T == 0) return MOEVIE_OK;
    if (!x || !dy || !idx || !dx || !dW_r || !dW1 || !dW2 || !ws || !Lr->W_r || !Lr->W1 || !Lr->W2)
        return MOEVIE_ERR_INVALID_ARG;
    if (swiglu && (!dW3 || !a16(dW3) || !a16(Lr->W3))) return MOEVIE_ERR_INVALID_ARG;
    if (!a16(x) || !a16(dy) || !a16(idx) || !a16(dx) || !a16(dW1) || !a16(dW2) || !a16(ws) || !a16(Lr->W1) ||
        !a16(Lr->W2))
        return MOEVIE_ERR_INVALID_ARG;
    if (shared) {   // the shared expert's weights and gradients (Ws3, dWs3 with SwiGLU experts)
        if (!Lr->Ws1 || !Lr->Ws2 || !dWs1 || !dWs2 || !a16(Lr->Ws1) || !a16(Lr->Ws2) || !a16(dWs1) ||
            !a16(dWs2))
            return MOEVIE_ERR_INVALID_ARG;
        if (swiglu && (!Lr->Ws3 || !dWs3 || !a16(Lr->Ws3) || !a16(dWs3))) return MOEVIE_ERR_INVALID_ARG;
    }
    const BwdLayout L = make_bwd_layout(T, d, E, k, h, hs, swiglu);
    if (ws_bytes < L.total) return MOEVIE_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    DevStatus* st = at<DevStatus>(ws, L.status);
    const int64_t n = T * k, Ep = route_epad((int)E), dp = route_dpad((int)d), hp = row_ld(h);
    const __nv_bfloat16* xb = static_cast<const __nv_bfloat16*>(x);
    float* wrt = at<float>(ws, L.wrt);
    int32_t* poff = at<int32_t>(ws, L.poff);
    int32_t* ptok = at<int32_t>(ws, L.ptok);
    float* pgate = at<float>(ws, L.pgate);
    void* H = at<void>(ws, L.H);
    void* U = at<void>(ws, L.U);
    void* DU = at<void>(ws, L.DU);
    void* V = swiglu ? at<void>(ws, L.V) : nullptr;
    void* DV = swiglu ? at<void>(ws, L.DV) : nullptr;
    void* Gm = at<void>(ws, L.Gm);
    void* Xp = at<void>(ws, L.Xp);
    float* dgp = at<float>(ws, L.dgp);
    __nv_bfloat16* DS = at<__nv_bfloat16>(ws, L.DS);
    float* dwr = at<float>(ws, L.dwr);
    int bn_d = 0, nt_d = 0, bn_h = 0, nt_h = 0, bn_e = 0, nt_e = 0;
    choose_bn((int)d, &bn_d, &nt_d);
    choose_bn((int)h, &bn_h, &nt_h);
    choose_bn((int)Ep, &bn_e, &nt_e);

    // 1. W_r's transposed fp32 copy (the router's split kernel), the gates of the held
    //    selection (Eqs. 4-5), and the stable expert-major order (Algorithm 1, phase 1)
    MV_TRY(launch_route_split(Lr->W_r, (int)d, (int)E, at<__nv_bfloat16>(ws, L.wsplit), wrt,
                              at<float>(ws, L.wpart), at<int32_t>(ws, L.wexp), st, s));
    MV_TRY(launch_bwd_gates(xb, wrt, (int)dp, idx, T, (int)d, (int)E, (int)k, at<float>(ws, L.sig),
                            at<float>(ws, L.gate), st, s));
    MV_TRY(launch_permute(idx, n, (int)k, (int)E, GM_BM, perm_chunk(n, num_sms()), nullptr,
                          at<int32_t>(ws, L.hist), at<int32_t>(ws, L.counts), at<int32_t>(ws, L.offsets),
                          at<int4>(ws, L.tiles), at<int32_t>(ws, L.n_tiles), at<int32_t>(ws, L.perm),
                          at<int32_t>(ws, L.inv), nullptr, nullptr, st, s));
    // 2. segments padded to 64 rows: row maps, m-tiles, weight-gradient items
    MV_TRY(launch_bwd_pad(at<int32_t>(ws, L.counts), (int)E, poff, s));
    MV_TRY(launch_bwd_rows(idx, at<int32_t>(ws, L.inv), at<int32_t>(ws, L.counts), at<int32_t>(ws, L.offsets),
                           poff, at<float>(ws, L.gate), n, (int)k, (int)E, ptok, pgate,
                           at<int32_t>(ws, L.slot_prow), s));
    MV_TRY(launch_tile_table(poff, (int)E, GM_BM, at<int4>(ws, L.ptiles), at<int32_t>(ws, L.n_ptiles), s));
    MV_TRY(launch_bwd_items(poff, (int)E, 0, (int)h, (int)d, bn_d, (int)L.max_it2, at<int4>(ws, L.it2),
                            at<int32_t>(ws, L.n_it2), at<int32_t>(ws, L.gc2), st, s));
    MV_TRY(launch_bwd_items(poff, (int)E, 0, (int)d, (int)h, bn_h, (int)L.max_it1, at<int4>(ws, L.it1),
                            at<int32_t>(ws, L.n_it1), at<int32_t>(ws, L.gc1), st, s));
    MV_TRY(launch_bwd_items(nullptr, 1, T, (int)d, (int)Ep, bn_e, (int)L.max_itr, at<int4>(ws, L.itr),
                            at<int32_t>(ws, L.n_itr), at<int32_t>(ws, L.gcr), st, s));
    int bn_s = 0, nt_s = 0;
    const int64_t hsp = shared ? row_ld(hs) : 0;
    if (shared) {
        choose_bn((int)hs, &bn_s, &nt_s);
        MV_TRY(launch_bwd_items(nullptr, 1, T, (int)hs, (int)d, bn_d, (int)L.max_its2, at<int4>(ws, L.its2),
                                at<int32_t>(ws, L.n_its2), at<int32_t>(ws, L.gcs2), st, s));
        MV_TRY(launch_bwd_items(nullptr, 1, T, (int)d, (int)hs, bn_s, (int)L.max_its1, at<int4>(ws, L.its1),
                                at<int32_t>(ws, L.n_its1), at<int32_t>(ws, L.gcs1), st, s));
    }
    // 3. accumulators cleared (of the weight gradients only what their items will add
    //    into, or not write at all); gathered copies of x and g dy
    const int sms = num_sms();
    MV_TRY(launch_zero_f32(dx, T * d, s));
    MV_TRY(launch_bwd_zero(at<int32_t>(ws, L.gc1), (int)E, (int)d, (int)h, hp, dW1, sms, s));
    MV_TRY(launch_bwd_zero(at<int32_t>(ws, L.gc2), (int)E, (int)h, (int)d, d, dW2, sms, s));
    if (swiglu) MV_TRY(launch_bwd_zero(at<int32_t>(ws, L.gc1), (int)E, (int)d, (int)h, hp, dW3, sms, s));
    if (shared) {
        MV_TRY(launch_bwd_zero(at<int32_t>(ws, L.gcs1), 1, (int)d, (int)hs, hsp, dWs1, sms, s));
        MV_TRY(launch_bwd_zero(at<int32_t>(ws, L.gcs2), 1, (int)hs, (int)d, d, dWs2, sms, s));
        if (swiglu) MV_TRY(launch_bwd_zero(at<int32_t>(ws, L.gcs1), 1, (int)d, (int)hs, hsp, dWs3, sms, s));
    }
    MV_TRY(launch_bwd_zero(at<int32_t>(ws, L.gcr), 1, (int)d, (int)Ep, Ep, dwr, sms, s));
    MV_TRY(launch_zero_f32(reinterpret_cast<float*>(DS), T * Ep / 2, s));
    MV_TRY(launch_bwd_gather(xb, static_cast<const __nv_bfloat16*>(dy), ptok, pgate, poff, (int)E, (int)d,
                             L.rows_max, static_cast<__nv_bfloat16*>(Xp), static_cast<__nv_bfloat16*>(Gm), s));
    // 4. up-projection again: u = x W1[e] and a = GELU(u), both kept (bf16; SwiGLU: u, v and a)
    {
        GemmSpec g{};
        g.A = x;
        g.lda = d;
        g.a_rows = ptok;
        g.a_div = 1;
        g.a_nrows = T;
        g.a_neg_zero = 1;
        g.m_total = L.rows_max;
        g.tiles = at<int4>(ws, L.ptiles);
        g.n_tiles = at<int32_t>(ws, L.n_ptiles);
        g.G = (int)E;
        g.W = Lr->W1;
        g.K = (int)d;
        g.N = (int)h;
        g.N_ld = hp;
        g.epi = EPI_GELU2_BF16;
        if (swiglu) {   // a = SiLU(u) v with u = x W1[e] (gate), v = x W3[e] (up); u and v kept
            g.epi = EPI_SWIGLU_BF16;
            g.W3 = Lr->W3;
            g.out3 = V;
        }
        g.out = H;
        g.out2 = U;
        g.ldo = hp;
        if ((c = run_gemm(g, st, s)) != MOEVIE_OK) return c;
    }
    // 5. da' = dy W2[e]^T (K-major W2), epilogue du = g da' GELU'(u) and dg = da' . a
    {
        GemmSpec g{};
        g.A = dy;
        g.lda = d;
        g.a_rows = ptok;
        g.a_div = 1;
        g.a_nrows = T;
        g.a_neg_zero = 1;
        g.m_total = L.rows_max;
        g.tiles = at<int4>(ws, L.ptiles);
        g.n_tiles = at<int32_t>(ws, L.n_ptiles);
        g.G = (int)E;
        g.W = Lr->W2;
        g.b_kmajor = 1;
        g.b_k_ld = d;
        g.b_g_ld = h * d;
        g.K = (int)d;
        g.N = (int)h;
        g.N_ld = hp;
        g.epi = swiglu ? EPI_DSWIGLU_BF16 : EPI_DGELU_BF16;
        g.row_scale = pgate;
        g.epi_u = U;
        g.epi_v = V;
        g.epi_a = H;
        g.out = DU;
        g.out2 = DV;
        g.ldo = hp;
        g.dg_part = dgp;
        if ((c = run_gemm(g, st, s)) != MOEVIE_OK) return c;
    }
    // 6. dx += du W1[e]^T (K-major W1), scattered to the rows' tokens; band-ordered like the
    //    forward's down-projection when the fp32 dx would not stay in L2
    {
        const BandPlan bp = choose_bands(T, d, E, k, h);
        const bool banded = (bp.nb > 1 || bp.gsz < nt_d) && max_mtiles(L.rows_max, E) <= ITEM_MAX_TILES;
        if (banded)
            MV_TRY(launch_item_order(at<int4>(ws, L.ptiles), at<int32_t>(ws, L.n_ptiles), ptok, T, bp.nb, nt_d,
                                     bp.gsz, bn_d, (int)max_mtiles(L.rows_max, E), at<int4>(ws, L.dx_items),
                                     at<int32_t>(ws, L.n_dx_items), s));
        for (int pass = 0; pass < (swiglu ? 2 : 1); ++pass) {   // du W1^T, then dv W3^T (SwiGLU)
            GemmSpec g{};
            g.A = pass ? DV : DU;
            g.lda = hp;
            g.a_cols = h;
            g.a_nrows = L.rows_max;
            g.m_total = L.rows_max;
            g.tiles = banded ? at<int4>(ws, L.dx_items) : at<int4>(ws, L.ptiles);
            g.n_tiles = banded ? at<int32_t>(ws, L.n_dx_items) : at<int32_t>(ws, L.n_ptiles);
            g.item_table = banded ? 1 : 0;
            g.G = (int)E;
            g.W = pass ? Lr->W3 : Lr->W1;
            g.b_kmajor = 1;
            g.b_k_ld = hp;
            g.b_g_ld = d * hp;
            g.K = (int)h;
            g.N = (int)d;
            g.epi = EPI_ADD_F32;
            g.yacc = dx;
            g.ldy = d;
            g.o_nrows = T;
            g.o_rows = ptok;
            g.o_div = 1;
            g.o_neg_skip = 1;
            g.scale = 1.0f;
            if ((c = run_gemm(g, st, s)) != MOEVIE_OK) return c;
        }
    }
    // 7. the router (Eqs. 4-5): ds per token, dx += ds W_r^T, ds into [T][E_pad] bf16
    MV_TRY(launch_bwd_router(idx, at<float>(ws, L.sig), at<float>(ws, L.gate), at<int32_t>(ws, L.slot_prow), dgp,
                             2 * nt_h, L.rows_max, wrt, (int)dp, T, (int)d, (int)E, (int)k, (int)Ep, dx, DS, s));
    // 8. weight gradients, per expert over its padded rows: dW2[e] = a^T (g dy),
    //    dW1[e] = x^T du; and dW_r = x^T ds over all tokens
    auto wgrad = [&](const void* A, int64_t a_cols, int64_t a_rows, int64_t lda, const void* B, int64_t N,
                     int64_t n_ld, int64_t b_rows, int G, int M, size_t items, size_t n_items, int64_t max_items,
                     float* out, int64_t ldy, float scale = 1.0f) {
        GemmSpec g{};
        g.A = A;
        g.a_mn = 1;
        g.a_cols = a_cols;
        g.a_nrows = a_rows;
        g.lda = lda;
        g.W = B;
        g.N = (int)N;
        g.N_ld = n_ld;
        g.b_rows = b_rows;
        g.K = 64;
        g.G = G;
        g.wg_M = M;
        g.item_table = 2;
        g.tiles = at<int4>(ws, items);
        g.n_tiles = at<int32_t>(ws, n_items);
        g.max_items = max_items;
        g.m_total = (int64_t)G * M;
        g.epi = EPI_ADD_F32;
        g.yacc = out;
        g.ldy = ldy;
        g.o_nrows = (int64_t)G * M;
        g.scale = scale;
        return run_gemm(g, st, s);
    };
    if ((c = wgrad(H, h, L.rows_max, hp, Gm, d, d, L.rows_max, (int)E, (int)h, L.it2, L.n_it2, L.max_it2, dW2,
                   d)) != MOEVIE_OK)
        return c;
    if ((c = wgrad(Xp, d, L.rows_max, d, DU, h, hp, L.rows_max, (int)E, (int)d, L.it1, L.n_it1, L.max_it1, dW1,
                   hp)) != MOEVIE_OK)
        return c;
    if (swiglu && (c = wgrad(Xp, d, L.rows_max, d, DV, h, hp, L.rows_max, (int)E, (int)d, L.it1, L.n_it1,
                             L.max_it1, dW3, hp)) != MOEVIE_OK)   // dW3[e] = x^T dv
        return c;
    if ((c = wgrad(x, d, T, d, DS, Ep, Ep, T, 1, (int)d, L.itr, L.n_itr, L.max_itr, dwr, Ep)) != MOEVIE_OK)
        return c;
    MV_TRY(launch_bwd_copy(dwr, Ep, dW_r, d, E, s));
    if (!shared) return MOEVIE_OK;
    // 9. the shared expert (Eq. 6, second term), every token with the constant weight lambda,
    //    one dense group of h_s hidden units through the same GEMMs: u_s = x Ws1 and a_s again,
    //    du_s = lambda (dy Ws2^T) GELU'(u_s) (SwiGLU: du_s, dv_s), dx += du_s Ws1^T (+ dv_s Ws3^T),
    //    dWs2 = lambda a_s^T dy, dWs1 = x^T du_s, dWs3 = x^T dv_s
    void* Hs = at<void>(ws, L.Hs);
    void* Us = at<void>(ws, L.Us);
    void* DUs = at<void>(ws, L.DUs);
    void* Vs = swiglu ? at<void>(ws, L.Vs) : nullptr;
    void* DVs = swiglu ? at<void>(ws, L.DVs) : nullptr;
    {
        GemmSpec g{};
        g.A = x;
        g.lda = d;
        g.a_ident = 1;
        g.a_nrows = T;
        g.m_total = T;
        g.G = 1;
        g.W = Lr->Ws1;
        g.K = (int)d;
        g.N = (int)hs;
        g.N_ld = hsp;
        g.epi = EPI_GELU2_BF16;
        if (swiglu) {
            g.epi = EPI_SWIGLU_BF16;
            g.W3 = Lr->Ws3;
            g.out3 = Vs;
        }
        g.out = Hs;
        g.out2 = Us;
        g.ldo = hsp;
        if ((c = run_gemm(g, st, s)) != MOEVIE_OK) return c;
    }
    {
        GemmSpec g{};
        g.A = dy;
        g.lda = d;
        g.a_ident = 1;
        g.a_nrows = T;
        g.m_total = T;
        g.G = 1;
        g.W = Lr->Ws2;
        g.b_kmajor = 1;
        g.b_k_ld = d;
        g.b_g_ld = hs * d;
        g.K = (int)d;
        g.N = (int)hs;
        g.N_ld = hsp;
        g.epi = swiglu ? EPI_DSWIGLU_BF16 : EPI_DGELU_BF16;
        g.scale = Lr->lambda;
        g.epi_u = Us;
        g.epi_v = Vs;
        g.epi_a = Hs;
        g.out = DUs;
        g.out2 = DVs;
        g.ldo = hsp;
        if ((c = run_gemm(g, st, s)) != MOEVIE_OK) return c;
    }
    for (int pass = 0; pass < (swiglu ? 2 : 1); ++pass) {
        GemmSpec g{};
        g.A = pass ? DVs : DUs;
        g.lda = hsp;
        g.a_cols = hs;
        g.a_nrows = T;
        g.m_total = T;
        g.G = 1;
        g.W = pass ? Lr->Ws3 : Lr->Ws1;
        g.b_kmajor = 1;
        g.b_k_ld = hsp;
        g.b_g_ld = d * hsp;
        g.K = (int)hs;
        g.N = (int)d;
        g.epi = EPI_ADD_F32;
        g.yacc = dx;
        g.ldy = d;
        g.o_nrows = T;
        g.scale = 1.0f;
        if ((c = run_gemm(g, st, s)) != MOEVIE_OK) return c;
    }
    if ((c = wgrad(Hs, hs, T, hsp, dy, d, d, T, 1, (int)hs, L.its2, L.n_its2, L.max_its2, dWs2, d,
                   Lr->lambda)) != MOEVIE_OK)
        return c;
    if ((c = wgrad(x, d, T, d, DUs, hs, hsp, T, 1, (int)d, L.its1, L.n_its1, L.max_its1, dWs1, hsp)) !=
        MOEVIE_OK)
        return c;
    if (swiglu && (c = wgrad(x, d, T, d, DVs, hs, hsp, T, 1, (int)d, L.its1, L.n_its1, L.max_its1, dWs3,
                             hsp)) != MOEVIE_OK)
        return c;
    return MOEVIE_OK;
}

// ------------------------------------------------------------ test hooks

moevie_status moevie_test_route_logits(const void* x, const float* W_r, int64_t T, int64_t d,
                                       int64_t E, float* s_out, void* ws, size_t ws_bytes,
                                       void* stream) {
    moevie_status c = check_sizes(T, d, E, 1, 0, 0);
    if (c != MOEVIE_OK) return c;
    if (T == 0) return MOEVIE_OK;
    if (!x || !W_r || !s_out || !ws || !a16(x) || !a16(ws) || !a16(s_out)) return MOEVIE_ERR_INVALID_ARG;
    const Layout L = make_layout(T, d, E, 1, 0, 0);
    if (ws_bytes < L.total) return MOEVIE_ERR_WORKSPACE;
    // s_out receives the padded [T, route_epad(E)] logits
    return route_impl(x, W_r, nullptr, T, d, E, 1, nullptr, nullptr, L, ws,
                      static_cast<cudaStream_t>(stream), true, s_out);
}

moevie_status moevie_test_fallback_count(const void* ws, void* stream, int32_t* out) {
    if (!ws || !out) return MOEVIE_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(static_cast<cudaStream_t>(stream)) != cudaSuccess) return MOEVIE_ERR_CUDA;
    DevStatus h;
    if (cudaMemcpy(&h, ws, sizeof h, cudaMemcpyDeviceToHost) != cudaSuccess) return MOEVIE_ERR_CUDA;
    *out = h.fb_count;
    return MOEVIE_OK;
}

moevie_status moevie_test_expert_hidden(const void* x, const int32_t* perm, const int32_t* offsets,
                                        const void* W1, int64_t T, int64_t d, int64_t h, int64_t E,
                                        int64_t k, void* hidden, void* ws, size_t ws_bytes,
                                        void* stream) {
    moevie_status c = check_sizes(T, d, E, k, h, 0);
    if (c != MOEVIE_OK) return c;
    if (h == 0) return MOEVIE_ERR_UNSUPPORTED;
    if (T == 0) return MOEVIE_OK;
    if (!x || !perm || !offsets || !W1 || !hidden || !ws) return MOEVIE_ERR_INVALID_ARG;
    if (!a16(x) || !a16(W1) || !a16(hidden) || !a16(ws)) return MOEVIE_ERR_INVALID_ARG;
    const Layout L = make_layout(T, 0, E, k, 0, 0);
    if (ws_bytes < L.total) return MOEVIE_ERR_WORKSPACE;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    int4* tiles = at<int4>(ws, L.tiles);
    int32_t* n_tiles = at<int32_t>(ws, L.n_tiles);
    MV_TRY(launch_tile_table(offsets, (int)E, GM_BM, tiles, n_tiles, s));
    return expert_up(x, perm, (int)k, tiles, n_tiles, W1, T, d, h, E, k, hidden,
                     at<DevStatus>(ws, L.status), s);
}

moevie_status moevie_test_moe_forward_events(const moevie_layer* layer, const void* x, int64_t T,
                                             void* y, void* ws, size_t ws_bytes, void* stream,
                                             void* const* events, int n_events) {
    if (!events) return MOEVIE_ERR_INVALID_ARG;
    return forward_impl(layer, x, T, y, nullptr, ws, ws_bytes, stream, events, n_events);
}

moevie_status moevie_test_wait_timeout(void* ws, size_t ws_bytes, uint64_t limit_ns, void* stream) {
    if (!ws || ws_bytes < sizeof(DevStatus) || !a16(ws)) return MOEVIE_ERR_INVALID_ARG;
    if (limit_ns == 0 || limit_ns > 10000000000ull) return MOEVIE_ERR_INVALID_ARG;
    return cuda_status(launch_wait_probe(static_cast<DevStatus*>(ws), limit_ns,
                                         static_cast<cudaStream_t>(stream)));
}

}  // extern "C"
