// permute.cu -- expert-major order of the flat routing slots (App. B, Algorithm 1,
// phase 1: Sort by expert id, index = pos // K, BinCount, CumSum), sm_103a.
//
// A stable counting sort over chunks of flat slots (about two chunks per SM):
//   perm_hist_kernel    per-chunk histograms (16-byte vector loads of idx), stored
//                       expert-major: hist[e][chunk]
//   perm_chunk_scan_kernel  one warp per expert: exclusive scan over its chunks
//                       (each chunk's first row inside the expert's segment) and
//                       the expert's count
//   perm_offsets_kernel exclusive offsets over experts and the m-tile table used
//                       by the grouped GEMMs (one CTA)
//   perm_scatter_kernel stages its chunk in shared memory (16-byte loads), ranks
//                       every slot among the earlier slots of the same expert
//                       (warp match + per-warp running counts), and writes perm,
//                       inv and the per-row token (pos // K) and gate.
// Inside one expert's segment, rows keep ascending slot order t*k + j.
#include <atomic>
#include <mutex>

#include "internal.h"

namespace mv {

namespace {

constexpr int PT = 256;                      // threads per CTA
constexpr int PW = PT / 32;                  // warps per CTA

__device__ __forceinline__ bool valid_id(int e, int E) { return e >= 0 && e < E; }

// Histogram of chunk b (of nchunks) into hist[e][b]; cnt: E ints of shared memory.
__device__ __forceinline__ void perm_hist_body(const int32_t* __restrict__ idx, int64_t n, int E,
                                               int chunk, int b, int nchunks,
                                               int32_t* __restrict__ hist, DevStatus* st,
                                               int32_t* cnt) {
    for (int e = threadIdx.x; e < E; e += PT) cnt[e] = 0;
    __syncthreads();
    const int64_t c0 = (int64_t)b * chunk;
    const int64_t c1 = c0 + chunk < n ? c0 + chunk : n;
    const int64_t nvec = (c1 - c0) >> 2;
    const int4* v = reinterpret_cast<const int4*>(idx + c0);   // c0 % 4 == 0, idx 16-B aligned
    for (int64_t i = threadIdx.x; i < nvec; i += PT) {
        const int4 q = v[i];
        const int e4[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            if (valid_id(e4[j], E)) atomicAdd(&cnt[e4[j]], 1);
            else report(st, MOEVIE_ERR_DEVICE, SITE_PERMUTE_ID, (int)(c0 + 4 * i + j), e4[j]);
        }
    }
    for (int64_t i = c0 + 4 * nvec + threadIdx.x; i < c1; i += PT) {
        const int e = idx[i];
        if (valid_id(e, E)) atomicAdd(&cnt[e], 1);
        else report(st, MOEVIE_ERR_DEVICE, SITE_PERMUTE_ID, (int)i, e);
    }
    __syncthreads();
    for (int e = threadIdx.x; e < E; e += PT) hist[(int64_t)e * nchunks + b] = cnt[e];
}

__global__ void __launch_bounds__(PT) perm_hist_kernel(const int32_t* __restrict__ idx,
                                                       int64_t n, int E, int chunk,
                                                       int32_t* __restrict__ hist,
                                                       DevStatus* st) {
    pdl_wait();
    extern __shared__ int32_t cnt[];
    perm_hist_body(idx, n, E, chunk, blockIdx.x, gridDim.x, hist, st, cnt);
}

// Exclusive scan of one int per thread over the block (up to 1024 threads).
__device__ int block_exclusive_scan_1024(int v, int* total) {
    __shared__ int wsum[32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int inc = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int u = __shfl_up_sync(0xffffffffu, inc, o);
        if (lane >= o) inc += u;
    }
    if (lane == 31) wsum[warp] = inc;
    __syncthreads();
    if (warp == 0) {
        const int w = lane < (int)(blockDim.x >> 5) ? wsum[lane] : 0;
        int wi = w;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(0xffffffffu, wi, o);
            if (lane >= o) wi += u;
        }
        wsum[lane] = wi - w;
        if (lane == 31) *total = wi;
    }
    __syncthreads();
    const int r = wsum[warp] + inc - v;
    __syncthreads();
    return r;
}

// One warp per expert: hist[e][0 .. nchunks) becomes its exclusive prefix (the first
// row of expert e inside each chunk, relative to the expert's segment); counts[e] is
// the total.  Coalesced: lanes over consecutive chunks.
__device__ __forceinline__ void perm_chunk_scan_warp(int32_t* __restrict__ hist, int nchunks, int e,
                                                     int lane, int32_t* __restrict__ counts) {
    int32_t* h = hist + (int64_t)e * nchunks;
    int running = 0;
    for (int c0 = 0; c0 < nchunks; c0 += 32) {
        const int c = c0 + lane;
        const int v = c < nchunks ? __ldcg(h + c) : 0;   // L2: written by other CTAs
        int inc = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int u = __shfl_up_sync(0xffffffffu, inc, o);
            if (lane >= o) inc += u;
        }
        if (c < nchunks) h[c] = running + inc - v;
        running += __shfl_sync(0xffffffffu, inc, 31);
    }
    if (lane == 0) counts[e] = running;
}

__global__ void __launch_bounds__(256) perm_chunk_scan_kernel(int32_t* __restrict__ hist,
                                                              int nchunks, int E,
                                                              int32_t* __restrict__ counts) {
    pdl_wait();
    const int e = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    if (e >= E) return;
    perm_chunk_scan_warp(hist, nchunks, e, threadIdx.x & 31, counts);
}

// One CTA of 1024 threads (E <= 1024): exclusive offsets over experts, the number
// of bm-row m-tiles, and the m-tile table (warps over experts, lanes over tiles).
__global__ void __launch_bounds__(1024) perm_offsets_kernel(const int32_t* __restrict__ counts,
                                                            int E, int bm,
                                                            int32_t* __restrict__ offsets,
                                                            int4* __restrict__ tiles,
                                                            int32_t* __restrict__ n_tiles) {
    pdl_wait();
    __shared__ int s_total, s_tiles;
    __shared__ int s_cnt[1024], s_off[1024], s_toff[1024];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int e = threadIdx.x;
    const int cnt = e < E ? counts[e] : 0;
    const int off = block_exclusive_scan_1024(cnt, &s_total);
    const int toff = block_exclusive_scan_1024((cnt + bm - 1) / bm, &s_tiles);
    if (e < E) {
        offsets[e] = off;
        s_cnt[e] = cnt;
        s_off[e] = off;
        s_toff[e] = toff;
    }
    if (e == 0) {
        offsets[E] = s_total;
        *n_tiles = s_tiles;
    }
    __syncthreads();
    for (int g = warp; g < E; g += 32) {
        const int c = s_cnt[g], o = s_off[g], to = s_toff[g];
        for (int m = lane; m * bm < c; m += 32)
            tiles[to + m] = make_int4(g, o + m * bm, min(bm, c - m * bm), 0);
    }
}

// Scatter of chunk b: ps_smem holds chunk ints (the chunk's ids) + PW * E ints
// (per-warp counts); offsets may live in global or shared memory.
__device__ __forceinline__ void perm_scatter_body(
    const int32_t* __restrict__ idx, int64_t n, int k, int E, int chunk, int b, int nchunks,
    const int32_t* __restrict__ base, const int32_t* offsets,
    const float* __restrict__ gate_flat, int32_t* __restrict__ perm, int32_t* __restrict__ inv,
    int32_t* __restrict__ row_tok, float* __restrict__ row_gate, int32_t* ps_smem) {
    int32_t* sidx = ps_smem;
    int32_t* wc = ps_smem + chunk;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int per_warp = chunk / PW;
    const int64_t c0 = (int64_t)b * chunk;
    const int len = (int)(c0 + chunk < n ? chunk : n - c0);
    {
        const int nvec = len >> 2;
        const int4* v = reinterpret_cast<const int4*>(idx + c0);
        int4* sv = reinterpret_cast<int4*>(sidx);
        for (int i = tid; i < nvec; i += PT) sv[i] = v[i];
        for (int i = 4 * nvec + tid; i < len; i += PT) sidx[i] = idx[c0 + i];
    }
    for (int i = tid; i < PW * E; i += PT) wc[i] = 0;
    __syncthreads();
    const int wbeg = warp * per_warp;
    const int wend = wbeg + per_warp < len ? wbeg + per_warp : len;
    int32_t* my = wc + warp * E;
    for (int s0 = wbeg; s0 < wend; s0 += 32) {          // pass 1: per-warp histogram
        const int i = s0 + lane;
        int e = (i < wend) ? sidx[i] : -1;
        if (!valid_id(e, E)) e = -1;
        const uint32_t m = __match_any_sync(0xffffffffu, e);
        if (e >= 0 && lane == __ffs(m) - 1) my[e] += __popc(m);
        __syncwarp();
    }
    __syncthreads();
    for (int e = tid; e < E; e += PT) {                  // pass 2: first row per (warp, e)
        int run = offsets[e] + __ldcg(base + (int64_t)e * nchunks + b);   // L2: written by other CTAs
        for (int w = 0; w < PW; ++w) {
            const int c = wc[w * E + e];
            wc[w * E + e] = run;
            run += c;
        }
    }
    __syncthreads();
    const uint32_t lt = (1u << lane) - 1u;
    for (int s0 = wbeg; s0 < wend; s0 += 32) {          // pass 3: stable ranks
        const int i = s0 + lane;
        int e = (i < wend) ? sidx[i] : -1;
        if (!valid_id(e, E)) e = -1;
        const uint32_t m = __match_any_sync(0xffffffffu, e);
        const int first = (e >= 0) ? my[e] : 0;
        __syncwarp();
        if (e >= 0 && lane == __ffs(m) - 1) my[e] = first + __popc(m);
        __syncwarp();
        if (i < wend) {
            const int64_t slot = c0 + i;
            if (e >= 0) {
                const int row = first + __popc(m & lt);
                perm[row] = (int32_t)slot;
                inv[slot] = row;
                if (row_tok) row_tok[row] = (int32_t)(slot / k);
                if (row_gate) row_gate[row] = gate_flat[slot];
            } else {
                inv[slot] = -1;
            }
        }
    }
}

__global__ void __launch_bounds__(PT) perm_scatter_kernel(
    const int32_t* __restrict__ idx, int64_t n, int k, int E, int chunk,
    const int32_t* __restrict__ base, const int32_t* __restrict__ offsets,
    const float* __restrict__ gate_flat, int32_t* __restrict__ perm, int32_t* __restrict__ inv,
    int32_t* __restrict__ row_tok, float* __restrict__ row_gate) {
    pdl_wait();
    extern __shared__ __align__(16) int32_t ps_smem[];
    perm_scatter_body(idx, n, k, E, chunk, blockIdx.x, gridDim.x, base, offsets, gate_flat, perm, inv,
                      row_tok, row_gate, ps_smem);
}

// The whole permute in one cooperative launch (one CTA per chunk, all resident):
// histograms, grid barrier, per-expert chunk scans (warps over experts), grid barrier,
// then every CTA forms the expert offsets in shared memory (CTA 0 also writes offsets,
// the m-tile table and its size) and scatters its chunk.  The barriers are bounded
// (grid_barrier: 2 s, then MOEVIE_ERR_TIMEOUT and the CTA stops).  Launched with
// programmatic stream serialization as well: every CTA first waits (griddepcontrol.wait)
// for the previous kernel to complete, so by the time any CTA reaches a barrier the
// previous kernel has released its SMs and the whole cooperative grid (sized from the
// occupancy of an idle device) is resident; the previous kernel never waits on this
// one, so a late CTA only delays the barrier, it cannot block it.
constexpr uint64_t PERM_BARRIER_LIMIT_NS = 2000000000ull;
__global__ void __launch_bounds__(PT) perm_fused_kernel(
    const int32_t* __restrict__ idx, int64_t n, int k, int E, int bm, int chunk,
    const float* __restrict__ gate_flat, int32_t* __restrict__ hist, int32_t* __restrict__ counts,
    int32_t* __restrict__ offsets, int4* __restrict__ tiles, int32_t* __restrict__ n_tiles,
    int32_t* __restrict__ perm, int32_t* __restrict__ inv, int32_t* __restrict__ row_tok,
    float* __restrict__ row_gate, DevStatus* st, int S, int64_t T, float lambda) {
    pdl_wait();
    extern __shared__ __align__(16) int32_t ps_smem[];
    __shared__ int s_off[1024], s_tot;
    const int nchunks = gridDim.x;
    const int lane = threadIdx.x & 31;
    perm_hist_body(idx, n, E, chunk, blockIdx.x, nchunks, hist, st, ps_smem);
    if (!grid_barrier(st, gridDim.x, PERM_BARRIER_LIMIT_NS, SITE_PERMUTE_BARRIER)) return;
    const int gw = (int)(((int64_t)blockIdx.x * PT + threadIdx.x) >> 5);
    for (int e = gw; e < E; e += nchunks * PW) perm_chunk_scan_warp(hist, nchunks, e, lane, counts);
    if (!grid_barrier(st, gridDim.x, PERM_BARRIER_LIMIT_NS, SITE_PERMUTE_BARRIER)) return;
    // exclusive offsets over the E <= 1024 experts, four per thread
    int loc[4], sum = 0;
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int e = 4 * threadIdx.x + q;
        loc[q] = e < E ? __ldcg(counts + e) : 0;
        sum += loc[q];
    }
    int ex = block_exclusive_scan_1024(sum, &s_tot);
#pragma unroll
    for (int q = 0; q < 4; ++q) {
        const int e = 4 * threadIdx.x + q;
        if (e < E) s_off[e] = ex;
        ex += loc[q];
    }
    __syncthreads();
    if (blockIdx.x == 0) {
        for (int e = threadIdx.x; e < E; e += PT) offsets[e] = s_off[e];
        if (threadIdx.x == 0) offsets[E] = s_tot;
        int tl[4], tsum = 0;
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            tl[q] = (loc[q] + bm - 1) / bm;
            tsum += tl[q];
        }
        __shared__ int s_ttot;
        int tex = block_exclusive_scan_1024(tsum, &s_ttot);
        // the always-on groups' m-tiles follow the routed ones
        const int64_t smt = S > 0 ? (T + bm - 1) / bm : 0;
        for (int64_t j = threadIdx.x; j < S * smt; j += PT) {
            const int c = (int)(j / smt);
            const int64_t r0 = (j - (int64_t)c * smt) * bm;
            tiles[s_ttot + j] = make_int4(E + c, (int)(n + (int64_t)c * T + r0),
                                          (int)(T - r0 < bm ? T - r0 : bm), 0);
        }
        if (threadIdx.x == 0) *n_tiles = s_ttot + (int)(S * smt);
#pragma unroll
        for (int q = 0; q < 4; ++q) {
            const int g = 4 * threadIdx.x + q;
            for (int m = 0; m < tl[q]; ++m)
                tiles[tex + m] = make_int4(g, s_off[g] + m * bm, min(bm, loc[q] - m * bm), 0);
            tex += tl[q];
        }
    }
    perm_scatter_body(idx, n, k, E, chunk, blockIdx.x, nchunks, hist, s_off, gate_flat, perm, inv,
                      row_tok, row_gate, ps_smem);
    for (int64_t i = (int64_t)blockIdx.x * PT + threadIdx.x; i < S * T; i += (int64_t)nchunks * PT) {
        row_tok[n + i] = (int32_t)(i % T);   // always-on group c = i / T, token t = i % T
        row_gate[n + i] = lambda;
    }
}

// m-tile table from given offsets (one thread per group, E <= 1024).
__global__ void __launch_bounds__(1024) tile_table_kernel(const int32_t* __restrict__ offsets,
                                                          int G, int bm, int4* __restrict__ tiles,
                                                          int32_t* __restrict__ n_tiles) {
    pdl_wait();
    __shared__ int s_total;
    const int g = threadIdx.x;
    const int cnt = (g < G) ? max(0, offsets[g + 1] - offsets[g]) : 0;
    const int nt = (cnt + bm - 1) / bm;
    const int toff = block_exclusive_scan_1024(nt, &s_total);
    if (g < G)
        for (int m = 0; m < nt; ++m)
            tiles[toff + m] = make_int4(g, offsets[g] + m * bm, min(bm, cnt - m * bm), 0);
    if (g == 0) *n_tiles = s_total;
}

// One CTA of 1024 threads.  Orders the (m-tile, n-tile) work items of a grouped GEMM
// in nb token bands x column groups of gsz n-tiles: band b holds the m-tiles whose
// middle row's token lies in [b T / nb, (b + 1) T / nb) (expert-major order kept
// inside a band).  Items run band-major, then column group, then m-tile, then n-tile,
// so the rows of y that the running items accumulate into stay within one band and
// one column group, a block small enough to stay in L2.
// items[i] = {expert, first row, rows, first column}; *n_items = m-tiles x n_ntiles.
__global__ void __launch_bounds__(1024) item_order_kernel(
    const int4* __restrict__ tiles, const int32_t* __restrict__ n_tiles_dev,
    const int32_t* __restrict__ row_tok, int64_t T, int nb, int n_ntiles, int gsz, int BN,
    int max_tiles, int4* __restrict__ items, int32_t* __restrict__ n_items) {
    pdl_wait();
    extern __shared__ int32_t io_smem[];
    int32_t* band = io_smem;                 // [max_tiles]
    int32_t* rank = io_smem + max_tiles;     // [max_tiles]
    __shared__ int s_cnt[ITEM_MAX_BANDS + 1];
    int nt = *n_tiles_dev;
    if (nt < 0 || nt > max_tiles) nt = 0;    // the GEMM reports an inconsistent table
    for (int i = threadIdx.x; i < nt; i += blockDim.x) {
        const int4 t = tiles[i];
        const int64_t tok = t.z > 0 ? row_tok[t.y + t.z / 2] : 0;
        const int64_t b = tok * nb / (T > 0 ? T : 1);
        band[i] = b < 0 ? 0 : (b >= nb ? nb - 1 : (int)b);
    }
    __syncthreads();
    // stable rank of each m-tile inside its band, 1024 tiles per pass: warp-level ranks
    // (match_any), then a running prefix over warps per band
    __shared__ int s_wcnt[32][ITEM_MAX_BANDS];
    __shared__ int s_carry[ITEM_MAX_BANDS];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    if (threadIdx.x < ITEM_MAX_BANDS) s_carry[threadIdx.x] = 0;
    for (int i0 = 0; i0 < nt; i0 += blockDim.x) {
        for (int q = threadIdx.x; q < 32 * ITEM_MAX_BANDS; q += blockDim.x) (&s_wcnt[0][0])[q] = 0;
        __syncthreads();
        const int i = i0 + threadIdx.x;
        const int b = i < nt ? band[i] : -1;
        const uint32_t m = __match_any_sync(0xffffffffu, b);
        const int lrank = __popc(m & ((1u << lane) - 1u));
        if (b >= 0 && lrank == 0) s_wcnt[warp][b] = __popc(m);
        __syncthreads();
        if (threadIdx.x < nb) {
            int run = s_carry[threadIdx.x];
            for (int w = 0; w < 32; ++w) {
                const int c = s_wcnt[w][threadIdx.x];
                s_wcnt[w][threadIdx.x] = run;
                run += c;
            }
            s_carry[threadIdx.x] = run;
        }
        __syncthreads();
        if (b >= 0) rank[i] = s_wcnt[warp][b] + lrank;
        __syncthreads();
    }
    if (threadIdx.x < nb) s_cnt[threadIdx.x] = s_carry[threadIdx.x];
    __syncthreads();
    if (threadIdx.x == 0) {   // exclusive prefix of the band sizes
        int run = 0;
        for (int b = 0; b < nb; ++b) {
            const int c = s_cnt[b];
            s_cnt[b] = run;
            run += c;
        }
        s_cnt[nb] = run;
        *n_items = run * n_ntiles;
    }
    __syncthreads();
    for (int i = threadIdx.x; i < nt; i += blockDim.x) {
        const int4 t = tiles[i];
        const int b = band[i];
        const int cnt_b = s_cnt[b + 1] - s_cnt[b];
        for (int j = 0; j < n_ntiles; ++j) {
            const int c = j / gsz, jl = j - c * gsz;
            const int in_group = min(gsz, n_ntiles - c * gsz);
            const int64_t pos = (int64_t)s_cnt[b] * n_ntiles + (int64_t)cnt_b * (c * gsz) +
                                (int64_t)rank[i] * in_group + jl;
            items[pos] = make_int4(t.x, t.y, t.z, j * BN);
        }
    }
}

}  // namespace

// Scratch of moevie_permute_static: fixed size, so that entry point needs neither a
// workspace from its caller nor an allocation of its own (layout in internal.h).
static __device__ __align__(256) unsigned char g_perm_static_scratch[PERM_STATIC_SCRATCH_BYTES];

// The current context (driver cuCtxGetCurrent, reached through the runtime's entry-point
// query so that the library links only the runtime); nullptr when it cannot be read.
void* current_context() {
    using GetCtx = CUresult (*)(CUcontext*);
    static std::atomic<GetCtx> fn{nullptr};
    GetCtx f = fn.load(std::memory_order_acquire);
    if (!f) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &ptr, 12000, cudaEnableDefault, &q) !=
                cudaSuccess ||
            q != cudaDriverEntryPointSuccess || !ptr)
            return nullptr;
        f = reinterpret_cast<GetCtx>(ptr);
        fn.store(f, std::memory_order_release);
    }
    CUcontext c = nullptr;
    return f(&c) == CUDA_SUCCESS ? static_cast<void*>(c) : nullptr;
}

cudaError_t perm_static_scratch(unsigned char** out) {
    constexpr int kMaxDevices = 64;
    static std::mutex mu;
    static unsigned char* addr[kMaxDevices] = {};
    static void* ctx[kMaxDevices] = {};
    int dev = -1;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev < 0 || dev >= kMaxDevices) return cudaErrorInvalidDevice;
    // The address belongs to the context it was looked up in: after a device reset
    // the runtime makes a new primary context, and the address is looked up again.
    void* cur = current_context();
    std::lock_guard<std::mutex> lock(mu);
    if (!addr[dev] || cur == nullptr || cur != ctx[dev]) {   // with that device current
        void* p = nullptr;
        err = cudaGetSymbolAddress(&p, g_perm_static_scratch);
        if (err != cudaSuccess) return err;
        addr[dev] = static_cast<unsigned char*>(p);
        ctx[dev] = current_context();   // the context the runtime has now made current
    }
    *out = addr[dev];
    return cudaSuccess;
}

int perm_chunk(int64_t n, int num_sms) {
    int64_t c = (n + 2 * num_sms - 1) / (2 * num_sms);
    c = (c + 255) / 256 * 256;
    if (c < 256) c = 256;
    if (c > PERM_CHUNK_MAX) c = PERM_CHUNK_MAX;
    return (int)c;
}

cudaError_t launch_permute(const int32_t* idx, int64_t n_slots, int k, int E, int bm, int chunk,
                           const float* gate_flat, int32_t* hist, int32_t* counts,
                           int32_t* offsets, int4* tiles, int32_t* n_tiles, int32_t* perm,
                           int32_t* inv, int32_t* row_tok, float* row_gate, DevStatus* st,
                           cudaStream_t s, const SharedRows* sh) {
    const int nchunks = (int)((n_slots + chunk - 1) / chunk);
    int S = sh ? sh->S : 0;
    int64_t T = sh ? sh->T : 0;
    float lambda = sh ? sh->lambda : 0.f;
    const size_t smem = (size_t)(chunk + PW * E) * 4;
    // per-device set-up on the first call (kernel attributes, co-resident CTAs of
    // perm_fused_kernel; 0: no cooperative launch), safe for concurrent first calls
    static std::mutex setup_mu;
    static std::atomic<bool> attr_set[64];
    static std::atomic<int> coop_ctas[64];
    int dev = 0;
    cudaError_t err = cudaGetDevice(&dev);
    if (err != cudaSuccess) return err;
    if (dev >= 0 && dev < 64 && !attr_set[dev].load(std::memory_order_acquire)) {
        std::lock_guard<std::mutex> lock(setup_mu);
        if (!attr_set[dev].load(std::memory_order_relaxed)) {
            const int max_smem = (int)((PERM_CHUNK_MAX + PW * 1024) * 4);
            if ((err = cudaFuncSetAttribute(perm_scatter_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                            max_smem)) != cudaSuccess)
                return err;
            if ((err = cudaFuncSetAttribute(perm_fused_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                            max_smem)) != cudaSuccess)
                return err;
            int coop = 0, sms = 0, per_sm = 0;
            cudaDeviceGetAttribute(&coop, cudaDevAttrCooperativeLaunch, dev);
            cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
            if (coop && cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, perm_fused_kernel, PT,
                                                                      (size_t)max_smem) == cudaSuccess)
                coop_ctas[dev].store(per_sm * sms, std::memory_order_relaxed);
            attr_set[dev].store(true, std::memory_order_release);
        }
    }
    if (dev >= 0 && dev < 64 && nchunks <= coop_ctas[dev].load(std::memory_order_relaxed)) {
        err = launch_pdl_coop(perm_fused_kernel, dim3(nchunks), dim3(PT), smem, s, idx, n_slots, k, E,
                              bm, chunk, gate_flat, hist, counts, offsets, tiles, n_tiles, perm, inv,
                              row_tok, row_gate, st, S, T, lambda);
        count_launches(1);
        return err;
    }
    if ((err = launch_pdl(perm_hist_kernel, dim3(nchunks), dim3(PT), (size_t)E * 4, s, idx, n_slots, E,
                          chunk, hist, st)) != cudaSuccess)
        return err;
    if ((err = launch_pdl(perm_chunk_scan_kernel, dim3((E + 7) / 8), dim3(256), 0, s, hist, nchunks, E,
                          counts)) != cudaSuccess)
        return err;
    if ((err = launch_pdl(perm_offsets_kernel, dim3(1), dim3(1024), 0, s, (const int32_t*)counts, E, bm,
                          offsets, tiles, n_tiles)) != cudaSuccess)
        return err;
    err = launch_pdl(perm_scatter_kernel, dim3(nchunks), dim3(PT), smem, s, idx, n_slots, k, E, chunk,
                     (const int32_t*)hist, (const int32_t*)offsets, gate_flat, perm, inv, row_tok,
                     row_gate);
    count_launches(4);
    if (err == cudaSuccess && S > 0)
        err = launch_shared_rows(T, n_slots, S, E, lambda, row_tok, row_gate, tiles, n_tiles,
                                 max_mtiles(n_slots, E), st, s);
    return err;
}

cudaError_t launch_item_order(const int4* tiles, const int32_t* n_tiles, const int32_t* row_tok,
                              int64_t T, int nb, int n_ntiles, int gsz, int BN, int max_tiles,
                              int4* items, int32_t* n_items, cudaStream_t s) {
    if (nb < 1 || nb > ITEM_MAX_BANDS || max_tiles > ITEM_MAX_TILES || gsz < 1)
        return cudaErrorInvalidValue;
    const size_t smem = (size_t)2 * max_tiles * sizeof(int32_t);
    static std::atomic<bool> attr_set[64];
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev].load(std::memory_order_acquire)) {
        cudaError_t err = cudaFuncSetAttribute(item_order_kernel,   // idempotent: no lock needed
                                               cudaFuncAttributeMaxDynamicSharedMemorySize,
                                               2 * ITEM_MAX_TILES * (int)sizeof(int32_t));
        if (err != cudaSuccess) return err;
        attr_set[dev].store(true, std::memory_order_release);
    }
    const cudaError_t err = launch_pdl(item_order_kernel, dim3(1), dim3(1024), smem, s, tiles, n_tiles,
                                       row_tok, T, nb, n_ntiles, gsz, BN, max_tiles, items, n_items);
    count_launches(1);
    return err;
}

cudaError_t launch_tile_table(const int32_t* offsets, int G, int bm, int4* tiles,
                              int32_t* n_tiles, cudaStream_t s) {
    const cudaError_t err = launch_pdl(tile_table_kernel, dim3(1), dim3(1024), 0, s, offsets, G, bm, tiles,
                                       n_tiles);
    count_launches(1);
    return err;
}

}  // namespace mv
