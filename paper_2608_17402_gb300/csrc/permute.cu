// permute.cu -- expert-major order of the flat routing slots (App. B, Algorithm 1,
// phase 1: Sort by expert id, index = pos // K, BinCount, CumSum), sm_103a.
//
// A stable counting sort over chunks of PERM_CHUNK flat slots:
//   perm_hist_kernel    per-chunk histograms (16-byte vector loads of idx)
//   perm_scan_kernel    counts, exclusive offsets, each chunk's first row per
//                       expert, and the m-tile prefix used by the grouped GEMMs
//   perm_scatter_kernel stages its chunk in shared memory (16-byte loads), ranks
//                       every slot among the earlier slots of the same expert
//                       (warp match + per-warp running counts), and writes perm,
//                       inv and the per-row token (pos // K) and gate.
// Inside one expert's segment, rows keep ascending slot order t*k + j.
#include "internal.h"

namespace mv {

namespace {

constexpr int PT = 256;                      // threads per CTA
constexpr int PW = PT / 32;                  // warps per CTA
constexpr int PER_WARP = PERM_CHUNK / PW;    // slots per warp in the scatter

__device__ __forceinline__ bool valid_id(int e, int E) { return e >= 0 && e < E; }

__global__ void __launch_bounds__(PT) perm_hist_kernel(const int32_t* __restrict__ idx,
                                                       int64_t n, int E,
                                                       int32_t* __restrict__ hist,
                                                       DevStatus* st) {
    extern __shared__ int32_t cnt[];
    for (int e = threadIdx.x; e < E; e += PT) cnt[e] = 0;
    __syncthreads();
    const int64_t c0 = (int64_t)blockIdx.x * PERM_CHUNK;
    const int64_t c1 = c0 + PERM_CHUNK < n ? c0 + PERM_CHUNK : n;
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
    for (int e = threadIdx.x; e < E; e += PT) hist[(int64_t)blockIdx.x * E + e] = cnt[e];
}

// Exclusive scan of one int per thread over a 1024-thread block.
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
        const int w = wsum[lane];
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

// One thread per expert (E <= 1024).  Rewrites hist[c][e] in place with the
// first row of expert e inside chunk c.
__global__ void __launch_bounds__(1024) perm_scan_kernel(int32_t* __restrict__ hist, int nchunks,
                                                         int E, int bm,
                                                         int32_t* __restrict__ counts,
                                                         int32_t* __restrict__ offsets,
                                                         int32_t* __restrict__ tile_off) {
    __shared__ int s_total, s_tiles;
    const int e = threadIdx.x;
    int cnt = 0;
    if (e < E)
        for (int c = 0; c < nchunks; ++c) cnt += hist[(int64_t)c * E + e];
    const int off = block_exclusive_scan_1024(e < E ? cnt : 0, &s_total);
    const int nt = (cnt + bm - 1) / bm;
    const int toff = block_exclusive_scan_1024(e < E ? nt : 0, &s_tiles);
    if (e < E) {
        if (counts) counts[e] = cnt;
        offsets[e] = off;
        tile_off[e] = toff;
        int run = off;
        for (int c = 0; c < nchunks; ++c) {
            const int h = hist[(int64_t)c * E + e];
            hist[(int64_t)c * E + e] = run;
            run += h;
        }
    }
    if (e == 0) {
        offsets[E] = s_total;
        tile_off[E] = s_tiles;
    }
}

// Dynamic smem: PERM_CHUNK ints (the chunk's ids) + PW * E ints (per-warp counts).
__global__ void __launch_bounds__(PT) perm_scatter_kernel(
    const int32_t* __restrict__ idx, int64_t n, int k, int E, const int32_t* __restrict__ base,
    const float* __restrict__ gate_flat, int32_t* __restrict__ perm, int32_t* __restrict__ inv,
    int32_t* __restrict__ row_tok, float* __restrict__ row_gate) {
    extern __shared__ __align__(16) int32_t ps_smem[];
    int32_t* sidx = ps_smem;
    int32_t* wc = ps_smem + PERM_CHUNK;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t c0 = (int64_t)blockIdx.x * PERM_CHUNK;
    const int len = (int)(c0 + PERM_CHUNK < n ? PERM_CHUNK : n - c0);
    {
        const int nvec = len >> 2;
        const int4* v = reinterpret_cast<const int4*>(idx + c0);
        int4* sv = reinterpret_cast<int4*>(sidx);
        for (int i = tid; i < nvec; i += PT) sv[i] = v[i];
        for (int i = 4 * nvec + tid; i < len; i += PT) sidx[i] = idx[c0 + i];
    }
    for (int i = tid; i < PW * E; i += PT) wc[i] = 0;
    __syncthreads();
    const int wbeg = warp * PER_WARP;
    const int wend = wbeg + PER_WARP < len ? wbeg + PER_WARP : len;
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
        int run = base[(int64_t)blockIdx.x * E + e];
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

__global__ void tile_prefix_kernel(const int32_t* __restrict__ offsets, int G, int bm,
                                   int32_t* __restrict__ tile_off) {
    __shared__ int s_total;
    int acc_base = 0;
    for (int g0 = 0; g0 < G; g0 += 1024) {
        const int g = g0 + threadIdx.x;
        const int cnt = (g < G) ? offsets[g + 1] - offsets[g] : 0;
        const int nt = cnt > 0 ? (cnt + bm - 1) / bm : 0;
        const int ex = block_exclusive_scan_1024(nt, &s_total);
        if (g < G) tile_off[g] = acc_base + ex;
        acc_base += s_total;
        __syncthreads();
    }
    if (threadIdx.x == 0) tile_off[G] = acc_base;
}

__global__ void single_group_kernel(int32_t* offsets, int32_t* tile_off, int T, int bm) {
    offsets[0] = 0;
    offsets[1] = T;
    tile_off[0] = 0;
    tile_off[1] = (T + bm - 1) / bm;
}

}  // namespace

cudaError_t launch_single_group(int32_t* offsets, int32_t* tile_off, int T, int bm, cudaStream_t s) {
    single_group_kernel<<<1, 1, 0, s>>>(offsets, tile_off, T, bm);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_permute(const int32_t* idx, int64_t n_slots, int k, int E, int bm,
                           const float* gate_flat, int32_t* hist, int32_t* counts,
                           int32_t* offsets, int32_t* tile_off, int32_t* perm, int32_t* inv,
                           int32_t* row_tok, float* row_gate, DevStatus* st, cudaStream_t s) {
    const int nchunks = (int)((n_slots + PERM_CHUNK - 1) / PERM_CHUNK);
    perm_hist_kernel<<<nchunks, PT, (size_t)E * 4, s>>>(idx, n_slots, E, hist, st);
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    perm_scan_kernel<<<1, 1024, 0, s>>>(hist, nchunks, E, bm, counts, offsets, tile_off);
    if ((err = cudaGetLastError()) != cudaSuccess) return err;
    const size_t smem = (size_t)(PERM_CHUNK + PW * E) * 4;
    static bool attr_set[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        err = cudaFuncSetAttribute(perm_scatter_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                   (int)((PERM_CHUNK + PW * 1024) * 4));
        if (err != cudaSuccess) return err;
        attr_set[dev] = true;
    }
    perm_scatter_kernel<<<nchunks, PT, smem, s>>>(idx, n_slots, k, E, hist, gate_flat, perm, inv,
                                                  row_tok, row_gate);
    count_launches(3);
    return cudaGetLastError();
}

cudaError_t launch_tile_prefix(const int32_t* offsets, int G, int bm, int32_t* tile_off,
                               cudaStream_t s) {
    tile_prefix_kernel<<<1, 1024, 0, s>>>(offsets, G, bm, tile_off);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace mv
