// misc.cu -- memory-bound helper kernels of the MoE-ViE layer, sm_103a.
//   zero_f32_kernel      y accumulator := 0 (float4 stores)
//   f32_to_bf16_kernel   y := bf16(y accumulator)  (32-byte loads, 16-byte stores)
//   combine_kernel       Eq. (6) as a stand-alone gather-reduce over expert-major
//                        rows: y[t] = sum_j gate[t, j] rows[inv[t*k + j]] + lambda * shared[t]
//   wait_probe_kernel    bounded wait on a barrier nobody arrives at (error-path test)
#include "internal.h"

namespace mv {

namespace {

__global__ void zero_f32_kernel(float4* __restrict__ p, int64_t n4) {
    pdl_wait();
    const float4 z = make_float4(0.f, 0.f, 0.f, 0.f);
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n4;
         i += (int64_t)gridDim.x * blockDim.x)
        p[i] = z;
}

// n8 groups of 8 values.
__global__ void f32_to_bf16_kernel(const float4* __restrict__ src, uint4* __restrict__ dst,
                                   int64_t n8) {
    pdl_wait();
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < n8;
         i += (int64_t)gridDim.x * blockDim.x) {
        const float4 a = src[2 * i], b = src[2 * i + 1];
        uint4 u;
        u.x = pack_bf16x2(a.x, a.y);
        u.y = pack_bf16x2(a.z, a.w);
        u.z = pack_bf16x2(b.x, b.y);
        u.w = pack_bf16x2(b.z, b.w);
        dst[i] = u;
    }
}

// One thread per (token, 8 columns).
__global__ void combine_kernel(const __nv_bfloat16* __restrict__ rows,
                               const int32_t* __restrict__ inv, const float* __restrict__ gate,
                               const __nv_bfloat16* __restrict__ shared, float lambda, int64_t T,
                               int k, int d, __nv_bfloat16* __restrict__ y) {
    pdl_wait();
    const int cpr = d >> 3;   // 8-column groups per row
    for (int64_t i = blockIdx.x * (int64_t)blockDim.x + threadIdx.x; i < T * cpr;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t t = i / cpr;
        const int c = (int)(i - t * cpr) * 8;
        float acc[8];
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] = 0.f;
        for (int j = 0; j < k; ++j) {
            const int r = inv[t * k + j];
            if (r < 0 || r >= T * k) continue;   // a dropped slot contributes nothing
            const float g = gate[t * k + j];
            float v[8];
            unpack_bf16x8(*reinterpret_cast<const uint4*>(rows + (int64_t)r * d + c), v);
#pragma unroll
            for (int q = 0; q < 8; ++q) acc[q] = fmaf(g, v[q], acc[q]);
        }
        if (shared) {
            float v[8];
            unpack_bf16x8(*reinterpret_cast<const uint4*>(shared + t * d + c), v);
#pragma unroll
            for (int q = 0; q < 8; ++q) acc[q] = fmaf(lambda, v[q], acc[q]);
        }
        uint4 u;
        u.x = pack_bf16x2(acc[0], acc[1]);
        u.y = pack_bf16x2(acc[2], acc[3]);
        u.z = pack_bf16x2(acc[4], acc[5]);
        u.w = pack_bf16x2(acc[6], acc[7]);
        *reinterpret_cast<uint4*>(y + t * d + c) = u;
    }
}

__global__ void wait_probe_kernel(DevStatus* st, uint64_t limit_ns) {
    __shared__ __align__(8) uint64_t bar;
    const uint32_t b = smem_u32(&bar);
    if (threadIdx.x == 0) {
        mbar_init(b, 1);
        mbar_fence_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        // Nothing ever arrives: the wait must give up after limit_ns.
        if (!mbar_wait(b, 0, limit_ns, nullptr))
            report(st, MOEVIE_ERR_TIMEOUT, SITE_TIMEOUT_PROBE, 0, 0);
    }
}

// Rows of the shared expert's S always-on groups (E .. E + S - 1): row base + c T + t
// is token t with gate lambda.  Block 0 also appends the groups' m-tiles after the
// routed ones that the permute step counted in *n_tiles.
__global__ void shared_rows_kernel(int64_t T, int64_t base, int S, int E, float lambda,
                                   int32_t* __restrict__ row_tok, float* __restrict__ row_gate,
                                   int4* __restrict__ tiles, int32_t* __restrict__ n_tiles,
                                   int64_t max_routed, DevStatus* st) {
    pdl_wait();   // the permute step's tile count
    const int64_t n = T * S;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        row_tok[base + i] = (int32_t)(i % T);
        row_gate[base + i] = lambda;
    }
    if (blockIdx.x == 0) {
        const int n0 = *n_tiles;
        if (n0 < 0 || n0 > max_routed) {   // inconsistent count: leave the table alone
            if (threadIdx.x == 0) report(st, MOEVIE_ERR_DEVICE, SITE_GEMM_TILES, n0, -2);
            return;
        }
        const int64_t mt = (T + GM_BM - 1) / GM_BM;
        for (int64_t j = threadIdx.x; j < S * mt; j += blockDim.x) {
            const int c = (int)(j / mt);
            const int64_t r0 = (j - (int64_t)c * mt) * GM_BM;
            const int64_t nr = T - r0 < GM_BM ? T - r0 : GM_BM;
            tiles[n0 + j] = make_int4(E + c, (int)(base + (int64_t)c * T + r0), (int)nr, 0);
        }
        __syncthreads();   // every thread of the block has read *n_tiles
        if (threadIdx.x == 0) *n_tiles = n0 + (int)(S * mt);
    }
}

// Loss-free balancing bias update from one step's expert loads t_e = counts[e]
// (Sec. 2.2.2), one CTA with one thread per expert (E <= 1024):
//   rule 0, z-score (Eq. 9): b_e -= alpha (t_e - mu) / sigma  (sigma = 0: no update)
//   rule 1, sign (Eq. 8):    b_e -= alpha sign(t_e - mu)
// mu = (exact integer sum) / E and sigma = sqrt(sum (t_e - mu)^2 / E) (population) in
// fp64; the sign is taken exactly as sign(E t_e - sum) in integers.  Each new b_e is
// computed in fp64 with separately rounded operations and rounded to fp32.  A negative
// load is a device error and leaves b unchanged.
__global__ void __launch_bounds__(1024) update_bias_kernel(const int32_t* __restrict__ counts, int E,
                                                           float alpha, int rule, float* __restrict__ b,
                                                           DevStatus* st) {
    pdl_wait();
    __shared__ long long s_isum[32];
    __shared__ double s_dsum[32];
    __shared__ long long s_S;
    __shared__ double s_sigma;
    __shared__ int s_bad;
    const int e = threadIdx.x, lane = e & 31, warp = e >> 5, nwarps = blockDim.x >> 5;
    const int t = e < E ? counts[e] : 0;
    if (e == 0) s_bad = 0;
    __syncthreads();
    if (t < 0) atomicOr(&s_bad, 1);
    long long is = t;
#pragma unroll
    for (int o = 16; o; o >>= 1) is += __shfl_xor_sync(0xffffffffu, is, o);
    if (lane == 0) s_isum[warp] = is;
    __syncthreads();
    if (warp == 0) {   // the exact integer total
        long long v = lane < nwarps ? s_isum[lane] : 0;
#pragma unroll
        for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
        if (lane == 0) s_S = v;
    }
    __syncthreads();
    if (s_bad) {
        if (e == 0) report(st, MOEVIE_ERR_DEVICE, SITE_BIAS_COUNTS, 0, 0);
        return;
    }
    const long long S = s_S;
    const double mu = __ddiv_rn((double)S, (double)E);
    const double dev = __dsub_rn((double)t, mu);
    double sq = e < E ? __dmul_rn(dev, dev) : 0.0;
#pragma unroll
    for (int o = 16; o; o >>= 1) sq = __dadd_rn(sq, __shfl_xor_sync(0xffffffffu, sq, o));
    if (lane == 0) s_dsum[warp] = sq;
    __syncthreads();
    if (warp == 0) {   // population standard deviation
        double v = lane < nwarps ? s_dsum[lane] : 0.0;
#pragma unroll
        for (int o = 16; o; o >>= 1) v = __dadd_rn(v, __shfl_xor_sync(0xffffffffu, v, o));
        if (lane == 0) s_sigma = __dsqrt_rn(__ddiv_rn(v, (double)E));
    }
    __syncthreads();
    const double sigma = s_sigma;
    if (e >= E) return;
    double step;
    if (rule == 0) {
        if (sigma == 0.0) return;
        step = __ddiv_rn(dev, sigma);
    } else {
        const long long c = (long long)E * t - S;
        step = (double)((c > 0) - (c < 0));
    }
    b[e] = __double2float_rn(__dsub_rn((double)b[e], __dmul_rn((double)alpha, step)));
}

int grid_for(int64_t n, int threads) {
    int64_t g = (n + threads - 1) / threads;
    if (g > 152 * 16) g = 152 * 16;
    return (int)(g < 1 ? 1 : g);
}

}  // namespace

cudaError_t launch_zero_f32(float* p, int64_t n, cudaStream_t s) {
    const int64_t n4 = n / 4;   // callers pass multiples of 4
    cudaError_t e = launch_pdl(zero_f32_kernel, dim3(grid_for(n4, 256)), dim3(256), 0, s,
                               reinterpret_cast<float4*>(p), n4);
    if (e != cudaSuccess) return e;
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_f32_to_bf16(const float* src, __nv_bfloat16* dst, int64_t n, cudaStream_t s) {
    const int64_t n8 = n / 8;   // callers pass multiples of 8
    const cudaError_t e = launch_pdl(f32_to_bf16_kernel, dim3(grid_for(n8, 256)), dim3(256), 0, s,
                                     reinterpret_cast<const float4*>(src), reinterpret_cast<uint4*>(dst),
                                     n8);
    count_launches(1);
    return e;
}

cudaError_t launch_shared_rows(int64_t T, int64_t base, int S, int E, float lambda,
                               int32_t* row_tok, float* row_gate, int4* tiles, int32_t* n_tiles,
                               int64_t max_routed, DevStatus* st, cudaStream_t s) {
    const cudaError_t e = launch_pdl(shared_rows_kernel, dim3(grid_for(T * S, 256)), dim3(256), 0, s, T,
                                     base, S, E, lambda, row_tok, row_gate, tiles, n_tiles,
                                     max_routed, st);
    count_launches(1);
    return e;
}

cudaError_t launch_update_bias(const int32_t* counts, int E, float alpha, int rule, float* b,
                               DevStatus* st, cudaStream_t s) {
    const cudaError_t e = launch_pdl(update_bias_kernel, dim3(1), dim3((E + 31) / 32 * 32), 0, s, counts,
                                     E, alpha, rule, b, st);
    count_launches(1);
    return e;
}

cudaError_t launch_combine(const __nv_bfloat16* rows, const int32_t* inv, const float* gate,
                           const __nv_bfloat16* shared, float lambda, int64_t T, int k, int d,
                           __nv_bfloat16* y, cudaStream_t s) {
    const int64_t n = T * (d / 8);
    cudaError_t e = launch_pdl(combine_kernel, dim3(grid_for(n, 256)), dim3(256), 0, s, rows, inv, gate,
                               shared, lambda, T, k, d, y);
    if (e != cudaSuccess) return e;
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_wait_probe(DevStatus* st, uint64_t limit_ns, cudaStream_t s) {
    wait_probe_kernel<<<1, 32, 0, s>>>(st, limit_ns);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace mv
