// route.cu -- router of the MoE-ViE layer (Eqs. 1, 7, 4-5), sm_103a.
//
//  1. route_logits_kernel: s = x . W_r in fp32 on CUDA cores (64 tokens x 64
//     experts per CTA), plus |x_t|^2 and |W_r[:, e]|^2 for the error bound.
//  2. route_topk_kernel: one warp per token; keys sigmoid(s) + b, k rounds of warp
//     arg-max (ties to the lower id), and a certificate: the gap between the k-th
//     and (k+1)-th key must exceed twice the key error bound.  Certified tokens
//     write ascending ids and gates sigmoid(s)/sum (the bias only selects).
//  3. route_fallback_kernel: for every token without a certificate, experts whose
//     key interval overlaps the boundary get exact logits (fp64: each product
//     x_i * w_i of a bf16 and an fp32 value is exact in double) and the remaining
//     places are filled from them, ties to the lower id.
#include <math.h>

#include "internal.h"

namespace mv {

namespace {

constexpr int LG_TT = 64;   // tokens per CTA
constexpr int LG_TE = 64;   // experts per CTA
constexpr int LG_TK = 32;   // K per smem stage

__global__ void __launch_bounds__(256) route_logits_kernel(const __nv_bfloat16* __restrict__ x,
                                                           const float* __restrict__ Wr, int T,
                                                           int d, int E, float* __restrict__ s,
                                                           float* __restrict__ xnorm2,
                                                           float* __restrict__ wnorm2,
                                                           DevStatus* st) {
    __shared__ float xs[LG_TK][LG_TT + 4];
    __shared__ float wsm[LG_TK][LG_TE + 4];
    __shared__ float wred[8][LG_TE];
    const int t0 = blockIdx.x * LG_TT, e0 = blockIdx.y * LG_TE;
    const int tid = threadIdx.x;
    const int ty = tid >> 4, tx = tid & 15;
    const int xl_t = tid >> 2, xl_k = (tid & 3) * 8;      // x loader: token, first k
    const int wl_k = tid >> 3, wl_e = (tid & 7) * 8;      // W loader: k row, first expert
    float acc[4][4];
#pragma unroll
    for (int i = 0; i < 4; ++i)
#pragma unroll
        for (int j = 0; j < 4; ++j) acc[i][j] = 0.f;
    float xsq = 0.f;
    float wsq[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) wsq[i] = 0.f;

    for (int k0 = 0; k0 < d; k0 += LG_TK) {
        {
            const int t = t0 + xl_t, kk = k0 + xl_k;
            float v[8];
            if (t < T && kk < d) {   // d % 8 == 0: the 8 values are all inside the row
                const uint4 u = *reinterpret_cast<const uint4*>(x + (int64_t)t * d + kk);
                unpack_bf16x8(u, v);
            } else {
#pragma unroll
                for (int i = 0; i < 8; ++i) v[i] = 0.f;
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                xs[xl_k + i][xl_t] = v[i];
                xsq = fmaf(v[i], v[i], xsq);
            }
        }
        {
            const int kk = k0 + wl_k;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const int e = e0 + wl_e + i;
                const float v = (kk < d && e < E) ? __ldg(Wr + (int64_t)kk * E + e) : 0.f;
                wsm[wl_k][wl_e + i] = v;
                wsq[i] = fmaf(v, v, wsq[i]);
            }
        }
        __syncthreads();
#pragma unroll
        for (int kk = 0; kk < LG_TK; ++kk) {
            float a[4], b[4];
#pragma unroll
            for (int i = 0; i < 4; ++i) a[i] = xs[kk][ty * 4 + i];
#pragma unroll
            for (int j = 0; j < 4; ++j) b[j] = wsm[kk][tx * 4 + j];
#pragma unroll
            for (int i = 0; i < 4; ++i)
#pragma unroll
                for (int j = 0; j < 4; ++j) acc[i][j] = fmaf(a[i], b[j], acc[i][j]);
        }
        __syncthreads();
    }
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const int t = t0 + ty * 4 + i;
        if (t >= T) continue;
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const int e = e0 + tx * 4 + j;
            if (e < E) s[(int64_t)t * E + e] = acc[i][j];
        }
    }
    if (blockIdx.y == 0) {   // |x_t|^2: 4 consecutive lanes hold one token
        xsq += __shfl_xor_sync(0xffffffffu, xsq, 1);
        xsq += __shfl_xor_sync(0xffffffffu, xsq, 2);
        if ((tid & 3) == 0 && t0 + xl_t < T) xnorm2[t0 + xl_t] = xsq;
    }
    if (blockIdx.x == 0) {   // |W_r[:, e]|^2: lanes l, l+8, l+16, l+24 share experts
#pragma unroll
        for (int i = 0; i < 8; ++i) {
            float v = wsq[i];
            v += __shfl_xor_sync(0xffffffffu, v, 8);
            v += __shfl_xor_sync(0xffffffffu, v, 16);
            if ((tid & 31) < 8) wred[tid >> 5][wl_e + i] = v;
        }
        __syncthreads();
        if (tid < LG_TE && e0 + tid < E) {
            float v = 0.f;
            for (int w = 0; w < 8; ++w) v += wred[w][tid];
            wnorm2[e0 + tid] = v;
        }
    }
    if (blockIdx.x == 0 && blockIdx.y == 0 && tid == 0) st->fb_count = 0;
}

__device__ __forceinline__ float sigmoid_f32(float v) { return 1.0f / (1.0f + expf(-v)); }

// Half-width of the key interval of token t: key error <= 0.25 * logit error +
// fp32 evaluation slack (the slope of the sigmoid is at most 1/4).
__device__ __forceinline__ float key_tau(float xn2, float wmax2) {
    const float tau_s = ROUTE_TAU_C * 5.9604645e-8f * sqrtf(xn2 * wmax2);
    return 0.25f * tau_s + ROUTE_KEY_SLACK;
}

__device__ __forceinline__ float warp_max_wnorm(const float* wnorm2, int E, int lane) {
    float wm = 0.f;
    for (int e = lane; e < E; e += 32) wm = fmaxf(wm, wnorm2[e]);
#pragma unroll
    for (int o = 16; o; o >>= 1) wm = fmaxf(wm, __shfl_xor_sync(0xffffffffu, wm, o));
    return wm;
}

// One warp per token.  NPL = experts per lane (expert e sits in lane e % 32, slot e / 32).
template <int NPL>
__global__ void __launch_bounds__(256) route_topk_kernel(
    const float* __restrict__ s, const float* __restrict__ b, const float* __restrict__ xnorm2,
    const float* __restrict__ wnorm2, int T, int E, int k, int32_t* __restrict__ idx,
    float* __restrict__ gate, int32_t* __restrict__ fb_tokens, DevStatus* st) {
    const int lane = threadIdx.x & 31;
    const int t = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (t >= T) return;
    const float wmax2 = warp_max_wnorm(wnorm2, E, lane);
    const float tau = key_tau(xnorm2[t], wmax2);
    float key[NPL], sg[NPL];
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
        const int e = lane + 32 * i;
        if (e < E) {
            sg[i] = sigmoid_f32(s[(int64_t)t * E + e]);
            key[i] = sg[i] + b[e];
        } else {
            sg[i] = 0.f;
            key[i] = -INFINITY;
        }
    }
    uint32_t taken = 0;
    float kth = 0.f, next = -INFINITY;
    const int rounds = (k < E) ? k + 1 : k;
    for (int j = 0; j < rounds; ++j) {
        float bv = -INFINITY;
        int bi = 0x7fffffff;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const int e = lane + 32 * i;
            if (e < E && !((taken >> i) & 1u) && (key[i] > bv || bi == 0x7fffffff)) {
                bv = key[i];
                bi = e;
            }
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            const float ov = __shfl_xor_sync(0xffffffffu, bv, o);
            const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
            if (ov > bv || (ov == bv && oi < bi)) {
                bv = ov;
                bi = oi;
            }
        }
        if (j < k) {
            if ((bi & 31) == lane) taken |= 1u << (bi >> 5);
            kth = bv;
        } else {
            next = bv;
        }
    }
    const bool certain = (k >= E) || (kth - next > 2.0f * tau);
    if (!certain) {
        if (lane == 0) {
            const int p = atomicAdd(&st->fb_count, 1);
            fb_tokens[p] = t;
        }
        return;
    }
    float ssum = 0.f;
#pragma unroll
    for (int i = 0; i < NPL; ++i)
        if ((taken >> i) & 1u) ssum += sg[i];
#pragma unroll
    for (int o = 16; o; o >>= 1) ssum += __shfl_xor_sync(0xffffffffu, ssum, o);
    const uint32_t lt = (1u << lane) - 1u;
    int base = 0;
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
        const uint32_t m = __ballot_sync(0xffffffffu, (taken >> i) & 1u);
        if ((taken >> i) & 1u) {
            const int pos = base + __popc(m & lt);
            idx[(int64_t)t * k + pos] = lane + 32 * i;
            gate[(int64_t)t * k + pos] = sg[i] / ssum;
        }
        base += __popc(m);
    }
}

constexpr int FB_THREADS = 256;

// Exact re-decision of uncertified tokens.  Dynamic smem: E floats (fast keys),
// E floats (fast sigmoid), E bytes (class), E doubles (exact keys).
__global__ void __launch_bounds__(FB_THREADS) route_fallback_kernel(
    const __nv_bfloat16* __restrict__ x, const float* __restrict__ Wr,
    const float* __restrict__ b, const float* __restrict__ s, const float* __restrict__ xnorm2,
    const float* __restrict__ wnorm2, int d, int E, int k, int32_t* __restrict__ idx,
    float* __restrict__ gate, const int32_t* __restrict__ fb_tokens, DevStatus* st) {
    extern __shared__ __align__(16) uint8_t fb_smem[];
    double* exk = reinterpret_cast<double*>(fb_smem);
    float* key = reinterpret_cast<float*>(exk + E);
    float* sg = key + E;
    uint8_t* cls = reinterpret_cast<uint8_t*>(sg + E);   // 1 sure in, 2 sure out, 3 candidate, 4 chosen
    __shared__ int s_in, s_cand;
    __shared__ float s_wmax2;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    if (warp == 0) {
        const float wm = warp_max_wnorm(wnorm2, E, lane);
        if (lane == 0) s_wmax2 = wm;
    }
    __syncthreads();
    const int nfb = st->fb_count;
    for (int i = blockIdx.x; i < nfb; i += gridDim.x) {
        const int t = fb_tokens[i];
        const float tau = key_tau(xnorm2[t], s_wmax2);
        for (int e = tid; e < E; e += FB_THREADS) {
            sg[e] = sigmoid_f32(s[(int64_t)t * E + e]);
            key[e] = sg[e] + b[e];
        }
        if (tid == 0) {
            s_in = 0;
            s_cand = 0;
        }
        __syncthreads();
        // classify against the fast-key intervals [key - tau, key + tau]
        for (int e = tid; e < E; e += FB_THREADS) {
            int maybe_above = 0, surely_above = 0;
            for (int f = 0; f < E; ++f) {
                if (f == e) continue;
                if (key[f] + tau >= key[e] - tau) ++maybe_above;
                if (key[f] - tau > key[e] + tau) ++surely_above;
            }
            uint8_t c = 3;
            if (maybe_above < k) c = 1;
            else if (surely_above >= k) c = 2;
            cls[e] = c;
            if (c == 1) atomicAdd(&s_in, 1);
            if (c == 3) atomicAdd(&s_cand, 1);
        }
        __syncthreads();
        // exact keys of the candidates: one warp per candidate
        for (int e = warp; e < E; e += FB_THREADS / 32) {
            if (cls[e] != 3) continue;
            double acc = 0.0;
            for (int j = lane; j < d; j += 32)
                acc += static_cast<double>(__bfloat162float(x[(int64_t)t * d + j])) *
                       static_cast<double>(Wr[(int64_t)j * E + e]);
#pragma unroll
            for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            if (lane == 0) exk[e] = 1.0 / (1.0 + exp(-acc)) + static_cast<double>(b[e]);
        }
        __syncthreads();
        if (tid == 0) {
            const int need = k - s_in;
            if (need < 0 || need > s_cand) report(st, MOEVIE_ERR_DEVICE, SITE_ROUTE_FALLBACK, t, need);
            for (int r = 0; r < need; ++r) {
                int best = -1;
                for (int e = 0; e < E; ++e)
                    if (cls[e] == 3 && (best < 0 || exk[e] > exk[best])) best = e;
                if (best < 0) break;
                cls[best] = 4;
            }
            float ssum = 0.f;
            for (int e = 0; e < E; ++e)
                if (cls[e] == 1 || cls[e] == 4) ssum += sg[e];
            int pos = 0;
            for (int e = 0; e < E && pos < k; ++e)
                if (cls[e] == 1 || cls[e] == 4) {
                    idx[(int64_t)t * k + pos] = e;
                    gate[(int64_t)t * k + pos] = sg[e] / ssum;
                    ++pos;
                }
            for (; pos < k; ++pos) {   // only after a reported inconsistency
                idx[(int64_t)t * k + pos] = 0;
                gate[(int64_t)t * k + pos] = 0.f;
            }
        }
        __syncthreads();
    }
}

}  // namespace

cudaError_t launch_route_logits(const __nv_bfloat16* x, const float* Wr, int T, int d, int E,
                                const RouteBufs& rb, DevStatus* st, cudaStream_t s) {
    dim3 grid((T + LG_TT - 1) / LG_TT, (E + LG_TE - 1) / LG_TE);
    route_logits_kernel<<<grid, 256, 0, s>>>(x, Wr, T, d, E, rb.logits, rb.xnorm2, rb.wnorm2, st);
    count_launches(1);
    return cudaGetLastError();
}

cudaError_t launch_route_select(const __nv_bfloat16* x, const float* Wr, const float* b, int T,
                                int d, int E, int k, int32_t* idx, float* gate,
                                const RouteBufs& rb, DevStatus* st, int num_sms, cudaStream_t s) {
    const int blocks = (int)(((int64_t)T * 32 + 255) / 256);
    const int npl = (E + 31) / 32;
#define MV_TOPK(N)                                                                            \
    route_topk_kernel<N><<<blocks, 256, 0, s>>>(rb.logits, b, rb.xnorm2, rb.wnorm2, T, E, k, \
                                                idx, gate, rb.fb_tokens, st)
    if (npl <= 1) MV_TOPK(1);
    else if (npl <= 2) MV_TOPK(2);
    else if (npl <= 4) MV_TOPK(4);
    else if (npl <= 8) MV_TOPK(8);
    else if (npl <= 16) MV_TOPK(16);
    else MV_TOPK(32);
#undef MV_TOPK
    cudaError_t err = cudaGetLastError();
    if (err != cudaSuccess) return err;
    const size_t smem = (size_t)E * (8 + 4 + 4 + 1);
    const int fb_grid = T < 2 * num_sms ? T : 2 * num_sms;
    route_fallback_kernel<<<fb_grid, FB_THREADS, smem, s>>>(x, Wr, b, rb.logits, rb.xnorm2,
                                                            rb.wnorm2, d, E, k, idx, gate,
                                                            rb.fb_tokens, st);
    count_launches(2);
    return cudaGetLastError();
}

}  // namespace mv
