// route.cu -- router of the MoE-ViE layer (Eqs. 1, 7, 4-5), sm_103a.
//
// The logits s = x . W_r run on the tensor cores (grouped_gemm_kernel, one dense
// group): W_r is split exactly into three bf16 pieces, W_r = hi + mid + lo, and
// the GEMM accumulates x . [hi; mid; lo] over K = 3 d_pad in fp32 (each piece padded
// to a multiple of 64 rows with zeros).  Every product of a
// bf16 x and a bf16 piece is exact in fp32, so the only error is the fp32
// accumulation.  This file holds the steps around that GEMM:
//
//  1. route_split_kernel / route_wnorm_kernel: the three pieces and |W_r[:, e]|.
//  2. route_topk_kernel: one warp per token; keys sigmoid(s) + b, k rounds of warp
//     arg-max (ties to the lower id), and a certificate.  Every expert's key lies in
//     [key_e - tau_e, key_e + tau_e]; tau_e is the logit error bound
//     (ROUTE_TAU_C 2^-24 |x_t| |W_r[:, e]|) times the largest sigmoid slope inside
//     the logit interval, plus fp32 evaluation slack.  The selection is certain when
//     the lowest selected lower end is above the highest unselected upper end (tried
//     first with the slope bound 1/4, then with the exact slope).  Certified tokens
//     write ascending ids and gates sigmoid(s) / sum (the bias only selects).
//  3. route_fallback_kernel: one warp per uncertified token.  An expert is surely in
//     when its lower end is above the k-th largest upper end of the others, surely
//     out when its upper end is below the k-th largest lower end; the rest get exact
//     logits (fp64: each product of a bf16 and an fp32 value is exact in double, and
//     the sum of d terms has relative error below d 2^-53), and the remaining places
//     are filled from them, ties to the lower id.
#include <math.h>

#include "internal.h"

namespace mv {

namespace {

constexpr int SPLIT_ROWS = 256;   // W_r rows per CTA of the split kernel

// CTA (bx, by): experts 32 bx .. +31, rows SPLIT_ROWS by .. +SPLIT_ROWS-1; 32 x 8 threads.
__global__ void __launch_bounds__(256) route_split_kernel(const float* __restrict__ Wr, int d,
                                                          int dp, int E, int Ep,
                                                          __nv_bfloat16* __restrict__ Wsplit,
                                                          float* __restrict__ wpart) {
    __shared__ float red[8][32];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int e = blockIdx.x * 32 + tx;
    const int i0 = blockIdx.y * SPLIT_ROWS;
    const int i1 = min(dp, i0 + SPLIT_ROWS);
    float sq = 0.f;
    if (e < Ep) {
        const size_t piece = (size_t)dp * Ep;
        for (int i = i0 + ty; i < i1; i += 8) {
            const float w = (e < E && i < d) ? Wr[(int64_t)i * E + e] : 0.f;
            const __nv_bfloat16 hi = __float2bfloat16_rn(w);
            const float r1 = w - __bfloat162float(hi);          // exact
            const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
            const __nv_bfloat16 lo = __float2bfloat16_rn(r1 - __bfloat162float(mid));   // exact
            const size_t o = (size_t)i * Ep + e;
            Wsplit[o] = hi;
            Wsplit[piece + o] = mid;
            Wsplit[2 * piece + o] = lo;
            sq = fmaf(w, w, sq);
        }
    }
    red[ty][tx] = sq;
    __syncthreads();
    if (ty == 0 && e < Ep) {
        float v = 0.f;
        for (int q = 0; q < 8; ++q) v += red[q][tx];
        wpart[(int64_t)blockIdx.y * Ep + e] = v;
    }
}

// |W_r[:, e]| from the per-CTA partial sums, in a fixed order.
__global__ void route_wnorm_kernel(const float* __restrict__ wpart, int nparts, int E, int Ep,
                                   float* __restrict__ wnorm) {
    const int e = blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= E) return;
    float v = 0.f;
    for (int p = 0; p < nparts; ++p) v += wpart[(int64_t)p * Ep + e];
    wnorm[e] = sqrtf(v);
}

// Fast sigmoid: __expf (ex2.approx) and __fdividef.  For the keys compared below
// its absolute error stays under 1e-6, inside ROUTE_KEY_SLACK (2e-6): the relative
// error of e^{-v} is at most |v| log2(e) 2^-24 + 2^-22 and enters the sigmoid
// multiplied by s(1 - s) <= 1/4 (and by e^{-|v|} for large |v|); the division adds
// two ulp.
__device__ __forceinline__ float sigmoid_fast(float v) {
    return __fdividef(1.0f, 1.0f + __expf(-v));
}

// Logit error bound of expert e for a token: ROUTE_TAU_C 2^-24 |x_t| |W_r[:, e]|.
__device__ __forceinline__ float logit_tau(float xn, float wn) {
    return ROUTE_TAU_C * 5.9604645e-8f * xn * wn;
}

// Key half-width with the largest sigmoid slope inside [s - tau_s, s + tau_s]
// (the slope s(1 - s) falls with |s|).
__device__ __forceinline__ float key_tau_exact_slope(float s, float tau_s) {
    const float z = fmaxf(fabsf(s) - tau_s, 0.f);
    const float sz = sigmoid_fast(z);
    return tau_s * (sz * (1.f - sz)) + ROUTE_KEY_SLACK;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// |x_t| by one warp (16-byte loads; d % 8 == 0).
__device__ __forceinline__ float row_norm(const __nv_bfloat16* xt, int d, int lane) {
    float acc = 0.f;
    for (int c = lane; c < d / 8; c += 32) {
        float v[8];
        unpack_bf16x8(*reinterpret_cast<const uint4*>(xt + 8 * c), v);
#pragma unroll
        for (int q = 0; q < 8; ++q) acc = fmaf(v[q], v[q], acc);
    }
    return sqrtf(warp_sum(acc));
}

// Warp arg-max of (value, id): largest value, ties to the lower id.
__device__ __forceinline__ void warp_argmax(float& v, int& id) {
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const float ov = __shfl_xor_sync(0xffffffffu, v, o);
        const int oi = __shfl_xor_sync(0xffffffffu, id, o);
        if (ov > v || (ov == v && oi < id)) {
            v = ov;
            id = oi;
        }
    }
}

// One warp per token.  NPL = experts per lane (expert e sits in lane e % 32, slot e / 32).
template <int NPL>
__global__ void __launch_bounds__(256) route_topk_kernel(
    const __nv_bfloat16* __restrict__ x, const float* __restrict__ s, int ld,
    const float* __restrict__ b, const float* __restrict__ wnorm, int T, int d, int E, int k,
    int32_t* __restrict__ idx, float* __restrict__ gate, float* __restrict__ xnorm,
    int32_t* __restrict__ fb_tokens, DevStatus* st) {
    const int lane = threadIdx.x & 31;
    const int t = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    if (t >= T) return;
    const float xn = row_norm(x + (int64_t)t * d, d, lane);
    if (lane == 0) xnorm[t] = xn;
    float sv[NPL], key[NPL], ts[NPL];
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
        const int e = lane + 32 * i;
        if (e < E) {
            sv[i] = s[(int64_t)t * ld + e];
            key[i] = sigmoid_fast(sv[i]) + b[e];
            ts[i] = logit_tau(xn, wnorm[e]);
        } else {
            sv[i] = 0.f;
            key[i] = -INFINITY;
            ts[i] = 0.f;
        }
    }
    uint32_t taken = 0;
    for (int j = 0; j < k; ++j) {
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
        warp_argmax(bv, bi);
        if ((bi & 31) == lane) taken |= 1u << (bi >> 5);
    }
    bool certain = k >= E;
    for (int pass = 0; pass < 2 && !certain; ++pass) {
        float lo_in = INFINITY, hi_out = -INFINITY;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const int e = lane + 32 * i;
            if (e >= E) continue;
            const float tk = pass == 0 ? 0.25f * ts[i] + ROUTE_KEY_SLACK
                                       : key_tau_exact_slope(sv[i], ts[i]);
            if ((taken >> i) & 1u) lo_in = fminf(lo_in, key[i] - tk);
            else hi_out = fmaxf(hi_out, key[i] + tk);
        }
#pragma unroll
        for (int o = 16; o; o >>= 1) {
            lo_in = fminf(lo_in, __shfl_xor_sync(0xffffffffu, lo_in, o));
            hi_out = fmaxf(hi_out, __shfl_xor_sync(0xffffffffu, hi_out, o));
        }
        certain = lo_in > hi_out;
    }
    if (!certain) {
        if (lane == 0) {
            const int p = atomicAdd(&st->fb_count, 1);
            fb_tokens[p] = t;
        }
        return;
    }
    float ssum = 0.f;
    float sg[NPL];
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
        sg[i] = ((taken >> i) & 1u) ? sigmoid_fast(sv[i]) : 0.f;
        ssum += sg[i];
    }
    ssum = warp_sum(ssum);
    const uint32_t lt = (1u << lane) - 1u;
    int base = 0;
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
        const uint32_t m = __ballot_sync(0xffffffffu, (taken >> i) & 1u);
        if ((taken >> i) & 1u) {
            const int pos = base + __popc(m & lt);
            idx[(int64_t)t * k + pos] = lane + 32 * i;
            gate[(int64_t)t * k + pos] = __fdividef(sg[i], ssum);
        }
        base += __popc(m);
    }
}

constexpr int FB_BATCH = 8;   // candidates whose exact logits are summed together

// k-th and (k+1)-th largest of v over the warp (k rounds of arg-max; k <= E).
template <int NPL>
__device__ __forceinline__ void warp_kth_values(const float (&v)[NPL], int E, int k, int lane,
                                                float& kth, float& kth1) {
    uint32_t used = 0;
    kth = -INFINITY;
    kth1 = -INFINITY;
    const int rounds = k < E ? k + 1 : k;
    for (int j = 0; j < rounds; ++j) {
        float bv = -INFINITY;
        int bi = 0x7fffffff;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const int e = lane + 32 * i;
            if (e < E && !((used >> i) & 1u) && (v[i] > bv || bi == 0x7fffffff)) {
                bv = v[i];
                bi = e;
            }
        }
        warp_argmax(bv, bi);
        if ((bi & 31) == lane) used |= 1u << (bi >> 5);
        if (j == k - 1) kth = bv;
        if (j == k) kth1 = bv;
    }
}

// Exact re-decision of uncertified tokens, one warp per token.
template <int NPL>
__global__ void __launch_bounds__(256) route_fallback_kernel(
    const __nv_bfloat16* __restrict__ x, const float* __restrict__ Wr,
    const float* __restrict__ b, const float* __restrict__ s, int ld,
    const float* __restrict__ xnorm, const float* __restrict__ wnorm, int d, int E, int k,
    int32_t* __restrict__ idx, float* __restrict__ gate, const int32_t* __restrict__ fb_tokens,
    DevStatus* st) {
    const int lane = threadIdx.x & 31;
    const int64_t wid = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int64_t nwarps = ((int64_t)gridDim.x * blockDim.x) >> 5;
    const int nfb = st->fb_count;
    for (int64_t f = wid; f < nfb; f += nwarps) {
        const int t = fb_tokens[f];
        const float xn = xnorm[t];
        float sv[NPL], up[NPL], lo[NPL];
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const int e = lane + 32 * i;
            if (e < E) {
                sv[i] = s[(int64_t)t * ld + e];
                const float key = sigmoid_fast(sv[i]) + b[e];
                const float tk = key_tau_exact_slope(sv[i], logit_tau(xn, wnorm[e]));
                up[i] = key + tk;
                lo[i] = key - tk;
            } else {
                sv[i] = 0.f;
                up[i] = lo[i] = -INFINITY;
            }
        }
        // k-th / (k+1)-th largest upper ends and k-th largest lower end
        float u_k, u_k1, l_k, l_k1;
        warp_kth_values<NPL>(up, E, k, lane, u_k, u_k1);
        warp_kth_values<NPL>(lo, E, k, lane, l_k, l_k1);
        uint32_t sure_in = 0, cand = 0;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const int e = lane + 32 * i;
            if (e >= E) continue;
            // k-th largest upper end among the others (u_k when e may sit at rank k: conservative)
            const float thr = up[i] > u_k ? u_k1 : u_k;
            if (k >= E || lo[i] > thr) sure_in |= 1u << i;
            else if (!(up[i] < l_k)) cand |= 1u << i;
        }
        int n_in = 0, n_cand = 0;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            n_in += __popc(__ballot_sync(0xffffffffu, (sure_in >> i) & 1u));
            n_cand += __popc(__ballot_sync(0xffffffffu, (cand >> i) & 1u));
        }
        const int need = k - n_in;
        if (need < 0 || need > n_cand) {
            if (lane == 0) report(st, MOEVIE_ERR_DEVICE, SITE_ROUTE_FALLBACK, t, need);
            continue;
        }
        // exact keys of the candidates, FB_BATCH at a time, lanes over d
        double exk[NPL];
#pragma unroll
        for (int i = 0; i < NPL; ++i) exk[i] = -INFINITY;
        for (int done = 0; done < n_cand;) {
            int ids[FB_BATCH];
            int nb = 0, seen = 0;
#pragma unroll
            for (int i = 0; i < NPL; ++i) {
                uint32_t m = __ballot_sync(0xffffffffu, (cand >> i) & 1u);
                while (m && nb < FB_BATCH) {
                    const int l = __ffs(m) - 1;
                    m &= m - 1;
                    if (seen++ >= done) ids[nb++] = l + 32 * i;
                }
            }
#pragma unroll
            for (int q = 0; q < FB_BATCH; ++q)
                if (q >= nb) ids[q] = ids[0];
            double acc[FB_BATCH];
#pragma unroll
            for (int q = 0; q < FB_BATCH; ++q) acc[q] = 0.0;
            for (int j = lane; j < d; j += 32) {
                const double xv = (double)__bfloat162float(x[(int64_t)t * d + j]);
                const float* wrow = Wr + (int64_t)j * E;
#pragma unroll
                for (int q = 0; q < FB_BATCH; ++q) acc[q] += xv * (double)wrow[ids[q]];
            }
#pragma unroll
            for (int q = 0; q < FB_BATCH; ++q) {
                double v = acc[q];
#pragma unroll
                for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                const int e = ids[q];
                if (q < nb && (e & 31) == lane) {
                    const double key = 1.0 / (1.0 + exp(-v)) + (double)b[e];
#pragma unroll
                    for (int i = 0; i < NPL; ++i)
                        if (i == (e >> 5)) exk[i] = key;
                }
            }
            done += nb;
        }
        // choose `need` candidates by exact key, ties to the lower id
        uint32_t chosen = sure_in;
        for (int r = 0; r < need; ++r) {
            double bv = -INFINITY;
            int bi = 0x7fffffff;
#pragma unroll
            for (int i = 0; i < NPL; ++i) {
                const int e = lane + 32 * i;
                if (((cand >> i) & 1u) && !((chosen >> i) & 1u) && (exk[i] > bv || bi == 0x7fffffff)) {
                    bv = exk[i];
                    bi = e;
                }
            }
#pragma unroll
            for (int o = 16; o; o >>= 1) {
                const double ov = __shfl_xor_sync(0xffffffffu, bv, o);
                const int oi = __shfl_xor_sync(0xffffffffu, bi, o);
                if (ov > bv || (ov == bv && oi < bi)) {
                    bv = ov;
                    bi = oi;
                }
            }
            if ((bi & 31) == lane) chosen |= 1u << (bi >> 5);
        }
        float sg[NPL];
        float ssum = 0.f;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            sg[i] = ((chosen >> i) & 1u) ? sigmoid_fast(sv[i]) : 0.f;
            ssum += sg[i];
        }
        ssum = warp_sum(ssum);
        const uint32_t lt = (1u << lane) - 1u;
        int base = 0;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const uint32_t m = __ballot_sync(0xffffffffu, (chosen >> i) & 1u);
            if ((chosen >> i) & 1u) {
                const int pos = base + __popc(m & lt);
                idx[(int64_t)t * k + pos] = lane + 32 * i;
                gate[(int64_t)t * k + pos] = __fdividef(sg[i], ssum);
            }
            base += __popc(m);
        }
    }
}

__global__ void reset_fallback_count(DevStatus* st) { st->fb_count = 0; }

}  // namespace

int route_split_parts(int d) { return (route_dpad(d) + SPLIT_ROWS - 1) / SPLIT_ROWS; }

cudaError_t launch_route_split(const float* Wr, int d, int E, __nv_bfloat16* Wsplit, float* wpart,
                               float* wnorm, cudaStream_t s) {
    const int Ep = route_epad(E);
    const int parts = route_split_parts(d);
    route_split_kernel<<<dim3((Ep + 31) / 32, parts), 256, 0, s>>>(Wr, d, route_dpad(d), E, Ep,
                                                                   Wsplit, wpart);
    route_wnorm_kernel<<<(E + 255) / 256, 256, 0, s>>>(wpart, parts, E, Ep, wnorm);
    count_launches(2);
    return cudaGetLastError();
}

cudaError_t launch_route_select(const __nv_bfloat16* x, const float* Wr, const float* b,
                                const float* logits, int ld, const float* wnorm, int T, int d,
                                int E, int k, int32_t* idx, float* gate, int32_t* fb_tokens,
                                float* xnorm, DevStatus* st, int num_sms, cudaStream_t s) {
    reset_fallback_count<<<1, 1, 0, s>>>(st);
    const int blocks = (int)(((int64_t)T * 32 + 255) / 256);
    const int64_t fb_warps = T < 16 * (int64_t)num_sms ? (int64_t)T : 16 * (int64_t)num_sms;
    const int fb_blocks = (int)((fb_warps * 32 + 255) / 256);
    const int npl = (E + 31) / 32;
#define MV_ROUTE(N)                                                                              \
    do {                                                                                         \
        route_topk_kernel<N><<<blocks, 256, 0, s>>>(x, logits, ld, b, wnorm, T, d, E, k, idx,    \
                                                    gate, xnorm, fb_tokens, st);                 \
        route_fallback_kernel<N><<<fb_blocks, 256, 0, s>>>(x, Wr, b, logits, ld, xnorm, wnorm, d, \
                                                           E, k, idx, gate, fb_tokens, st);      \
    } while (0)
    if (npl <= 1) MV_ROUTE(1);
    else if (npl <= 2) MV_ROUTE(2);
    else if (npl <= 4) MV_ROUTE(4);
    else if (npl <= 8) MV_ROUTE(8);
    else if (npl <= 16) MV_ROUTE(16);
    else MV_ROUTE(32);
#undef MV_ROUTE
    count_launches(3);
    return cudaGetLastError();
}

}  // namespace mv
