// route.cu -- router of the MoE-ViE layer (Eqs. 1, 7, 4-5), sm_103a.
//
// The logits s = x . W_r run on the tensor cores (grouped_gemm_kernel, one dense
// group): W_r is split exactly into bf16 pieces, W_r = hi + mid + lo, and the GEMM
// accumulates the fast logits x . (hi + mid) in fp32 (each piece padded to a multiple of
// 64 rows with zeros; for E <= 128 the two pieces sit side by side along N and the
// epilogue adds them, otherwise one after another along K).  Every product of a bf16 x
// and a bf16 piece is exact in fp32, so the error is the fp32 accumulation plus the
// left-out x . lo, which Cauchy-Schwarz bounds by |x_t| |lo_e| (lo holds the last 8 of
// w's 24 significand bits).  When there are few tokens, K is split over several CTA
// pairs (route_ksplit) and each split writes its own fp32 partial logits; they are summed
// in a fixed order.  This file holds the steps around that GEMM:
//
//  1. route_split_kernel: the two pieces, an fp32 copy of W_r transposed to
//     [E][d_pad] (read by the exact re-decision), and per-CTA partial sums of squares
//     of W_r's columns and of lo's (the router GEMM's idle warps finish |W_r[:, e]| and
//     |lo_e| from them).
//  2. route_topk_kernel: one warp per token; the partial logits summed, keys
//     sigmoid(s) + b, k rounds of warp arg-max (ties to the lower id), and a
//     certificate.  Every expert's key lies in
//     [key_e - tau_e, key_e + tau_e]; tau_e is the logit error bound (logit_tau) times
//     the largest sigmoid slope inside the logit interval, plus fp32 evaluation slack.
//     The selection is certain when the lowest selected lower end is above the highest
//     unselected upper end (tried first with the slope bound 1/4, then with the exact
//     slope).  Certified tokens write ascending ids and gates sigmoid(s) / sum (the bias
//     only selects).
//  3. route_fallback_kernel: one CTA per uncertified token.  An expert is surely in
//     when its lower end is above the k-th largest upper end of the others, surely
//     out when its upper end is below the k-th largest lower end; the rest get exact
//     logits (each product of a bf16 and an fp32 value is an integer of at most 32 bits
//     times a power of two; the CTA sums them in 128-bit fixed-point accumulators on
//     the integer pipes, see long_acc_term), and the remaining places are filled from
//     their keys (fp64), ties to the lower id.
#include <math.h>

#include "internal.h"

namespace mv {

namespace {

constexpr int SPLIT_TILE = 32;    // W_r rows (and experts) per CTA of the split kernel

// CTA (bx, by): experts 32 bx .. +31 and rows 32 by .. +31 of W_r (rows past d are
// zero); 32 x 8 threads.  Writes the two bf16 pieces hi, mid, the transposed fp32 copy
// and the CTA's partial sums of w^2 and of lo^2 per expert (lo = w - hi - mid, the
// piece the fast logits leave out).
__global__ void __launch_bounds__(256) route_split_kernel(const float* __restrict__ Wr, int d,
                                                          int dp, int E, int Ep,
                                                          __nv_bfloat16* __restrict__ Wsplit,
                                                          float* __restrict__ wrt,
                                                          float* __restrict__ wpart, int parts,
                                                          int32_t* __restrict__ wexp,
                                                          DevStatus* st, int concat) {
    pdl_wait();
    if (st && blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) st->fb_count = 0;
    __shared__ float tile[SPLIT_TILE][SPLIT_TILE + 1];
    __shared__ float red[2][8][32];
    __shared__ int redx[8][32];
    const int tx = threadIdx.x & 31, ty = threadIdx.x >> 5;
    const int e = blockIdx.x * SPLIT_TILE + tx;
    const int i0 = blockIdx.y * SPLIT_TILE;
    // piece p of element (i, e): [p][dp][Ep] (along K), or [dp][2 Ep] (side by side along N)
    const size_t piece = concat ? (size_t)Ep : (size_t)dp * Ep;
    const size_t row = concat ? (size_t)2 * Ep : (size_t)Ep;
    float sq = 0.f, sql = 0.f;
    int ex = 1;   // largest exponent field (subnormals and zero count as 1)
#pragma unroll
    for (int r = ty; r < SPLIT_TILE; r += 8) {
        const int i = i0 + r;
        const float w = (e < E && i < d) ? Wr[(int64_t)i * E + e] : 0.f;
        ex = max(ex, (int)((__float_as_uint(w) >> 23) & 0xffu));
        const __nv_bfloat16 hi = __float2bfloat16_rn(w);
        const float r1 = w - __bfloat162float(hi);                 // exact
        const __nv_bfloat16 mid = __float2bfloat16_rn(r1);
        const float lo = r1 - __bfloat162float(mid);               // exact
        if (e < Ep) {
            const size_t o = (size_t)i * row + e;
            Wsplit[o] = hi;
            Wsplit[piece + o] = mid;
        }
        tile[r][tx] = w;
        sq = fmaf(w, w, sq);
        sql = fmaf(lo, lo, sql);
    }
    red[0][ty][tx] = sq;
    red[1][ty][tx] = sql;
    redx[ty][tx] = ex;
    __syncthreads();
    if (ty < 2 && e < Ep) {
        float v = 0.f;
        for (int q = 0; q < 8; ++q) v += red[ty][q][tx];
        wpart[((int64_t)ty * parts + blockIdx.y) * Ep + e] = v;
    } else if (ty == 2 && e < Ep) {
        int m = 1;
        for (int q = 0; q < 8; ++q) m = max(m, redx[q][tx]);
        wexp[(int64_t)blockIdx.y * Ep + e] = m;
    }
#pragma unroll
    for (int r = ty; r < SPLIT_TILE; r += 8) {
        const int ee = blockIdx.x * SPLIT_TILE + r;
        if (ee < E) wrt[(int64_t)ee * dp + i0 + tx] = tile[tx][r];
    }
}

// Fast sigmoid: __expf (ex2.approx) and __fdividef.  For the keys compared below
// its absolute error stays under 1e-6, inside ROUTE_KEY_SLACK (2e-6): the relative
// error of e^{-v} is at most |v| log2(e) 2^-24 + 2^-22 and enters the sigmoid
// multiplied by s(1 - s) <= 1/4 (and by e^{-|v|} for large |v|); the division adds
// two ulp.
__device__ __forceinline__ float sigmoid_fast(float v) {
    return __fdividef(1.0f, 1.0f + __expf(-v));
}

// Logit error bound of expert e for a token (internal.h): the accumulation error
// ROUTE_TAU_C 2^-24 |x_t| (|W_r[:, e]| + |lo_e|) plus the left-out piece |x_t| |lo_e|,
// rounded up by the factor 1.001: the norms are fp32 sums of squares along chains far
// shorter than 2^14 terms, so their relative error (and that of the few operations
// here) stays below 2^-10.
__device__ __forceinline__ float logit_tau(float xn, float wn, float wl) {
    return (ROUTE_TAU_C * 5.9604645e-8f * (wn + wl) + wl) * xn * 1.001f;
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

// Order-preserving code of a float (larger float, larger code; no NaNs here).
__device__ __forceinline__ uint32_t ord_f32(float f) {
    const uint32_t u = __float_as_uint(f);
    return u ^ ((u & 0x80000000u) ? 0xffffffffu : 0x80000000u);
}

__device__ __forceinline__ float from_ord_f32(uint32_t c) {
    return __uint_as_float(c ^ ((c & 0x80000000u) ? 0x80000000u : 0xffffffffu));
}

// k-th and (k+1)-th largest of v over the warp, counting equal values separately
// (k or k + 1 rounds: warp maximum of the order codes by redux.sync, then one holder
// of that maximum leaves; k <= E).
template <int NPL>
__device__ __forceinline__ void warp_kth_values(const float (&v)[NPL], int E, int k, int lane,
                                                float& kth, float& kth1) {
    uint32_t code[NPL];
#pragma unroll
    for (int i = 0; i < NPL; ++i) code[i] = (lane + 32 * i < E) ? ord_f32(v[i]) : 0u;
    uint32_t used = 0;
    kth = -INFINITY;
    kth1 = -INFINITY;
    const int rounds = k < E ? k + 1 : k;
    for (int j = 0; j < rounds; ++j) {
        uint32_t best = 0;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const uint32_t c = ((used >> i) & 1u) ? 0u : code[i];
            best = c > best ? c : best;
        }
        best = __reduce_max_sync(0xffffffffu, best);
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const uint32_t m = __ballot_sync(0xffffffffu, !((used >> i) & 1u) && code[i] == best);
            if (m) {
                if (lane == __ffs(m) - 1) used |= 1u << i;
                break;
            }
        }
        const float bv = from_ord_f32(best);
        if (j == k - 1) kth = bv;
        if (j == k) kth1 = bv;
    }
}

// Exact logits by a long fixed-point accumulator (the exact dot product of Kulisch
// and Miranker, with a window fitted to the operands).  A bf16 x_i is mx 2^(ex - 134)
// and an fp32 w_i is mw 2^(ew - 150) (mx < 2^8, mw < 2^24 integers; ex, ew the biased
// exponents, 1 for subnormals), so x_i w_i = P 2^(q - 284) with the integer P = mx mw
// < 2^32 and q = ex + ew.  With a window Q >= every q, the term is P 2^(64 - (Q - q))
// units of 2^(Q - 348): a left shift (exact) when Q - q <= 64, else a right shift that
// drops less than one unit.  The units of d terms sum in a 128-bit integer (|sum| <
// 2^120 for d < 2^24), exactly and in any order; the logit is that sum times
// 2^(Q - 348), within d 2^(Q - 348) + 2^-51 |s| of the exact value.  Everything but the
// final conversion runs on the integer pipes.
__device__ __forceinline__ int bf16_exp_field(uint32_t hx) { return (int)((hx >> 7) & 0xffu); }
__device__ __forceinline__ int f32_exp_field(uint32_t uw) { return (int)((uw >> 23) & 0xffu); }

// acc += x w in units of 2^(Q - 348) (hx: bf16 bits of x, uw: fp32 bits of w).
__device__ __forceinline__ void long_acc_term(uint32_t hx, uint32_t uw, int Q, unsigned __int128& acc) {
    const int ex = bf16_exp_field(hx), ew = f32_exp_field(uw);
    const uint64_t mx = (hx & 0x7fu) | (ex ? 0x80u : 0u);
    const uint64_t mw = (uw & 0x7fffffu) | (ew ? 0x800000u : 0u);
    const uint64_t P = mx * mw;
    const int sh = 64 - (Q - (max(ex, 1) + max(ew, 1)));   // <= 64
    unsigned __int128 t;
    if (sh >= 0) t = (unsigned __int128)P << sh;
    else t = sh > -64 ? (unsigned __int128)(P >> -sh) : (unsigned __int128)0;
    if ((hx ^ (uw >> 16)) & 0x8000u) acc -= t;
    else acc += t;
}

__device__ __forceinline__ unsigned __int128 warp_sum_u128(unsigned __int128 v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) {
        const uint64_t lo = __shfl_xor_sync(0xffffffffu, (unsigned long long)(uint64_t)v, o);
        const uint64_t hi = __shfl_xor_sync(0xffffffffu, (unsigned long long)(uint64_t)(v >> 64), o);
        v += ((unsigned __int128)hi << 64) | lo;
    }
    return v;
}

// The signed 128-bit sum `u` (two's complement) times 2^(Q - 348), in double: the
// magnitude's two 64-bit words are rounded and added (relative error below 3 2^-53).
__device__ __forceinline__ double long_acc_value(unsigned __int128 u, int Q) {
    const bool neg = (long long)(uint64_t)(u >> 64) < 0;
    const unsigned __int128 m = neg ? (unsigned __int128)0 - u : u;
    const double hi = (double)(unsigned long long)(uint64_t)(m >> 64);
    const double lo = (double)(unsigned long long)(uint64_t)m;
    const double v = fma(hi, 18446744073709551616.0, lo);   // hi 2^64 + lo
    // 2^(Q - 348) with 2 <= Q <= 508: a normal double, so the product is exact
    const double r = v * __longlong_as_double((long long)((uint64_t)(Q - 348 + 1023) << 52));
    return neg ? -r : r;
}

// One warp per token.  NPL = experts per lane (expert e sits in lane e % 32, slot e / 32).
// s holds nparts partial logit arrays, part p at s + p * part_stride.  Each of the k
// selection rounds takes the warp maximum of the keys' order codes (redux.sync) and
// then the lowest id holding it (ballots in slot order), so ties go to the lower id.
// A token the certificate cannot settle is listed for route_fallback_kernel.
template <int NPL>
__global__ void __launch_bounds__(256) route_topk_kernel(
    const __nv_bfloat16* __restrict__ x, float* __restrict__ s, int ld, int nparts,
    int64_t part_stride, const float* __restrict__ b, const float* __restrict__ wnorm, int T,
    int d, int E, int k, int32_t* __restrict__ idx, float* __restrict__ gate,
    const float* __restrict__ xnorm, int32_t* __restrict__ fb_tokens, DevStatus* st,
    float4* __restrict__ zero, int64_t zero_n4) {
    pdl_wait();
    // Side job: clear another buffer (the layer's fp32 y accumulator) with 16-byte
    // evict-first stores, grid-strided; this kernel leaves HBM mostly idle.
    if (zero) {
        const uint4 z = make_uint4(0u, 0u, 0u, 0u);
        const uint64_t pol = l2_policy_evict_first();
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < zero_n4;
             i += (int64_t)gridDim.x * blockDim.x)
            st_global_v4_hint(zero + i, z, pol);
    }
    const int lane = threadIdx.x & 31;
    const int t = (int)(((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5);
    if (t >= T) return;
    float* srow = s + (int64_t)t * ld;
    float sv[NPL];
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
        const int e = lane + 32 * i;
        sv[i] = e < E ? srow[e] : 0.f;
    }
    for (int q = 1; q < nparts; ++q) {
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const int e = lane + 32 * i;
            if (e < E) sv[i] += srow[q * part_stride + e];
        }
    }
    const float xn = xnorm[t];   // |x_t|, written by the router GEMM
    float sg[NPL], key[NPL], ts[NPL];
    uint32_t code[NPL];
#pragma unroll
    for (int i = 0; i < NPL; ++i) {
        const int e = lane + 32 * i;
        if (e < E) {
            sg[i] = sigmoid_fast(sv[i]);
            key[i] = sg[i] + b[e];
            ts[i] = logit_tau(xn, wnorm[e], wnorm[E + e]);
            code[i] = ord_f32(key[i]);
        } else {
            sg[i] = 0.f;
            key[i] = -INFINITY;
            ts[i] = 0.f;
            code[i] = 0;
        }
    }
    uint32_t taken = 0;
    for (int j = 0; j < k; ++j) {
        uint32_t best = 0;
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const uint32_t c = ((taken >> i) & 1u) ? 0u : code[i];
            best = c > best ? c : best;
        }
        best = __reduce_max_sync(0xffffffffu, best);
#pragma unroll
        for (int i = 0; i < NPL; ++i) {
            const uint32_t m = __ballot_sync(0xffffffffu, !((taken >> i) & 1u) && code[i] == best);
            if (m) {
                if (lane == __ffs(m) - 1) taken |= 1u << i;
                break;
            }
        }
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
        certain = __reduce_min_sync(0xffffffffu, ord_f32(lo_in)) >
                  __reduce_max_sync(0xffffffffu, ord_f32(hi_out));
    }
    if (!certain) {
        if (nparts > 1) {   // the re-decision reads the summed logits from part 0
#pragma unroll
            for (int i = 0; i < NPL; ++i) {
                const int e = lane + 32 * i;
                if (e < E) srow[e] = sv[i];
            }
        }
        if (lane == 0) {
            const int p = atomicAdd(&st->fb_count, 1);
            fb_tokens[p] = t;
        }
        return;
    }
    float ssum = 0.f;
#pragma unroll
    for (int i = 0; i < NPL; ++i) ssum += ((taken >> i) & 1u) ? sg[i] : 0.f;
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


// Exact re-decision of uncertified tokens, one CTA (8 warps) per token.  The CTA stages
// the token's x row in shared memory (16-byte loads) and finds its largest exponent
// field; warp 0 bounds the keys and lists the candidates; then the candidates' exact
// logits are formed FB_BATCH at a time by all 256 threads (threads over the d terms,
// one long accumulator per candidate and thread, then a warp sum and a sum over the 8
// warps, all exact), their keys in fp64; finally warp 0 fills the remaining places from
// the exact keys, ties to the lower id, and writes ids and gates.
//
// The window of candidate e is Q = qx + qw(e), qx the largest exponent field of x_t and
// qw(e) that of W_r[:, e] (both at least 1: subnormals and zeros count as exponent 1), so
// every term's q is at most Q and one pass over the terms suffices; the logit is within
// d 2^(Q - 348) + 2^-51 |s| of the exact value, and d 2^(Q - 348) <= d 2^-64
// |x_t|_inf |W_r[:, e]|_inf.  A non-finite x_t or column (exponent field 255) gives a
// NaN logit.
constexpr int FB_BATCH = 4;       // candidates per pass over the terms
constexpr int FB_X_SMEM = 16384;  // largest d whose x row is staged in shared memory
// CTAs per SM the re-decision keeps resident for E <= 256 (its registers allow five), so
// that up to five tokens per SM are re-decided at once
constexpr int FB_CTAS_PER_SM = 5;
template <int NPL>
__global__ void __launch_bounds__(256, (NPL <= 8 ? FB_CTAS_PER_SM : 1)) route_fallback_kernel(
    const __nv_bfloat16* __restrict__ x, const float* __restrict__ wrt, int dp,
    const int32_t* __restrict__ wexp, int wexp_parts, int Ep,
    const float* __restrict__ b, const float* __restrict__ s, int ld,
    const float* __restrict__ xnorm, const float* __restrict__ wnorm, int d, int E, int k,
    int32_t* __restrict__ idx, float* __restrict__ gate, const int32_t* __restrict__ fb_tokens,
    DevStatus* st) {
    pdl_wait();
    extern __shared__ __align__(16) uint16_t fb_x[];   // the token's x row when d <= FB_X_SMEM
    __shared__ int s_cand[32 * NPL];
    __shared__ double s_key[32 * NPL];
    __shared__ unsigned long long s_acc[8][FB_BATCH][2];
    __shared__ int s_q[FB_BATCH];
    __shared__ int s_ncand;
    __shared__ int s_qx;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const uint32_t lt = (1u << lane) - 1u;
    const int nfb = st->fb_count;
    const bool staged = d <= FB_X_SMEM;
    for (int f = blockIdx.x; f < nfb; f += gridDim.x) {
        const int t = fb_tokens[f];
        const uint16_t* xg = reinterpret_cast<const uint16_t*>(x) + (int64_t)t * d;
        if (threadIdx.x == 0) s_qx = 1;
        __syncthreads();
        if (warp > 0 || !staged) {   // warps 1-7 stage x_t while warp 0 bounds the keys
            int m = 1;
            const int nthr = staged ? (int)blockDim.x - 32 : (int)blockDim.x;
            const int tid = staged ? (int)threadIdx.x - 32 : (int)threadIdx.x;
            for (int i = tid; i < d / 8; i += nthr) {   // d % 8 == 0, rows 16-byte aligned
                const uint4 v = reinterpret_cast<const uint4*>(xg)[i];
                if (staged) reinterpret_cast<uint4*>(fb_x)[i] = v;
                const uint32_t w4[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
                for (int j = 0; j < 4; ++j)
                    m = max(m, max((int)((w4[j] >> 7) & 0xffu), (int)((w4[j] >> 23) & 0xffu)));
            }
            m = __reduce_max_sync(0xffffffffu, m);
            if (lane == 0) atomicMax(&s_qx, m);
        }
        float sv[NPL];
        uint32_t sure_in = 0, cand = 0;
        int need = 0;
        if (warp == 0) {
            const float xn = xnorm[t];
            float up[NPL], lo[NPL];
#pragma unroll
            for (int i = 0; i < NPL; ++i) {
                const int e = lane + 32 * i;
                if (e < E) {
                    sv[i] = s[(int64_t)t * ld + e];
                    const float key = sigmoid_fast(sv[i]) + b[e];
                    const float tk = key_tau_exact_slope(sv[i], logit_tau(xn, wnorm[e], wnorm[E + e]));
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
                const uint32_t m = __ballot_sync(0xffffffffu, (cand >> i) & 1u);
                if ((cand >> i) & 1u) s_cand[n_cand + __popc(m & lt)] = lane + 32 * i;
                n_cand += __popc(m);
            }
            need = k - n_in;
            const bool bad = need < 0 || need > n_cand;
            if (lane == 0) {
                if (bad) report(st, MOEVIE_ERR_DEVICE, SITE_ROUTE_FALLBACK, t, need);
                s_ncand = bad ? -1 : (need == 0 ? 0 : n_cand);
            }
        }
        __syncthreads();
        const int nc = s_ncand;
        const int qx = s_qx;
        const uint16_t* xs = staged ? fb_x : xg;
        for (int c0 = 0; c0 < nc; c0 += FB_BATCH) {
            const int cn = min(FB_BATCH, nc - c0);
            if (warp < cn) {   // warp c: the window of candidate c0 + c
                const int e = s_cand[c0 + warp];
                int qw = 1;
                for (int pp = lane; pp < wexp_parts; pp += 32) qw = max(qw, __ldg(wexp + (int64_t)pp * Ep + e));
                qw = __reduce_max_sync(0xffffffffu, qw);
                if (lane == 0) s_q[warp] = (qx == 255 || qw == 255) ? -1 : qx + qw;   // -1: NaN
            }
            __syncthreads();
            unsigned __int128 acc[FB_BATCH];
            int Q[FB_BATCH];
            const float* wc[FB_BATCH];
#pragma unroll
            for (int c = 0; c < FB_BATCH; ++c) {
                acc[c] = 0;
                Q[c] = c < cn ? s_q[c] : -1;
                wc[c] = wrt + (int64_t)s_cand[c0 + (c < cn ? c : 0)] * dp;
            }
            for (int i = threadIdx.x; i < d; i += blockDim.x) {
                const uint32_t hx = xs[i];
                uint32_t uw[FB_BATCH];
#pragma unroll
                for (int c = 0; c < FB_BATCH; ++c) uw[c] = Q[c] > 0 ? __float_as_uint(__ldg(wc[c] + i)) : 0u;
#pragma unroll
                for (int c = 0; c < FB_BATCH; ++c)
                    if (Q[c] > 0) long_acc_term(hx, uw[c], Q[c], acc[c]);
            }
#pragma unroll
            for (int c = 0; c < FB_BATCH; ++c) {
                if (Q[c] <= 0) continue;   // uniform over the CTA
                const unsigned __int128 a = warp_sum_u128(acc[c]);
                if (lane == 0) {
                    s_acc[warp][c][0] = (unsigned long long)(uint64_t)a;
                    s_acc[warp][c][1] = (unsigned long long)(uint64_t)(a >> 64);
                }
            }
            __syncthreads();
            if (warp == 0 && lane < cn) {   // candidate c0 + lane: the sum over the 8 warps
                const int q = s_q[lane];
                double v = __longlong_as_double(0x7ff8000000000000ll);
                if (q > 0) {
                    unsigned __int128 u = 0;
#pragma unroll
                    for (int w = 0; w < 8; ++w)
                        u += ((unsigned __int128)s_acc[w][lane][1] << 64) | s_acc[w][lane][0];
                    v = long_acc_value(u, q);
                }
                s_key[c0 + lane] = 1.0 / (1.0 + exp(-v)) + (double)b[s_cand[c0 + lane]];
            }
            __syncthreads();
        }
        if (warp == 0 && nc >= 0) {
            double exk[NPL];
            int base = 0;
#pragma unroll
            for (int i = 0; i < NPL; ++i) {
                const uint32_t m = __ballot_sync(0xffffffffu, (cand >> i) & 1u);
                exk[i] = ((cand >> i) & 1u && nc > 0) ? s_key[base + __popc(m & lt)] : -INFINITY;
                base += __popc(m);
            }
            // choose `need` candidates by exact key, ties to the lower id
            uint32_t chosen = sure_in;
            for (int r = 0; r < need; ++r) {
                double bv = -INFINITY;
                int bi = 0x7fffffff;
#pragma unroll
                for (int i = 0; i < NPL; ++i) {
                    const int e = lane + 32 * i;
                    if (((cand >> i) & 1u) && !((chosen >> i) & 1u) &&
                        (exk[i] > bv || bi == 0x7fffffff)) {
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
            int pbase = 0;
#pragma unroll
            for (int i = 0; i < NPL; ++i) {
                const uint32_t m = __ballot_sync(0xffffffffu, (chosen >> i) & 1u);
                if ((chosen >> i) & 1u) {
                    const int pos = pbase + __popc(m & lt);
                    idx[(int64_t)t * k + pos] = lane + 32 * i;
                    gate[(int64_t)t * k + pos] = __fdividef(sg[i], ssum);
                }
                pbase += __popc(m);
            }
        }
        __syncthreads();   // s_cand / s_key / s_ncand / s_qx / fb_x are reused by the next token
    }
}

// out[t, e] = sum of the nparts partial logits, in order (used for inspection).
__global__ void route_sum_parts_kernel(const float* __restrict__ s, int64_t part_stride,
                                       int nparts, int64_t n, float* __restrict__ out) {
    pdl_wait();
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n) return;
    float v = s[i];
    for (int q = 1; q < nparts; ++q) v += s[q * part_stride + i];
    out[i] = v;
}

}  // namespace

int route_split_parts(int d) { return route_dpad(d) / SPLIT_TILE; }

int route_ksplit(int64_t T, int d, int E) {
    int BN = 0, n_ntiles = 0;
    const bool cc = route_concat(E);
    choose_bn(cc ? 2 * route_epad(E) : E, &BN, &n_ntiles);
    const int64_t items = (T + GM_BM - 1) / GM_BM * n_ntiles;
    const int nkb = (cc ? 1 : 2) * route_dpad(d) / GM_BK;
    // work items to aim for: with the pieces side by side (K = d_pad) fewer, longer
    // splits pay (measured: c1 64 items 4.8 us faster than 160)
    const int64_t target = cc ? ROUTE_SPLIT_TARGET_CONCAT : ROUTE_SPLIT_TARGET;
    int64_t p = items > 0 ? (target + items - 1) / items : 1;
    if (p > nkb / 3) p = nkb / 3;   // at least three K blocks per split
    if (p > ROUTE_MAX_KSPLIT) p = ROUTE_MAX_KSPLIT;
    return p < 1 ? 1 : (int)p;
}

int64_t route_logits_rows(int64_t T, int d, int E) {
    (void)d;
    int BN = 0, n_ntiles = 0;
    choose_bn(E, &BN, &n_ntiles);
    const int64_t a = (int64_t)ROUTE_MAX_KSPLIT * T;
    const int64_t b = (ROUTE_SPLIT_TARGET + (T + GM_BM - 1) / GM_BM * n_ntiles) * GM_BM;
    return a < b ? a : b;
}

cudaError_t launch_route_split(const float* Wr, int d, int E, __nv_bfloat16* Wsplit, float* wrt,
                               float* wpart, int32_t* wexp, DevStatus* st, cudaStream_t s) {
    const int Ep = route_epad(E);
    const int parts = route_split_parts(d);
    cudaError_t e = launch_pdl(route_split_kernel, dim3((Ep + SPLIT_TILE - 1) / SPLIT_TILE, parts),
                               dim3(256), 0, s, Wr, d, route_dpad(d), E, Ep, Wsplit, wrt, wpart, parts,
                               wexp, st, route_concat(E) ? 1 : 0);
    count_launches(1);
    return e;
}

cudaError_t launch_route_sum_parts(const float* logits, int64_t part_stride, int nparts, int64_t n,
                                   float* out, cudaStream_t s) {
    const cudaError_t e = launch_pdl(route_sum_parts_kernel, dim3((unsigned)((n + 255) / 256)),
                                     dim3(256), 0, s, logits, part_stride, nparts, n, out);
    count_launches(1);
    return e;
}

cudaError_t launch_route_select(const __nv_bfloat16* x, const float* wrt, const float* b,
                                float* logits, int ld, int nparts, int64_t part_stride,
                                const float* wnorm, const int32_t* wexp, int T, int d, int E, int k,
                                int32_t* idx, float* gate, int32_t* fb_tokens, float* xnorm,
                                DevStatus* st, int num_sms, cudaStream_t s, float* zero,
                                int64_t zero_n) {
    const int blocks = (int)(((int64_t)T * 32 + 255) / 256);
    const int fb_per_sm = (E + 31) / 32 <= 8 ? FB_CTAS_PER_SM : 3;
    const int fb_blocks = T < fb_per_sm * num_sms ? T : fb_per_sm * num_sms;   // one resident wave
    const size_t fb_smem = d <= FB_X_SMEM ? (size_t)2 * d : 0;
    const int npl = (E + 31) / 32;
    const int dp = route_dpad(d);
    const int parts = route_split_parts(d), Ep = route_epad(E);
    cudaError_t e = cudaSuccess;
#define MV_ROUTE(N)                                                                                \
    do {                                                                                           \
        e = launch_pdl(route_topk_kernel<N>, dim3(blocks), dim3(256), 0, s, x, logits, ld, nparts,  \
                       part_stride, b, wnorm, T, d, E, k, idx, gate, (const float*)xnorm,           \
                       fb_tokens, st, reinterpret_cast<float4*>(zero), zero ? zero_n / 4 : 0);      \
        if (e == cudaSuccess)                                                                      \
            e = launch_pdl(route_fallback_kernel<N>, dim3(fb_blocks), dim3(256), fb_smem, s, x,    \
                           wrt, dp, wexp, parts, Ep, b, (const float*)logits, ld,                  \
                           (const float*)xnorm, wnorm, d, E, k, idx, gate,                          \
                           (const int32_t*)fb_tokens, st);                                         \
    } while (0)
    if (npl <= 1) MV_ROUTE(1);
    else if (npl <= 2) MV_ROUTE(2);
    else if (npl <= 4) MV_ROUTE(4);
    else if (npl <= 8) MV_ROUTE(8);
    else if (npl <= 16) MV_ROUTE(16);
    else MV_ROUTE(32);
#undef MV_ROUTE
    count_launches(2);
    return e;
}

}  // namespace mv
