// backward.cu -- the training path of the MoE-ViE layer (App. B: grouped GEMMs with the
// activation as a separate step; gradients of sum_t dy_t . y_t with the top-k selection
// held fixed, through the renormalised gates of Eqs. 4-5 into W_r and x), sm_103a.
//
// The grouped GEMMs run on grouped_gemm_kernel (gemm.cu); this file holds the steps
// around them, all memory- or latency-bound:
//   bwd_gates_kernel   per token, the fp32 logits of its k selected experts (W_r's
//                      transposed copy), sigma, their sum S and the gates g = sigma / S
//   bwd_pad_kernel     expert segments padded to multiples of 64 rows (the K blocks of
//                      the weight-gradient GEMMs never straddle two experts)
//   bwd_rows_kernel    per padded row its token (-1 for padding) and gate (0), and per
//                      routing slot its padded row
//   bwd_items_kernel   the weight-gradient work items {g, m0 | n0 << 16, kb0, kb1}: per
//                      group, output tiles x chunks of at most BWD_KCH k-blocks (a group of
//                      one chunk stores its gradient instead of adding into it)
//   bwd_zero_kernel    clears what the items will add into or not write: the gradients of
//                      groups with no rows or several chunks, and pad columns
//   bwd_gather_kernel  the padded rows of x and of g dy (bf16; zero rows for padding)
//   bwd_router_kernel  per token: dg_j = dy . E_j(x) from the partial row dots, the gate
//                      derivative ds (Eqs. 4-5), dx += ds W_r^T, and ds into a dense
//                      [T][E_pad] bf16 matrix for dW_r = x^T ds
#include <math.h>

#include <algorithm>

#include "internal.h"

namespace mv {

namespace {

__device__ __forceinline__ float warp_sum_f(float v) {
#pragma unroll
    for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

// One warp per token: s_j = x_t . W_r[:, e_j] for its k experts (fp32, lanes over d; the
// k dot products advance together, so each lane has k loads in flight per step),
// sigma_j = 1 / (1 + e^-s_j), S = sum_j sigma_j, g_j = sigma_j / S.  KB >= k.
template <int KB>
__global__ void __launch_bounds__(256) bwd_gates_kernel(const __nv_bfloat16* __restrict__ x,
                                                        const float* __restrict__ wrt, int dp,
                                                        const int32_t* __restrict__ idx, int64_t T,
                                                        int d, int E, int k, float* __restrict__ sig,
                                                        float* __restrict__ gate, DevStatus* st) {
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t t = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (t >= T) return;
    const __nv_bfloat16* xr = x + t * d;
    const float* w[KB];
    float acc[KB];
#pragma unroll
    for (int j = 0; j < KB; ++j) {
        acc[j] = 0.f;
        const int e = j < k ? idx[t * k + j] : 0;
        const bool ok = e >= 0 && e < E;
        if (j < k && !ok && lane == 0) report(st, MOEVIE_ERR_DEVICE, SITE_PERMUTE_ID, (int)(t * k + j), e);
        w[j] = (j < k && ok) ? wrt + (int64_t)e * dp : nullptr;
    }
    for (int i = lane; i < d; i += 32) {
        const float xi = __bfloat162float(xr[i]);
#pragma unroll
        for (int j = 0; j < KB; ++j)
            if (w[j]) acc[j] = fmaf(xi, __ldg(w[j] + i), acc[j]);
    }
    float ssum = 0.f, mine = 0.f;   // lane j keeps sigma_j
#pragma unroll
    for (int j = 0; j < KB; ++j) {
        if (j >= k) break;
        const float sgm = 1.0f / (1.0f + expf(-warp_sum_f(acc[j])));
        if (lane == j) mine = sgm;
        ssum += sgm;
    }
    if (lane < k) {
        sig[t * k + lane] = mine;
        gate[t * k + lane] = mine / ssum;
    }
}

// One CTA of 1024 threads (E <= 1024): poff[e] = sum over e' < e of counts rounded up to
// 64 rows, poff[E] the padded total.
__global__ void __launch_bounds__(1024) bwd_pad_kernel(const int32_t* __restrict__ counts, int E,
                                                       int32_t* __restrict__ poff) {
    pdl_wait();
    __shared__ int wsum[32];
    const int e = threadIdx.x, lane = e & 31, warp = e >> 5;
    const int v = e < E ? (counts[e] + 63) / 64 * 64 : 0;
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
    }
    __syncthreads();
    const int ex = wsum[warp] + inc - v;
    if (e < E) poff[e] = ex;
    if (e == E - 1) poff[E] = ex + v;
}

// Threads over routing slots (t, j) and over (expert, padding row < 64): the padded row of
// slot t k + j is poff[e] + (its expert-major row - offsets[e]); padding rows of expert e
// (poff[e] + counts[e] .. poff[e + 1] - 1) get token -1 and gate 0.
__global__ void bwd_rows_kernel(const int32_t* __restrict__ idx, const int32_t* __restrict__ inv,
                                const int32_t* __restrict__ counts, const int32_t* __restrict__ offsets,
                                const int32_t* __restrict__ poff, const float* __restrict__ gate,
                                int64_t n_slots, int k, int E, int32_t* __restrict__ ptok,
                                float* __restrict__ pgate, int32_t* __restrict__ slot_prow) {
    pdl_wait();
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i < n_slots) {
        const int e = idx[i];
        const int r = inv[i];
        if (e >= 0 && e < E && r >= 0) {
            const int pr = poff[e] + (r - offsets[e]);
            ptok[pr] = (int32_t)(i / k);
            pgate[pr] = gate[i];
            slot_prow[i] = pr;
        } else {
            slot_prow[i] = -1;
        }
    }
    if (i < (int64_t)E * 64) {
        const int e = (int)(i >> 6), j = (int)(i & 63);
        const int pr = poff[e] + counts[e] + j;
        if (pr < poff[e + 1]) {
            ptok[pr] = -1;
            pgate[pr] = 0.f;
        }
    }
}

// One CTA of 1024 threads, one thread per group (G <= 1024): group g has the k-blocks
// [koff[g] / 64, koff[g + 1] / 64) (koff == nullptr: one group of ceil(K_rows / 64)
// k-blocks), cut into chunks of at most kch; its items are every (m-tile of 256 of M rows,
// n-tile of BN of N columns, chunk).  items[i] = {g, m0 | n0 << 16, kb0, kb1}; *n_items =
// their number (at most max_items; more is a device error and none are listed).  A group
// of one chunk writes each of its gradient's elements once: its items carry
// BWD_STORE_BIT in kb1 (the GEMM stores instead of adding) and gclear[g] = 0; a group
// with no rows or several chunks has gclear[g] = 1 (its gradient is cleared first).
__global__ void __launch_bounds__(1024) bwd_items_kernel(const int32_t* __restrict__ koff, int G,
                                                         int64_t K_rows, int M, int N, int BN, int kch,
                                                         int max_items, int4* __restrict__ items,
                                                         int32_t* __restrict__ n_items,
                                                         int32_t* __restrict__ gclear, DevStatus* st) {
    pdl_wait();
    __shared__ int wsum[32];
    __shared__ int s_total;
    const int g = threadIdx.x, lane = g & 31, warp = g >> 5;
    const int mt = (M + GM_BM - 1) / GM_BM, nt = (N + BN - 1) / BN;
    int kb0 = 0, kb1 = 0;
    if (g < G) {
        if (koff) {
            kb0 = koff[g] / GM_BK;
            kb1 = koff[g + 1] / GM_BK;
        } else {
            kb1 = (int)((K_rows + GM_BK - 1) / GM_BK);
        }
    }
    const int chunks = kb1 > kb0 ? (kb1 - kb0 + kch - 1) / kch : 0;
    const int v = chunks * mt * nt;
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
        if (lane == 31) s_total = wi;
    }
    __syncthreads();
    const int total = s_total;
    if (total > max_items) {
        if (g == 0) {
            report(st, MOEVIE_ERR_DEVICE, SITE_GEMM_TILES, total, max_items);
            *n_items = 0;
        }
        return;
    }
    int pos = wsum[warp] + inc - v;
    const int store = chunks == 1 ? BWD_STORE_BIT : 0;
    for (int c = 0; c < chunks; ++c) {
        const int a = kb0 + c * kch, b = min(kb1, a + kch);
        for (int m = 0; m < mt; ++m)
            for (int n = 0; n < nt; ++n)
                items[pos++] = make_int4(g, (m * GM_BM) | ((n * BN) << 16), a, b | store);
    }
    if (g < G) gclear[g] = chunks == 1 ? 0 : 1;
    if (g == 0) *n_items = total;
}

// The part of a weight gradient out [G][M][ld] (fp32) that the GEMM's items will not
// write: every row of a group with gclear[g] set, and the pad columns [N, ld) of the
// other groups' rows.  One warp per row, grid-strided; ld % 4 == 0.
__global__ void __launch_bounds__(256) bwd_zero_kernel(const int32_t* __restrict__ gclear, int G, int M,
                                                       int N, int64_t ld, float* __restrict__ out) {
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t rows = (int64_t)G * M;
    for (int64_t q = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; q < rows;
         q += ((int64_t)gridDim.x * blockDim.x) >> 5) {
        float* row = out + q * ld;
        if (gclear[q / M]) {
            float4* r4 = reinterpret_cast<float4*>(row);
            for (int64_t c = lane; c < ld / 4; c += 32) r4[c] = make_float4(0.f, 0.f, 0.f, 0.f);
        } else {
            for (int64_t c = N + lane; c < ld; c += 32) row[c] = 0.f;
        }
    }
}

// Padded rows r (threads over r and 8-column groups): xp[r] = x[ptok[r]], gdy[r] =
// pgate[r] dy[ptok[r]] (bf16), zero rows where ptok[r] < 0.
__global__ void bwd_gather_kernel(const __nv_bfloat16* __restrict__ x, const __nv_bfloat16* __restrict__ dy,
                                  const int32_t* __restrict__ ptok, const float* __restrict__ pgate,
                                  const int32_t* __restrict__ poff, int E, int d,
                                  __nv_bfloat16* __restrict__ xp, __nv_bfloat16* __restrict__ gdy) {
    pdl_wait();
    const int64_t rows = poff[E];
    const int cpr = d / 8;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < rows * cpr;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / cpr;
        const int c = (int)(i - r * cpr) * 8;
        const int t = ptok[r];
        uint4 xv = make_uint4(0u, 0u, 0u, 0u), gv = xv;
        if (t >= 0) {
            xv = *reinterpret_cast<const uint4*>(x + (int64_t)t * d + c);
            float f[8];
            unpack_bf16x8(*reinterpret_cast<const uint4*>(dy + (int64_t)t * d + c), f);
            const float g = pgate[r];
            gv.x = pack_bf16x2(g * f[0], g * f[1]);
            gv.y = pack_bf16x2(g * f[2], g * f[3]);
            gv.z = pack_bf16x2(g * f[4], g * f[5]);
            gv.w = pack_bf16x2(g * f[6], g * f[7]);
        }
        *reinterpret_cast<uint4*>(xp + r * d + c) = xv;
        *reinterpret_cast<uint4*>(gdy + r * d + c) = gv;
    }
}

// One warp per token (Eqs. 4-5 backward): dg_j = sum of the nparts partial row dots of
// its padded row, gdg = sum_j g_j dg_j, ds_j = sigma_j (1 - sigma_j) (dg_j - gdg) / S;
// dx_t += sum_j ds_j W_r[:, e_j] (after the grouped dx GEMM, same stream; the k columns
// advance together), and ds_j into ds[t][e_j] (bf16, the rest of the row already zero).
template <int KB>
__global__ void __launch_bounds__(256) bwd_router_kernel(
    const int32_t* __restrict__ idx, const float* __restrict__ sig, const float* __restrict__ gate,
    const int32_t* __restrict__ slot_prow, const float* __restrict__ dg_part, int nparts,
    int64_t part_stride, const float* __restrict__ wrt, int dp, int64_t T, int d, int E, int k,
    int Ep, float* __restrict__ dx, __nv_bfloat16* __restrict__ ds_out) {
    pdl_wait();
    const int lane = threadIdx.x & 31;
    const int64_t t = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (t >= T) return;
    // lanes j < k hold slot j: its dg, sigma and gate
    float dg = 0.f, sg = 0.f, g = 0.f;
    int e = -1;
    if (lane < k) {
        const int pr = slot_prow[t * k + lane];
        e = idx[t * k + lane];
        sg = sig[t * k + lane];
        g = gate[t * k + lane];
        if (pr >= 0)
            for (int q = 0; q < nparts; ++q) dg += dg_part[(int64_t)q * part_stride + pr];
    }
    const float S = warp_sum_f(sg);
    const float gdg = warp_sum_f(g * dg);
    const float ds = lane < k ? sg * (1.f - sg) * (dg - gdg) / S : 0.f;
    if (lane < k && e >= 0 && e < E) ds_out[t * Ep + e] = __float2bfloat16_rn(ds);
    const float* w[KB];
    float dsj[KB];
#pragma unroll
    for (int j = 0; j < KB; ++j) {
        dsj[j] = __shfl_sync(0xffffffffu, ds, j);
        const int ej = __shfl_sync(0xffffffffu, e, j);
        w[j] = (j < k && ej >= 0 && ej < E) ? wrt + (int64_t)ej * dp : nullptr;
    }
    float* dxr = dx + t * d;
    for (int i = lane; i < d; i += 32) {
        float a = dxr[i];
#pragma unroll
        for (int j = 0; j < KB; ++j)
            if (w[j]) a = fmaf(dsj[j], __ldg(w[j] + i), a);
        dxr[i] = a;
    }
}

// dst[r][c] = src[r][c] for c < cols (src rows ld_src apart).
__global__ void bwd_copy_kernel(const float* __restrict__ src, int64_t ld_src, float* __restrict__ dst,
                                int64_t rows, int64_t cols) {
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < rows * cols;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int64_t r = i / cols, c = i - r * cols;
        dst[i] = src[r * ld_src + c];
    }
}

int grid_of(int64_t n, int threads) {
    int64_t g = (n + threads - 1) / threads;
    if (g > 152 * 16) g = 152 * 16;
    return (int)(g < 1 ? 1 : g);
}

}  // namespace

cudaError_t launch_bwd_gates(const __nv_bfloat16* x, const float* wrt, int dp, const int32_t* idx, int64_t T,
                             int d, int E, int k, float* sig, float* gate, DevStatus* st, cudaStream_t s) {
    const dim3 grid((unsigned)((T * 32 + 255) / 256));
    cudaError_t e;
    if (k <= 8) e = launch_pdl(bwd_gates_kernel<8>, grid, dim3(256), 0, s, x, wrt, dp, idx, T, d, E, k, sig, gate, st);
    else if (k <= 32) e = launch_pdl(bwd_gates_kernel<32>, grid, dim3(256), 0, s, x, wrt, dp, idx, T, d, E, k, sig, gate, st);
    else return cudaErrorInvalidValue;
    count_launches(1);
    return e;
}

cudaError_t launch_bwd_pad(const int32_t* counts, int E, int32_t* poff, cudaStream_t s) {
    const cudaError_t e = launch_pdl(bwd_pad_kernel, dim3(1), dim3(1024), 0, s, counts, E, poff);
    count_launches(1);
    return e;
}

cudaError_t launch_bwd_rows(const int32_t* idx, const int32_t* inv, const int32_t* counts,
                            const int32_t* offsets, const int32_t* poff, const float* gate, int64_t n_slots,
                            int k, int E, int32_t* ptok, float* pgate, int32_t* slot_prow, cudaStream_t s) {
    const int64_t n = n_slots > (int64_t)E * 64 ? n_slots : (int64_t)E * 64;
    const cudaError_t e = launch_pdl(bwd_rows_kernel, dim3((unsigned)((n + 255) / 256)), dim3(256), 0, s, idx,
                                     inv, counts, offsets, poff, gate, n_slots, k, E, ptok, pgate, slot_prow);
    count_launches(1);
    return e;
}

int64_t bwd_max_items(int64_t rows, int G, int M, int N, int BN) {
    const int64_t mt = (M + GM_BM - 1) / GM_BM, nt = (N + BN - 1) / BN;
    return ((rows + GM_BK * BWD_KCH - 1) / (GM_BK * BWD_KCH) + G) * mt * nt;
}

cudaError_t launch_bwd_items(const int32_t* koff, int G, int64_t K_rows, int M, int N, int BN,
                             int max_items, int4* items, int32_t* n_items, int32_t* gclear, DevStatus* st,
                             cudaStream_t s) {
    if (G > 1024) return cudaErrorInvalidValue;
    const cudaError_t e = launch_pdl(bwd_items_kernel, dim3(1), dim3(1024), 0, s, koff, G, K_rows, M, N, BN,
                                     (int)BWD_KCH, max_items, items, n_items, gclear, st);
    count_launches(1);
    return e;
}

cudaError_t launch_bwd_zero(const int32_t* gclear, int G, int M, int N, int64_t ld, float* out, int num_sms,
                            cudaStream_t s) {
    if (ld % 4 != 0 || N > ld) return cudaErrorInvalidValue;
    const int64_t warps = (int64_t)G * M;
    const int64_t blocks = std::min<int64_t>((warps + 7) / 8, (int64_t)num_sms * 8);
    const cudaError_t e = launch_pdl(bwd_zero_kernel, dim3((unsigned)std::max<int64_t>(blocks, 1)), dim3(256), 0, s,
                                     gclear, G, M, N, ld, out);
    count_launches(1);
    return e;
}

cudaError_t launch_bwd_gather(const __nv_bfloat16* x, const __nv_bfloat16* dy, const int32_t* ptok,
                              const float* pgate, const int32_t* poff, int E, int d, int64_t max_rows,
                              __nv_bfloat16* xp, __nv_bfloat16* gdy, cudaStream_t s) {
    const cudaError_t e = launch_pdl(bwd_gather_kernel, dim3(grid_of(max_rows * (d / 8), 256)), dim3(256), 0, s,
                                     x, dy, ptok, pgate, poff, E, d, xp, gdy);
    count_launches(1);
    return e;
}

cudaError_t launch_bwd_router(const int32_t* idx, const float* sig, const float* gate, const int32_t* slot_prow,
                              const float* dg_part, int nparts, int64_t part_stride, const float* wrt, int dp,
                              int64_t T, int d, int E, int k, int Ep, float* dx, __nv_bfloat16* ds,
                              cudaStream_t s) {
    const dim3 grid((unsigned)((T * 32 + 255) / 256));
    cudaError_t e;
    if (k <= 8)
        e = launch_pdl(bwd_router_kernel<8>, grid, dim3(256), 0, s, idx, sig, gate, slot_prow, dg_part, nparts,
                       part_stride, wrt, dp, T, d, E, k, Ep, dx, ds);
    else if (k <= 32)
        e = launch_pdl(bwd_router_kernel<32>, grid, dim3(256), 0, s, idx, sig, gate, slot_prow, dg_part, nparts,
                       part_stride, wrt, dp, T, d, E, k, Ep, dx, ds);
    else
        return cudaErrorInvalidValue;
    count_launches(1);
    return e;
}

cudaError_t launch_bwd_copy(const float* src, int64_t ld_src, float* dst, int64_t rows, int64_t cols,
                            cudaStream_t s) {
    const cudaError_t e = launch_pdl(bwd_copy_kernel, dim3(grid_of(rows * cols, 256)), dim3(256), 0, s, src,
                                     ld_src, dst, rows, cols);
    count_launches(1);
    return e;
}

}  // namespace mv
