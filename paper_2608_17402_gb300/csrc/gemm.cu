// gemm.cu -- persistent grouped GEMM on tcgen05 / TMEM for the expert FFN of the
// MoE-ViE layer (App. B, Algorithm 1, Kernels 1 and 2), sm_103a.
//
// One launch computes, for every group g (an expert) and every row r of its
// segment [offsets[g], offsets[g+1]):   D[r, :] = A[row(r), :] . B[g]   (fp32)
// and hands each 128 x BN tile to a fused epilogue:
//   EPI_GELU_BF16   hidden = bf16(GELU(D))                      (Kernel 1, GELU)
//   EPI_STORE_BF16  out    = bf16(D)
//   EPI_ADD_F32     y[tok(r)] += gate(r) * D   (Kernel 2: routing weight + scatter-add)
//   EPI_STORE_F32   y[tok(r)]  = scale * D     (first writer of y, e.g. the shared expert)
//
// Work items are (m-tile, n-tile) pairs of all groups, in group-major order with
// the n-tile fastest; a persistent CTA per SM walks them with a static stride.
// There is no host read of segment sizes: the m-tile list comes from the device
// prefix tile_off, written by the permute step.
//
// Warp roles (320 threads, one CTA per SM):
//   warps 0-3  epilogue: tcgen05.ld of the fp32 accumulator rows (warp w owns TMEM
//              lanes 32w..32w+31), fused math, global stores / vector atomics
//   warp 4     TMEM allocation; lane 0 issues tcgen05.mma (M=128, N=BN, K=16)
//   warp 5     lane 0 issues TMA loads of B tiles (weights, 128-byte swizzle)
//   warps 6-9  gather A rows with 16-byte cp.async straight into the 128-byte
//              swizzled K-major layout (the token gather fused into the operand load)
// Shared memory: GM_STAGES x (A 128x64 + B 64x256) bf16 stages; TMEM: two fp32
// accumulators of 256 columns, so the epilogue of one tile overlaps the
// main loop of the next.
//
// Operand layouts (tcgen05 shared-memory descriptors, 128-byte swizzle):
//   A  K-major : row r of the 128x64 tile at byte r*128, 16-byte chunk c stored
//                at chunk c ^ (r % 8); 8-row groups 1024 B apart (SBO = 1024).
//                The k-th 16-wide K slice starts 32*k bytes into the tile.
//   B  MN-major: TMA box {64 (N), 64 (K)}: K row j at byte j*128 (swizzled), the
//                next 64 columns of N 8192 B further (LBO = 8192), 8-row K groups
//                1024 B apart (SBO = 1024).  The k-th K slice starts 2048*k bytes in.
#include <cudaTypedefs.h>
#include <math.h>

#include "internal.h"

namespace mv {

namespace {

struct Tile {
    int g, row0, nrows, n0;
};

__device__ __forceinline__ Tile decode_tile(const GemmArgs& p, int64_t w) {
    const int mt = (int)(w / p.n_ntiles);
    const int nt = (int)(w - (int64_t)mt * p.n_ntiles);
    int lo = 0, hi = p.G - 1;   // largest g with tile_off[g] <= mt (skips empty groups)
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (__ldg(p.tile_off + mid) <= mt) lo = mid;
        else hi = mid - 1;
    }
    Tile t;
    t.g = lo;
    const int seg0 = __ldg(p.offsets + lo), seg1 = __ldg(p.offsets + lo + 1);
    t.row0 = seg0 + (mt - __ldg(p.tile_off + lo)) * GM_BM;
    t.nrows = min(GM_BM, seg1 - t.row0);
    if ((int64_t)t.row0 + t.nrows > p.m_total) {   // inconsistent offsets: write nothing
        report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_TILES, t.row0, seg1);
        t.nrows = 0;
    }
    t.n0 = nt * p.BN;
    return t;
}

__device__ __forceinline__ float gelu_erf(float u) {
    return 0.5f * u * (1.0f + erff(u * 0.70710678118654752f));
}

struct Smem {
    uint32_t a0, b0;          // shared addresses of stage 0
    uint32_t full, empty;     // barrier arrays (8 bytes apart)
    uint32_t tfull, tempty;
    uint32_t drain;
};

__device__ __forceinline__ void set_abort(volatile int* flag, DevStatus* st, int site, int a,
                                          int b) {
    *flag = 1;
    report(st, MOEVIE_ERR_TIMEOUT, site, a, b);
}

// ------------------------------------------------------------- producers

__device__ void producer_a(const GemmArgs& p, const Smem& sm, int64_t n_work,
                           volatile int* abort_flag) {
    const int pt = threadIdx.x - 6 * 32;   // 0..127
    const int c = pt & 7, rb = pt >> 3;     // 16-byte chunk, first row
    int s = 0;
    uint32_t ph = 0;
    int pend = -1;                          // stage whose arrival waits for its copies
    bool ok = true;
    for (int64_t w = blockIdx.x; w < n_work && ok; w += gridDim.x) {
        const Tile t = decode_tile(p, w);
        const __nv_bfloat16* src[8];
#pragma unroll
        for (int j = 0; j < 8; ++j) {
            const int r = rb + 16 * j;
            if (r < t.nrows) {
                const int gr = t.row0 + r;
                const int ar = p.a_rows ? __ldg(p.a_rows + gr) / p.a_div : gr;
                if (ar >= 0 && ar < p.a_nrows) {
                    src[j] = p.A + (int64_t)ar * p.lda;
                } else {   // out-of-range gather index: zero row, device error
                    report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_A_ROW, gr, ar);
                    src[j] = nullptr;
                }
            } else {
                src[j] = nullptr;
            }
        }
        for (int kb = 0; kb < p.num_kb; ++kb) {
            if (!mbar_wait(sm.empty + 8 * s, ph ^ 1u, p.limit_ns, abort_flag)) {
                set_abort(abort_flag, p.status, SITE_GEMM_WAIT_EMPTY, blockIdx.x, 0);
                ok = false;
                break;
            }
            const uint32_t dst0 = sm.a0 + s * GM_A_BYTES;
            const int col = kb * GM_BK + c * 8;
            const bool col_ok = col < p.K;
#pragma unroll
            for (int j = 0; j < 8; ++j) {
                const int r = rb + 16 * j;
                const uint32_t dst = dst0 + r * 128 + ((c ^ (r & 7)) << 4);
                const bool v = col_ok && src[j] != nullptr;
                cp_async16(dst, v ? (const void*)(src[j] + col) : (const void*)p.A, v ? 16u : 0u);
            }
            cp_async_commit();
            if (pend >= 0) {
                cp_async_wait<1>();
                fence_proxy_async_smem();
                mbar_arrive(sm.full + 8 * pend);
            }
            pend = s;
            if (++s == GM_STAGES) {
                s = 0;
                ph ^= 1u;
            }
        }
    }
    cp_async_wait<0>();
    if (pend >= 0) {
        fence_proxy_async_smem();
        mbar_arrive(sm.full + 8 * pend);
    }
}

__device__ void producer_b(const GemmArgs& p, const Smem& sm, int64_t n_work,
                           volatile int* abort_flag) {
    tma_prefetch_desc(&p.tmB);
    const uint32_t stage_bytes = (uint32_t)p.nbox * GM_BK * 128;
    int s = 0;
    uint32_t ph = 0;
    for (int64_t w = blockIdx.x; w < n_work; w += gridDim.x) {
        const Tile t = decode_tile(p, w);
        for (int kb = 0; kb < p.num_kb; ++kb) {
            if (!mbar_wait(sm.empty + 8 * s, ph ^ 1u, p.limit_ns, abort_flag)) {
                set_abort(abort_flag, p.status, SITE_GEMM_WAIT_EMPTY, blockIdx.x, 1);
                return;
            }
            const uint32_t bar = sm.full + 8 * s;
            mbar_arrive_expect_tx(bar, stage_bytes);
            const uint32_t dst0 = sm.b0 + s * GM_B_BYTES;
            for (int j = 0; j < p.nbox; ++j)
                tma_load_3d(dst0 + j * (GM_BK * 128), &p.tmB, bar, t.n0 + 64 * j, kb * GM_BK, t.g);
            if (++s == GM_STAGES) {
                s = 0;
                ph ^= 1u;
            }
        }
    }
}

// ------------------------------------------------------------------- MMA

__device__ void mma_issuer(const GemmArgs& p, const Smem& sm, uint32_t tmem, int64_t n_work,
                           volatile int* abort_flag) {
    const uint32_t idesc = idesc_bf16_f32(GM_BM, p.BN, false, true);
    int s = 0;
    uint32_t ph = 0;
    int it = 0;
    bool issued = false;
    for (int64_t w = blockIdx.x; w < n_work; w += gridDim.x, ++it) {
        const int acc = it & 1;
        const uint32_t aph = (uint32_t)(it >> 1) & 1u;
        if (!mbar_wait(sm.tempty + 8 * acc, aph ^ 1u, p.limit_ns, abort_flag)) {
            set_abort(abort_flag, p.status, SITE_GEMM_WAIT_TEMPTY, blockIdx.x, it);
            break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + (uint32_t)acc * GM_MAXBN;
        bool ok = true;
        for (int kb = 0; kb < p.num_kb; ++kb) {
            if (!mbar_wait(sm.full + 8 * s, ph, p.limit_ns, abort_flag)) {
                set_abort(abort_flag, p.status, SITE_GEMM_WAIT_FULL, blockIdx.x, kb);
                ok = false;
                break;
            }
            tc_fence_after();
            const uint32_t a_addr = sm.a0 + s * GM_A_BYTES;
            const uint32_t b_addr = sm.b0 + s * GM_B_BYTES;
#pragma unroll
            for (int kk = 0; kk < GM_BK / 16; ++kk) {
                const uint64_t ad = smem_desc_sw128(a_addr + kk * 32, 16, 1024);
                const uint64_t bd = smem_desc_sw128(b_addr + kk * 2048, 8192, 1024);
                tc_mma_bf16(d_tmem, ad, bd, idesc, (kb | kk) != 0 ? 1u : 0u);
            }
            issued = true;
            tc_commit(sm.empty + 8 * s);
            if (++s == GM_STAGES) {
                s = 0;
                ph ^= 1u;
            }
        }
        if (!ok) break;
        tc_commit(sm.tfull + 8 * acc);
    }
    // Every tcgen05.mma must be complete before TMEM is released.
    if (issued) {
        tc_commit(sm.drain);
        if (!mbar_wait(sm.drain, 0, p.limit_ns, nullptr))
            report(p.status, MOEVIE_ERR_TIMEOUT, SITE_GEMM_DRAIN, blockIdx.x, 0);
    }
}

// -------------------------------------------------------------- epilogue

__device__ void epilogue(const GemmArgs& p, const Smem& sm, uint32_t tmem, int64_t n_work,
                         volatile int* abort_flag) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int row = warp * 32 + lane;
    int it = 0;
    for (int64_t w = blockIdx.x; w < n_work; w += gridDim.x, ++it) {
        const Tile t = decode_tile(p, w);
        const int acc = it & 1;
        const uint32_t aph = (uint32_t)(it >> 1) & 1u;
        if (!mbar_wait(sm.tfull + 8 * acc, aph, p.limit_ns, abort_flag)) {
            set_abort(abort_flag, p.status, SITE_GEMM_WAIT_TFULL, blockIdx.x, it);
            return;
        }
        tc_fence_after();
        const bool rv = row < t.nrows;
        const int gr = t.row0 + row;
        int64_t tok = gr;
        float sc = p.scale;
        bool rv_out = rv;
        if (rv) {
            if (p.o_rows) tok = __ldg(p.o_rows + gr) / p.o_div;
            if (p.row_scale) sc = __ldg(p.row_scale + gr);
            if ((p.epi == EPI_ADD_F32 || p.epi == EPI_STORE_F32) && (tok < 0 || tok >= p.o_nrows)) {
                report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_OUT_ROW, gr, (int)tok);
                rv_out = false;
            }
        }
        const uint32_t tbase = tmem + ((uint32_t)(warp * 32) << 16) + (uint32_t)acc * GM_MAXBN;
        for (int c0 = 0; c0 < p.BN; c0 += 32) {
            uint32_t v[32];
            tmem_ld_32x32b_x32(tbase + c0, v);
            tmem_wait_ld();
            if (!rv_out) continue;
#pragma unroll
            for (int g8 = 0; g8 < 4; ++g8) {
                const int cl = c0 + 8 * g8;      // column inside the tile
                const int n = t.n0 + cl;         // column of the output
                if (cl >= p.BN || n >= p.N) continue;
                float f[8];
#pragma unroll
                for (int i = 0; i < 8; ++i) f[i] = __uint_as_float(v[8 * g8 + i]);
                if (p.epi == EPI_GELU_BF16 || p.epi == EPI_STORE_BF16) {
                    if (p.epi == EPI_GELU_BF16) {
#pragma unroll
                        for (int i = 0; i < 8; ++i) f[i] = gelu_erf(f[i]);
                    }
                    uint4 u;
                    u.x = pack_bf16x2(f[0], f[1]);
                    u.y = pack_bf16x2(f[2], f[3]);
                    u.z = pack_bf16x2(f[4], f[5]);
                    u.w = pack_bf16x2(f[6], f[7]);
                    *reinterpret_cast<uint4*>(p.out + (int64_t)gr * p.ldo + n) = u;
                } else {
                    float4* dst = reinterpret_cast<float4*>(p.yacc + tok * p.ldy + n);
                    const float4 lo = make_float4(sc * f[0], sc * f[1], sc * f[2], sc * f[3]);
                    const float4 hi = make_float4(sc * f[4], sc * f[5], sc * f[6], sc * f[7]);
                    if (p.epi == EPI_ADD_F32) {
                        atomicAdd(dst, lo);
                        atomicAdd(dst + 1, hi);
                    } else {
                        dst[0] = lo;
                        dst[1] = hi;
                    }
                }
            }
        }
        tc_fence_before();
        mbar_arrive(sm.tempty + 8 * acc);
    }
}

__global__ void __launch_bounds__(GM_THREADS, 1) grouped_gemm_kernel(const __grid_constant__ GemmArgs p) {
    extern __shared__ uint8_t gm_smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(gm_smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* sA = smem;
    uint8_t* sB = smem + GM_STAGES * GM_A_BYTES;
    uint64_t* bars = reinterpret_cast<uint64_t*>(sB + GM_STAGES * GM_B_BYTES);
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 2 * GM_STAGES + 5);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);

    Smem sm;
    sm.a0 = smem_u32(sA);
    sm.b0 = smem_u32(sB);
    sm.full = smem_u32(bars);
    sm.empty = sm.full + 8 * GM_STAGES;
    sm.tfull = sm.empty + 8 * GM_STAGES;
    sm.tempty = sm.tfull + 16;
    sm.drain = sm.tempty + 16;

    const int warp = threadIdx.x >> 5;
    if (threadIdx.x == 0) {
        for (int s = 0; s < GM_STAGES; ++s) {
            mbar_init(sm.full + 8 * s, 128 + 1);   // 128 gather threads + 1 TMA arrival
            mbar_init(sm.empty + 8 * s, 1);        // tcgen05.commit
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(sm.tfull + 8 * a, 1);        // tcgen05.commit
            mbar_init(sm.tempty + 8 * a, 128);     // every epilogue thread
        }
        mbar_init(sm.drain, 1);
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == 4) {
        tmem_alloc(smem_u32(tmem_slot), 2 * GM_MAXBN);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    int64_t n_mtiles = __ldg(p.tile_off + p.G);
    if (n_mtiles < 0 || n_mtiles > p.max_mtiles) {   // inconsistent offsets: do no work
        if (threadIdx.x == 0) report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_TILES, (int)n_mtiles, -1);
        n_mtiles = 0;
    }
    const int64_t n_work = n_mtiles * p.n_ntiles;

    if (warp < 4) {
        epilogue(p, sm, tmem, n_work, abort_flag);
    } else if (warp == 4) {
        if ((threadIdx.x & 31) == 0) mma_issuer(p, sm, tmem, n_work, abort_flag);
    } else if (warp == 5) {
        if ((threadIdx.x & 31) == 0) producer_b(p, sm, n_work, abort_flag);
    } else {
        producer_a(p, sm, n_work, abort_flag);
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 4) {
        tc_fence_after();
        tmem_dealloc(tmem, 2 * GM_MAXBN);
    }
}

PFN_cuTensorMapEncodeTiled_v12000 get_encode_fn() {
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void* ptr = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &ptr, 12000,
                                             cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(ptr);
    }
    return fn;
}

}  // namespace

bool make_weight_tmap(CUtensorMap* tm, const void* base, int64_t N, int64_t K, int64_t G) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)N, (cuuint64_t)K, (cuuint64_t)G};
    cuuint64_t strides[2] = {(cuuint64_t)N * 2, (cuuint64_t)N * K * 2};
    cuuint32_t box[3] = {64, GM_BK, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                     strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

void choose_bn(int N, int* BN, int* n_ntiles) {
    const int nt = (N + GM_MAXBN - 1) / GM_MAXBN;
    int bn = (N + nt - 1) / nt;
    bn = (bn + 15) / 16 * 16;
    *BN = bn;
    *n_ntiles = (N + bn - 1) / bn;
}

cudaError_t launch_grouped_gemm(const GemmArgs& a, int grid, cudaStream_t s) {
    static bool attr_set[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        cudaError_t e = cudaFuncSetAttribute(grouped_gemm_kernel,
                                             cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             GM_SMEM_BYTES);
        if (e != cudaSuccess) return e;
        attr_set[dev] = true;
    }
    grouped_gemm_kernel<<<grid, GM_THREADS, GM_SMEM_BYTES, s>>>(a);
    count_launches(1);
    return cudaGetLastError();
}

}  // namespace mv
