// gemm.cu -- persistent grouped GEMM on tcgen05 / TMEM with 2-SM MMAs, for the
// MoE-ViE layer (App. B, Algorithm 1, Kernels 1 and 2; also the router logits),
// sm_103a.
//
// One launch computes, for every group g (an expert) and every row r of its
// segment:   D[r, :] = A[row(r), :] . B[g]   (bf16 inputs, fp32 accumulation)
// and hands each tile to a fused epilogue:
//   EPI_GELU_BF16   hidden = bf16(GELU(D))                      (Kernel 1, GELU)
//   EPI_STORE_BF16  out    = bf16(D)
//   EPI_ADD_F32     y[tok(r)] += gate(r) * D   (Kernel 2: routing weight + scatter-add)
//   EPI_STORE_F32   y[tok(r)]  = scale * D     (first writer of y; router logits)
//
// CTA pairs.  The grid is made of clusters of two CTAs on neighbouring SMs.  A
// pair computes a 256 x BN tile with tcgen05.mma.cta_group::2 (M = 256): CTA r
// holds rows 128 r .. 128 r + 127 of A and columns r BN/2 .. (r+1) BN/2 - 1 of B
// in its shared memory, and receives rows 128 r .. of D in its TMEM.  Per SM this
// halves the B traffic of a 128 x BN tile, so shared memory bandwidth (the MMA
// reads what TMA writes) no longer caps the tensor pipe.  CTA 0 of the pair (the
// leader) issues every MMA; its commits arrive on the barriers of both CTAs.
//
// Work items are (256-row m-tile, n-tile) pairs in group-major order with the
// n-tile fastest; a persistent pair walks them with a static stride.  The m-tiles
// come from a device tile table {group, first row, rows <= 256} written by the
// permute step (no host read of segment sizes), or, for one dense group, from
// arithmetic.
//
// Warp roles (608 threads per CTA, one CTA per SM):
//   warps 0-7   epilogue: tcgen05.ld of the CTA's 128 accumulator rows (warp w:
//               TMEM lanes 32 (w%4)..+31, every other 32-column chunk), fused math,
//               and 16-byte stores / reductions of each thread's own row
//   warp 8      TMEM allocation (both CTAs, jointly); leader lane 0 issues the MMAs
//   warp 9      lane 0: TMA loads of the B half and, for contiguous A rows, of A;
//               the leader posts the byte count of both CTAs on its full barrier
//   warps 10-17 token gather: 16-byte cp.async of A rows straight into the 128-byte
//               swizzled K-major layout; each thread hands the completion of its
//               copies to the stage's local afull barrier and moves on
//   warp 18     lane 0: waits for afull, fences the stage to the async proxy and
//               publishes it on the leader's full barrier (from the peer: a 16-byte
//               bulk copy that completes transaction bytes there)
// Shared memory: 7 stages (6 plus a reduction staging buffer for the y-accumulator
// epilogue) x (A 128x64 + B 64x128) bf16; TMEM: two fp32 accumulators
// of 256 columns, so the epilogue of one tile overlaps the main loop of the next.
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


// ------------------------------------------------------------ pair helpers

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}
// Address of the same shared-memory object in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t peer_addr(uint32_t addr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}
__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::
                     : "memory");
}
// 16-byte async-proxy copy from this CTA's shared memory to `dst_cluster` (shared
// memory of a CTA of the cluster) that completes 16 transaction bytes on the
// barrier `bar_cluster` of that CTA.
__device__ __forceinline__ void bulk_signal_remote(uint32_t dst_cluster, uint32_t src,
                                                   uint32_t bar_cluster) {
    asm volatile(
        "cp.async.bulk.shared::cluster.shared::cta.mbarrier::complete_tx::bytes [%0], [%1], 16, [%2];" ::
            "r"(dst_cluster), "r"(src), "r"(bar_cluster)
        : "memory");
}
// Arrival on a barrier of another CTA of the cluster, with the default (CTA-scope)
// release: used where the arriving thread has nothing to publish but completed
// tcgen05.ld reads (ordered by tcgen05 fences around the barrier), so no
// cluster-wide release of its earlier stores is needed.
__device__ __forceinline__ void mbar_arrive_remote(uint32_t bar_cluster) {
    asm volatile("mbarrier.arrive.shared::cluster.b64 _, [%0];" ::"r"(bar_cluster) : "memory");
}
// TMA loads into this CTA's shared memory that complete on a barrier of either CTA
// of the pair.
__device__ __forceinline__ void tma_load_3d_pair(uint32_t dst, const CUtensorMap* tm,
                                                 uint32_t bar_cluster, int c0, int c1, int c2) {
    asm volatile(
        "cp.async.bulk.tensor.3d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3, %4}], [%5];" ::"r"(dst),
        "l"(tm), "r"(c0), "r"(c1), "r"(c2), "r"(bar_cluster)
        : "memory");
}
__device__ __forceinline__ void tma_load_2d_pair(uint32_t dst, const CUtensorMap* tm,
                                                 uint32_t bar_cluster, int c0, int c1) {
    asm volatile(
        "cp.async.bulk.tensor.2d.cta_group::2.shared::cluster.global.tile.mbarrier::complete_tx::bytes"
        " [%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
        "l"(tm), "r"(c0), "r"(c1), "r"(bar_cluster)
        : "memory");
}
__device__ __forceinline__ void tmem_alloc_pair(uint32_t slot, uint32_t ncols) {
    asm volatile("tcgen05.alloc.cta_group::2.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot),
                 "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish_pair() {
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::2.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc_pair(uint32_t taddr, uint32_t ncols) {
    asm volatile("tcgen05.dealloc.cta_group::2.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tc_mma_bf16_pair(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                                 uint32_t idesc, uint32_t accumulate) {
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::2.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// Arrive once on the barrier at shared offset `bar` of both CTAs when all prior
// tcgen05 operations of this thread have completed.
__device__ __forceinline__ void tc_commit_pair(uint32_t bar) {
    asm volatile(
        "tcgen05.commit.cta_group::2.mbarrier::arrive::one.shared::cluster.multicast::cluster.b64"
        " [%0], %1;" ::"r"(bar),
        "h"((uint16_t)3)
        : "memory");
}

// ------------------------------------------------------------------ tiles

struct Tile {
    int g, row0, nrows, n0;
    int kb0, kb1;   // k-blocks [kb0, kb1) of this item's split of K
    int ks;         // split index
    int m0;         // weight-gradient items: first row of the output tile within its group
    int store;      // weight-gradient items: the only item of its output tile (store, not add)
};

// A work item's table entry, loaded but not yet checked.  The roles that walk the
// items load the entry of an item one item ahead (tile_load) and check it when the
// item starts (tile_finish), so that no role waits on that load at an item boundary.
struct TileLd {
    int4 d;   // table entry (unused for one dense group)
    int ks;   // split of K
    int q;    // item index without the split: table entry (item table) or m-tile x n-tile
};

// Work-item counts stay far below 2^31 (m-tiles x n-tiles x K splits), so item indices
// are split with 32-bit arithmetic, each division done once.
__device__ __forceinline__ TileLd tile_load(const GemmArgs& p, int64_t w64) {
    TileLd l;
    const int w = (int)w64;
    l.q = w / p.ksplit;   // split of K fastest
    l.ks = w - l.q * p.ksplit;
    if (p.item_table) l.d = __ldg(p.tiles + l.q);
    else if (p.tiles) l.d = __ldg(p.tiles + l.q / p.n_ntiles);
    else l.d = make_int4(0, 0, 0, 0);
    return l;
}

// k-blocks [kb0, kb1) of split ks of K.
__device__ __forceinline__ void tile_kb(const GemmArgs& p, int ks, int& kb0, int& kb1) {
    kb0 = (int)((int64_t)ks * p.num_kb / p.ksplit);
    kb1 = (int)((int64_t)(ks + 1) * p.num_kb / p.ksplit);
}

__device__ __forceinline__ Tile tile_finish(const GemmArgs& p, const TileLd& l) {
    Tile t;
    t.ks = l.ks;
    t.m0 = 0;
    t.store = 0;
    if (p.item_table == 2) {   // a weight-gradient item {g, m0 | n0 << 16, kb0, kb1 (| store bit)}
        t.g = l.d.x;
        t.m0 = l.d.y & 0xffff;
        t.n0 = (int)((uint32_t)l.d.y >> 16);
        t.kb0 = l.d.z;
        t.kb1 = l.d.w & (BWD_STORE_BIT - 1);
        t.store = (l.d.w & BWD_STORE_BIT) ? 1 : 0;
        t.row0 = t.g * p.wg_M + t.m0;
        t.nrows = min(GM_BM, p.wg_M - t.m0);
        if (t.g < 0 || t.g >= p.G || t.m0 >= p.wg_M || t.n0 >= p.N || t.kb0 < 0 || t.kb1 <= t.kb0 ||
            (int64_t)t.row0 + t.nrows > p.m_total) {
            report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_TILES, t.g, t.kb0);
            t.nrows = 0;
            t.g = 0;
            t.n0 = 0;
            t.kb1 = t.kb0 = 0;
        }
        return t;
    }
    tile_kb(p, l.ks, t.kb0, t.kb1);
    if (p.item_table) {   // an explicit (m-tile, n-tile) item
        t.g = l.d.x;
        t.row0 = l.d.y;
        t.nrows = l.d.z;
        t.n0 = l.d.w;
        if (t.nrows < 0 || t.nrows > GM_BM || t.g < 0 || t.g >= p.G || t.n0 < 0 || t.n0 >= p.N ||
            (int64_t)t.row0 + t.nrows > p.m_total) {
            report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_TILES, t.row0, t.nrows);
            t.nrows = 0;
            t.g = 0;
            t.n0 = 0;
        }
        return t;
    }
    const int mt = l.q / p.n_ntiles;
    const int nt = l.q - mt * p.n_ntiles;
    if (p.tiles) {
        t.g = l.d.x;
        t.row0 = l.d.y;
        t.nrows = l.d.z;
    } else {   // one dense group of m_total rows
        t.g = 0;
        t.row0 = mt * GM_BM;
        const int64_t left = p.m_total - t.row0;
        t.nrows = (int)(left < GM_BM ? left : GM_BM);
    }
    if (t.nrows < 0 || t.nrows > GM_BM || t.g < 0 || t.g >= p.G ||
        (int64_t)t.row0 + t.nrows > p.m_total) {
        report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_TILES, t.row0, t.nrows);
        t.nrows = 0;
        t.g = 0;
    }
    t.n0 = nt * p.n_step;
    return t;
}

__device__ __forceinline__ Tile decode_tile(const GemmArgs& p, int64_t w) {
    return tile_finish(p, tile_load(p, w));
}

// GELU(u) = u/2 (1 + erf(u / sqrt 2)) = max(u, 0) - |u|/2 erfc(|u| / sqrt 2), the
// second form free of the cancellation of 1 + erf for u < 0.  erfc from Abramowitz &
// Stegun 7.1.28: erfc(z) = (1 + a1 z + a2 z^2 + ... + a6 z^6)^-16 for z >= 0, with
// |error| <= 3e-7 (one reciprocal and no exponential; the sixteenth power by four
// squarings, which overflow to +inf, and so to erfc = 0, only where erfc is far
// below fp32 resolution).  Evaluated in fp32 the GELU error stays below 1e-6 in
// absolute value; the hidden activation is then rounded to bf16 (2^-9 relative).
// Two values at a time with the packed fp32x2 instructions.
__device__ __forceinline__ void erfc_as2(float a0, float a1, float& q0, float& q1) {   // a0, a1 >= 0
    const uint64_t z = f2_mul(f2_pack(a0, a1), f2_pack(0.70710678118654752f, 0.70710678118654752f));
    uint64_t P = f2_fma(z, f2_pack(0.0000430638f, 0.0000430638f), f2_pack(0.0002765672f, 0.0002765672f));
    P = f2_fma(P, z, f2_pack(0.0001520143f, 0.0001520143f));
    P = f2_fma(P, z, f2_pack(0.0092705272f, 0.0092705272f));
    P = f2_fma(P, z, f2_pack(0.0422820123f, 0.0422820123f));
    P = f2_fma(P, z, f2_pack(0.0705230784f, 0.0705230784f));
    P = f2_fma(P, z, f2_pack(1.0f, 1.0f));
    P = f2_mul(P, P);
    P = f2_mul(P, P);
    P = f2_mul(P, P);
    P = f2_mul(P, P);
    float p0, p1;
    f2_unpack(P, p0, p1);
    q0 = rcp_approx(p0);
    q1 = rcp_approx(p1);
}

__device__ __forceinline__ void gelu_erf2(float& u0, float& u1) {
    float q0, q1;
    erfc_as2(fabsf(u0), fabsf(u1), q0, q1);
    const uint64_t r = f2_fma(f2_mul(f2_pack(fabsf(u0), fabsf(u1)), f2_pack(-0.5f, -0.5f)), f2_pack(q0, q1),
                              f2_pack(fmaxf(u0, 0.0f), fmaxf(u1, 0.0f)));
    f2_unpack(r, u0, u1);
}

// GELU'(u) = Phi(u) + u phi(u) (the derivative of the erf form) of two values, for the
// training path: Phi(u) = erfc(-u / sqrt 2) / 2 from the erfc above (1 - q / 2 for
// u >= 0, q / 2 below), phi(u) = exp(-u^2 / 2) / sqrt(2 pi) with CUDA's __expf.
// Absolute error below 1e-6.
__device__ __forceinline__ void gelu_grad2(float& u0, float& u1) {
    float q0, q1;
    erfc_as2(fabsf(u0), fabsf(u1), q0, q1);
    const float c0 = u0 >= 0.0f ? 1.0f - 0.5f * q0 : 0.5f * q0;
    const float c1 = u1 >= 0.0f ? 1.0f - 0.5f * q1 : 0.5f * q1;
    u0 = fmaf(u0, 0.3989422804014327f * __expf(-0.5f * u0 * u0), c0);
    u1 = fmaf(u1, 0.3989422804014327f * __expf(-0.5f * u1 * u1), c1);
}

struct Smem {
    uint32_t a0, b0;          // shared addresses of stage 0
    uint32_t full, empty;     // barrier arrays (8 bytes apart)
    uint32_t afull;           // peer CTA: its gather warps' copies of a stage have landed
    uint32_t tfull, tempty;
    uint32_t drain;
    uint32_t sink;            // 16 bytes: target / source of the peer's stage signals
    int nstages;              // operand ring depth of this launch
    float* stg;               // reduction staging: STG_ROWS rows of GM_STG_LD floats per warp
    uint32_t rank;            // rank of this CTA in its pair
    int64_t pair, npairs;     // pair index and count
};

__device__ __forceinline__ void set_abort(volatile int* flag, DevStatus* st, int site, int a,
                                          int b) {
    *flag = 1;
    report(st, MOEVIE_ERR_TIMEOUT, site, a, b);
}

// Rows of tile t held by this CTA: 128 rank .. 128 rank + rows_half(t) - 1.
__device__ __forceinline__ int rows_half(const Tile& t, uint32_t rank) {
    const int r = t.nrows - (int)rank * GM_HALF;
    return r < 0 ? 0 : (r > GM_HALF ? GM_HALF : r);
}

// --------------------------------------------------------------- producers

// TMA producer (warp 9, lane 0): the CTA's half of B, and A when its rows are
// contiguous.  The leader posts the byte count of both CTAs on its full barrier.
template <bool GATHER, bool TRAIN>
__device__ void producer_tma(const GemmArgs& p, const Smem& sm, int64_t n_work,
                             volatile int* abort_flag) {
    tma_prefetch_desc(&p.tmB);
    if (p.g_split < p.G || p.swiglu) tma_prefetch_desc(&p.tmB2);
    if (p.g_split < p.G && p.swiglu) {
        tma_prefetch_desc(&p.tmB3);
        tma_prefetch_desc(&p.tmB4);
    }
    constexpr bool gather = GATHER;
    if (!gather) tma_prefetch_desc(&p.tmA);
    const uint32_t half_n = (uint32_t)p.BN / 2;
    const uint32_t nboxh = (half_n + 63) / 64;
    // B per CTA and stage: nboxh boxes of 64 columns x 64 K rows (N-major), or half_n rows
    // of 64 K values (K-major)
    const uint32_t b_bytes = (TRAIN && p.b_kmajor) ? half_n * 128u : nboxh * GM_BK * 128;
    const uint32_t cta_bytes = b_bytes + (gather ? 0u : (uint32_t)GM_A_BYTES);
    // gathering: plus the 16-byte signal with which the peer publishes its A half
    const uint32_t stage_tx = 2 * cta_bytes + (gather ? 16u : 0u);
    const uint32_t full_leader = peer_addr(sm.full, 0);
    int s = 0;
    uint32_t ph = 0;
    int64_t w = sm.pair;
    Tile t{};
    if (w < n_work) t = decode_tile(p, w);
    for (; w < n_work; w += sm.npairs) {
        const int64_t wn = w + sm.npairs;
        TileLd nl{};
        if (wn < n_work) nl = tile_load(p, wn);   // checked after this item's loads
        // B of this group: groups >= g_split from their own map; with swiglu the second
        // CTA of the pair loads the up projection (W3) beside the gate's (W1) columns
        const bool tail = t.g >= p.g_split;
        const CUtensorMap* tmb = tail ? &p.tmB2 : &p.tmB;
        if (p.swiglu)
            tmb = sm.rank == 1 ? (tail ? &p.tmB4 : &p.tmB2) : (tail ? &p.tmB3 : &p.tmB);
        const int gb = (TRAIN && p.item_table == 2) ? 0 : (tail ? t.g - p.g_split : t.g);
        const int ncol0 = p.swiglu ? t.n0 : t.n0 + (int)(sm.rank * half_n);
        for (int kb = t.kb0; kb < t.kb1; ++kb) {
            if (!mbar_wait(sm.empty + 8 * s, ph ^ 1u, p.limit_ns, abort_flag)) {
                set_abort(abort_flag, p.status, SITE_GEMM_WAIT_EMPTY, (int)sm.pair, 1);
                return;
            }
            const uint32_t bar = full_leader + 8 * s;
            if (sm.rank == 0) mbar_arrive_expect_tx(sm.full + 8 * s, stage_tx);
            const uint32_t b_dst = sm.b0 + s * GM_B_BYTES;
            const int kk = kb * GM_BK;
            if (TRAIN && p.b_kmajor) {   // half_n rows of the CTA's columns, 64 K values each
                tma_load_3d_pair(b_dst, tmb, bar, kk, ncol0, gb);
            } else {
                for (uint32_t j = 0; j < nboxh; ++j)
                    tma_load_3d_pair(b_dst + j * (GM_BK * 128), tmb, bar, ncol0 + (int)(64 * j), kk, gb);
            }
            if (!gather) {
                if (TRAIN && p.a_mn) {   // two 64-row halves of the CTA's 128 output rows, 64 K rows each
                    const int m = t.m0 + (int)sm.rank * GM_HALF;
                    tma_load_3d_pair(sm.a0 + s * GM_A_BYTES, &p.tmA, bar, m, kk, 0);
                    tma_load_3d_pair(sm.a0 + s * GM_A_BYTES + GM_BK * 128, &p.tmA, bar, m + 64, kk, 0);
                } else {
                    const int col = p.a_kperiod ? kk % p.a_kperiod : kk;
                    tma_load_2d_pair(sm.a0 + s * GM_A_BYTES, &p.tmA, bar, col,
                                     t.row0 + (int)sm.rank * GM_HALF);
                }
            }
            if (++s == sm.nstages) {
                s = 0;
                ph ^= 1u;
            }
        }
        if (wn < n_work) t = tile_finish(p, nl);
    }
}

// Table rows of this thread's GM_GATHER_ROWS rows of tile t (r = rb + GM_GATHER_RSTEP j of
// the CTA's half; -1 past the tile), loaded one item ahead of their use.
__device__ __forceinline__ void gather_rows_load(const GemmArgs& p, const Tile& t, uint32_t rank,
                                                 int rb, int (&raw)[GM_GATHER_ROWS]) {
    const int nh = rows_half(t, rank);
#pragma unroll
    for (int j = 0; j < GM_GATHER_ROWS; ++j) {
        const int r = rb + GM_GATHER_RSTEP * j;
        const int gr = t.row0 + (int)rank * GM_HALF + r;
        raw[j] = (r < nh) ? (p.a_ident ? gr : __ldg(p.a_rows + gr)) : -1;
    }
}

// A row pointers from the loaded table rows (nullptr past the tile; an A row outside
// [0, a_nrows) is a device error and is not read).
__device__ __forceinline__ void gather_rows_finish(const GemmArgs& p, const Tile& t, uint32_t rank,
                                                   int rb, const int (&raw)[GM_GATHER_ROWS],
                                                   const __nv_bfloat16* (&src)[GM_GATHER_ROWS]) {
    const int nh = rows_half(t, rank);
#pragma unroll
    for (int j = 0; j < GM_GATHER_ROWS; ++j) {
        const int r = rb + GM_GATHER_RSTEP * j;
        const int idx = r < nh ? raw[j] / p.a_div : -1;
        if (r < nh && idx >= 0 && idx < p.a_nrows) {
            src[j] = p.A + (int64_t)idx * p.lda;
        } else {
            if (r < nh && !(p.a_neg_zero && raw[j] < 0))   // padding rows read as zeros
                report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_A_ROW, t.row0 + (int)rank * GM_HALF + r,
                       idx);
            src[j] = nullptr;
        }
    }
}

// Token gather (GM_GATHER_WARPS warps): each thread copies one 16-byte chunk of
// GM_GATHER_ROWS rows per stage straight into the 128-byte swizzled K-major layout,
// then hands the completion of its copies to the stage's afull barrier
// (cp.async.mbarrier.arrive.noinc) and moves on without waiting; gather_forwarder
// publishes the stage once every gather thread's copies have landed.
__device__ void producer_gather(const GemmArgs& p, const Smem& sm, int64_t n_work,
                                volatile int* abort_flag) {
    const int pt = threadIdx.x - GM_WARP_GATHER * 32;   // 0 .. GM_GATHER_WARPS * 32 - 1
    const int lane = threadIdx.x & 31;
    const int c = pt & 7, rb = pt >> 3;                  // 16-byte chunk, first row
    // gathered rows are re-read by every expert of their tokens: keep them in L2
    const uint64_t keep_pol = l2_policy_evict_last();
    int s = 0;
    uint32_t ph = 0;
    bool ok = true;
    int64_t w = sm.pair;
    // The per-item set-up is pipelined so that no load is waited on at an item start:
    // item w's row pointers are ready when it starts; the next item's table rows were
    // loaded one item earlier, after its tile entry (loaded earlier still) was checked.
    const __nv_bfloat16* src[GM_GATHER_ROWS];
    int nraw[GM_GATHER_ROWS];
    Tile t{}, tn{};
    TileLd nnl{};
    if (w < n_work) {
        t = decode_tile(p, w);
        int raw[GM_GATHER_ROWS];
        gather_rows_load(p, t, sm.rank, rb, raw);
        gather_rows_finish(p, t, sm.rank, rb, raw, src);
    }
    if (w + sm.npairs < n_work) {
        tn = decode_tile(p, w + sm.npairs);
        gather_rows_load(p, tn, sm.rank, rb, nraw);
    }
    if (w + 2 * sm.npairs < n_work) nnl = tile_load(p, w + 2 * sm.npairs);
    for (; w < n_work && ok; w += sm.npairs) {
        const int64_t wn = w + sm.npairs;
        for (int kb = t.kb0; kb < t.kb1; ++kb) {
            int good = 1;
            if (lane == 0) good = mbar_wait(sm.empty + 8 * s, ph ^ 1u, p.limit_ns, abort_flag);
            good = __shfl_sync(0xffffffffu, good, 0);
            if (!good) {
                if (lane == 0) set_abort(abort_flag, p.status, SITE_GEMM_WAIT_EMPTY, (int)sm.pair, 0);
                ok = false;
                break;
            }
            const uint32_t dst0 = sm.a0 + s * GM_A_BYTES;
            const int kk = kb * GM_BK + c * 8;
            const bool col_ok = kk < p.K;
#pragma unroll
            for (int j = 0; j < GM_GATHER_ROWS; ++j) {
                const int r = rb + GM_GATHER_RSTEP * j;
                const uint32_t dst = dst0 + r * 128 + ((c ^ (r & 7)) << 4);
                const bool v = col_ok && src[j] != nullptr;
                cp_async16_hint(dst, v ? (const void*)(src[j] + kk) : (const void*)p.A, v ? 16u : 0u,
                                keep_pol);
            }
            cp_async_arrive_noinc(sm.afull + 8 * s);
            if (++s == sm.nstages) {
                s = 0;
                ph ^= 1u;
            }
        }
        if (wn < n_work) {   // advance: item wn's pointers, item wn + npairs's table rows
            gather_rows_finish(p, tn, sm.rank, rb, nraw, src);
            t = tn;
            if (wn + sm.npairs < n_work) {
                tn = tile_finish(p, nnl);
                gather_rows_load(p, tn, sm.rank, rb, nraw);
                if (wn + 2 * sm.npairs < n_work) nnl = tile_load(p, wn + 2 * sm.npairs);
            }
        }
    }
    cp_async_wait_all();
}

// Warp GM_WARP_FWD, lane 0, in both CTAs: once all of this CTA's gather threads'
// copies of a stage have landed (its afull barrier), make them visible to the async
// proxy that tcgen05.mma reads shared memory through, and publish the stage on the
// leader's full barrier: a local arrival in the leader; from the peer, a 16-byte
// async-proxy copy into the leader that completes 16 transaction bytes on that
// barrier (the leader's expect_tx counts them).  Being ordered after the proxy
// fence, the copy's completion implies the gathered rows are visible to the MMA,
// without the cost of a cluster-scope release by this thread.
__device__ void gather_forwarder(const GemmArgs& p, const Smem& sm, int64_t n_work,
                                 volatile int* abort_flag) {
    const uint32_t full_leader = peer_addr(sm.full, 0);
    const uint32_t sink_leader = peer_addr(sm.sink, 0);
    int s = 0;
    uint32_t ph = 0;
    for (int64_t w = sm.pair; w < n_work; w += sm.npairs) {
        int kb0, kb1;   // the item's stages; its table entry is not needed here
        tile_kb(p, (int)(w % p.ksplit), kb0, kb1);
        for (int kb = kb0; kb < kb1; ++kb) {
            if (!mbar_wait(sm.afull + 8 * s, ph, p.limit_ns, abort_flag)) {
                set_abort(abort_flag, p.status, SITE_GEMM_WAIT_FULL, (int)sm.pair, -1 - kb);
                return;
            }
            fence_proxy_async_smem();
            if (sm.rank == 0) mbar_arrive(sm.full + 8 * s);
            else bulk_signal_remote(sink_leader, sm.sink, full_leader + 8 * s);
            if (++s == sm.nstages) {
                s = 0;
                ph ^= 1u;
            }
        }
    }
}

// ------------------------------------------------------------------- MMA

// Leader CTA, warp 8, lane 0.
template <bool TRAIN>
__device__ void mma_issuer(const GemmArgs& p, const Smem& sm, uint32_t tmem, int64_t n_work,
                           volatile int* abort_flag) {
    // K-major operands: k-slice +32 B; MN-major operands: next 64-element atom LBO 8192,
    // k-slice +2048 B (16 K rows of 128 bytes).  The forward's A is K-major, its B MN-major.
    const bool a_mn = TRAIN && p.a_mn, b_km = TRAIN && p.b_kmajor;
    const uint32_t idesc = idesc_bf16_f32(2 * GM_HALF, p.BN, a_mn, !b_km);
    const uint64_t adesc0 = a_mn ? smem_desc_sw128(sm.a0, 8192, 1024) : smem_desc_sw128(sm.a0, 16, 1024);
    const uint64_t bdesc0 = b_km ? smem_desc_sw128(sm.b0, 16, 1024) : smem_desc_sw128(sm.b0, 8192, 1024);
    const uint32_t a_step = a_mn ? (2048 >> 4) : (32 >> 4);
    const uint32_t b_step = b_km ? (32 >> 4) : (2048 >> 4);
    static_assert(GM_BK == 64, "four k-slices of 16 per stage");
    int s = 0;
    uint32_t ph = 0;
    int it = 0;
    bool issued = false;
    TileLd nl{};   // next item's table entry, loaded one item ahead, checked when it starts
    if (sm.pair < n_work) nl = tile_load(p, sm.pair);
    for (int64_t w = sm.pair; w < n_work; w += sm.npairs, ++it) {
        const Tile t = tile_finish(p, nl);
        if (w + sm.npairs < n_work) nl = tile_load(p, w + sm.npairs);
        const int acc = it & 1;
        const uint32_t aph = (uint32_t)(it >> 1) & 1u;
        if (!mbar_wait(sm.tempty + 8 * acc, aph ^ 1u, p.limit_ns, abort_flag)) {
            set_abort(abort_flag, p.status, SITE_GEMM_WAIT_TEMPTY, (int)sm.pair, it);
            break;
        }
        tc_fence_after();
        const uint32_t d_tmem = tmem + (uint32_t)acc * GM_MAXBN;
        bool ok = true;
        for (int kb = t.kb0; kb < t.kb1; ++kb) {
            // Operands in shared memory are ordered by the barrier alone (TMA bytes, or
            // gathered rows fenced to the async proxy before they were published); the
            // tcgen05 thread-sync fence is needed only where TMEM changes hands.
            if (!mbar_wait(sm.full + 8 * s, ph, p.limit_ns, abort_flag)) {
                set_abort(abort_flag, p.status, SITE_GEMM_WAIT_FULL, (int)sm.pair, kb);
                ok = false;
                break;
            }
            // Descriptors differ from the stage-0 ones only in the start-address field
            // (bits 0-13, address >> 4; shared addresses stay below 256 KB, no carry).
            const uint64_t ad = adesc0 + (uint64_t)((s * GM_A_BYTES) >> 4);
            const uint64_t bd = bdesc0 + (uint64_t)((s * GM_B_BYTES) >> 4);
            tc_mma_bf16_pair(d_tmem, ad, bd, idesc, kb != t.kb0 ? 1u : 0u);
            tc_mma_bf16_pair(d_tmem, ad + a_step, bd + b_step, idesc, 1u);
            tc_mma_bf16_pair(d_tmem, ad + 2 * a_step, bd + 2 * b_step, idesc, 1u);
            tc_mma_bf16_pair(d_tmem, ad + 3 * a_step, bd + 3 * b_step, idesc, 1u);
            issued = true;
            tc_commit_pair(sm.empty + 8 * s);
            if (++s == sm.nstages) {
                s = 0;
                ph ^= 1u;
            }
        }
        if (!ok) break;
        tc_commit_pair(sm.tfull + 8 * acc);
    }
    // Every tcgen05.mma must be complete before TMEM is released.
    if (issued) {
        tc_commit_pair(sm.drain);
        if (!mbar_wait(sm.drain, 0, p.limit_ns, nullptr))
            report(p.status, MOEVIE_ERR_TIMEOUT, SITE_GEMM_DRAIN, (int)sm.pair, 0);
    }
}

// -------------------------------------------------------------- epilogue

// One 32-column chunk of the y-accumulator reductions of one warp: each lane holds
// its row's 32 values; ROWS rows at a time (all 32, or 16 when the staging buffer is
// halved) go to the warp's staging buffer, scaled and with the row's y offset; then
// every lane reduces 4 columns of one of 4 rows per instruction, so 8 lanes cover a
// row's 128 contiguous bytes (a whole L2 line).
template <int ROWS>
__device__ __forceinline__ void reduce_chunk(const GemmArgs& p, float* stg_all, int warp, int lane,
                                             const uint32_t (&v)[32], float sc, int64_t my_yoff,
                                             int n, bool store) {
    float* stg = stg_all + warp * (ROWS * GM_STG_LD);
    const int col = n + 4 * (lane & 7);
#pragma unroll
    for (int hh = 0; hh < 32 / ROWS; ++hh) {
        if (lane / ROWS == hh) {
            float* row = stg + (lane - hh * ROWS) * GM_STG_LD;
#pragma unroll
            for (int c = 0; c < 8; ++c)
                *reinterpret_cast<float4*>(row + 4 * c) =
                    make_float4(sc * __uint_as_float(v[4 * c]), sc * __uint_as_float(v[4 * c + 1]),
                                sc * __uint_as_float(v[4 * c + 2]), sc * __uint_as_float(v[4 * c + 3]));
            *reinterpret_cast<int64_t*>(row + 32) = my_yoff;
        }
        __syncwarp();
#pragma unroll
        for (int r = 0; r < ROWS / 4; ++r) {
            const float* row = stg + (4 * r + (lane >> 3)) * GM_STG_LD;
            const int64_t yo = *reinterpret_cast<const int64_t*>(row + 32);
            const float4 val = *reinterpret_cast<const float4*>(row + 4 * (lane & 7));
            if (yo >= 0 && col < p.N) {
                float4* dst = reinterpret_cast<float4*>(p.yacc + yo + col);
                if (store) *dst = val;   // the only contribution to these elements
                else atomicAdd(dst, val);
            }
        }
        __syncwarp();
    }
}

// Warp w reads TMEM lanes 32 (w % 4) .. +31 (its rows) and the 32-column chunks
// c = w / 4, w / 4 + 2, ... of each tile.  bf16 outputs and fp32 stores: each thread
// takes its own row (32x32b loads) and writes it straight from registers with
// 16-byte stores.  fp32 reductions (the y accumulator): the rows pass a small
// per-warp staging buffer so that each 16-byte vector reduction instruction of a
// warp covers four rows x 128 contiguous bytes, i.e. whole L2 lines.  When a warp has read
// its last chunk of the accumulator it arrives (once) on the leader's tempty barrier.
template <int STG_ROWS, bool GATHER, int ECLS, bool TRAIN>
__device__ void epilogue(const GemmArgs& p, const Smem& sm, uint32_t tmem, int64_t n_work,
                         volatile int* abort_flag) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int quad = warp & 3, half = warp >> 2;
    constexpr bool to_f32 = ECLS != ECLS_BF16;
    const int nchunk = p.BN / 32;
    // bf16 results are written once and read back later: let them leave L2 first
    const uint64_t stream_pol = l2_policy_evict_first();
    const uint32_t tempty_leader = peer_addr(sm.tempty, 0);
    int it = 0;
    for (int64_t w = sm.pair; w < n_work; w += sm.npairs, ++it) {
        const Tile t = decode_tile(p, w);
        const int acc = it & 1;
        const uint32_t aph = (uint32_t)(it >> 1) & 1u;
        const int myrow = quad * 32 + lane;
        const int gr = t.row0 + (int)sm.rank * GM_HALF + myrow;
        int64_t tok = gr;
        float sc = p.scale;
        bool ok_row = myrow < rows_half(t, sm.rank);
        if (ok_row) {
            if (p.o_rows) tok = __ldg(p.o_rows + gr) / p.o_div;
            if (p.row_scale) sc = __ldg(p.row_scale + gr);
            if (to_f32 && (tok < 0 || tok >= p.o_nrows)) {
                if (!(p.o_neg_skip && tok < 0))   // a padding row writes nothing
                    report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_OUT_ROW, gr, (int)tok);
                ok_row = false;
            }
        }
        if (!mbar_wait(sm.tfull + 8 * acc, aph, p.limit_ns, abort_flag)) {
            set_abort(abort_flag, p.status, SITE_GEMM_WAIT_TFULL, (int)sm.pair, it);
            return;
        }
        tc_fence_after();
        const uint32_t tbase = tmem + ((uint32_t)(quad * 32) << 16) + (uint32_t)acc * GM_MAXBN;
        if (ECLS == ECLS_F32 && p.epi == EPI_SUM2_F32) {
            // two column groups of N / 2 (one n-tile): chunk ch of the output is the sum of
            // accumulator chunks ch and ch + nc2
            const int nc2 = nchunk / 2;
            if (half >= nc2) {
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_remote(tempty_leader + 8 * acc);
            }
            for (int ch = half; ch < nc2; ch += 2) {
                uint32_t v[32];
                float s2[32];
                tmem_ld_32x32b_x32(tbase + ch * 32, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) s2[i] = __uint_as_float(v[i]);
                tmem_ld_32x32b_x32(tbase + (ch + nc2) * 32, v);
                tmem_wait_ld();
                if (ch + 2 >= nc2) {   // this warp's last read of the accumulator
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive_remote(tempty_leader + 8 * acc);
                }
                if (!ok_row) continue;
#pragma unroll
                for (int i = 0; i < 32; ++i) s2[i] += __uint_as_float(v[i]);
                float* yrow = p.yacc + t.ks * p.y_split_stride + tok * p.ldy + ch * 32;
#pragma unroll
                for (int q = 0; q < 8; ++q)
                    *reinterpret_cast<float4*>(yrow + 4 * q) =
                        make_float4(sc * s2[4 * q], sc * s2[4 * q + 1], sc * s2[4 * q + 2], sc * s2[4 * q + 3]);
            }
            continue;
        }
        if (GATHER && ECLS == ECLS_BF16 && p.epi == EPI_SWIGLU_BF16) {   // (gathered A only)
            // output chunk ch (32 columns): gate = accumulator chunk ch, up = chunk ch + nout
            const int nout = nchunk / 2;
            if (half >= nout) {
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_remote(tempty_leader + 8 * acc);
            }
            for (int ch = half; ch < nout; ch += 2) {
                uint32_t v[32];
                float gt[32];
                tmem_ld_32x32b_x32(tbase + ch * 32, v);
                tmem_wait_ld();
#pragma unroll
                for (int i = 0; i < 32; ++i) gt[i] = __uint_as_float(v[i]);
                tmem_ld_32x32b_x32(tbase + (ch + nout) * 32, v);
                tmem_wait_ld();
                if (ch + 2 >= nout) {   // this warp's last read of the accumulator
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive_remote(tempty_leader + 8 * acc);
                }
                if (!ok_row) continue;
                const int n = t.n0 + ch * 32;
                __nv_bfloat16* orow = p.out + (int64_t)gr * p.ldo + n;
#pragma unroll
                for (int g8 = 0; g8 < 4; ++g8) {
                    if (n + 8 * g8 >= p.N) break;
                    float f[8];
                    if (TRAIN && p.out2) {   // the training path keeps u and v as well
                        uint4 uu, vv;
                        uu.x = pack_bf16x2(gt[8 * g8 + 0], gt[8 * g8 + 1]);
                        uu.y = pack_bf16x2(gt[8 * g8 + 2], gt[8 * g8 + 3]);
                        uu.z = pack_bf16x2(gt[8 * g8 + 4], gt[8 * g8 + 5]);
                        uu.w = pack_bf16x2(gt[8 * g8 + 6], gt[8 * g8 + 7]);
                        vv.x = pack_bf16x2(__uint_as_float(v[8 * g8 + 0]), __uint_as_float(v[8 * g8 + 1]));
                        vv.y = pack_bf16x2(__uint_as_float(v[8 * g8 + 2]), __uint_as_float(v[8 * g8 + 3]));
                        vv.z = pack_bf16x2(__uint_as_float(v[8 * g8 + 4]), __uint_as_float(v[8 * g8 + 5]));
                        vv.w = pack_bf16x2(__uint_as_float(v[8 * g8 + 6]), __uint_as_float(v[8 * g8 + 7]));
                        *reinterpret_cast<uint4*>(p.out2 + (int64_t)gr * p.ldo + n + 8 * g8) = uu;
                        *reinterpret_cast<uint4*>(p.out3 + (int64_t)gr * p.ldo + n + 8 * g8) = vv;
                    }
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        // SiLU(g) u = g u / (1 + e^-g); e^-g = inf for g far below 0 gives 0
                        const float g = gt[8 * g8 + i];
                        f[i] = __fdividef(g, 1.0f + __expf(-g)) * __uint_as_float(v[8 * g8 + i]);
                    }
                    uint4 u;
                    u.x = pack_bf16x2(f[0], f[1]);
                    u.y = pack_bf16x2(f[2], f[3]);
                    u.z = pack_bf16x2(f[4], f[5]);
                    u.w = pack_bf16x2(f[6], f[7]);
                    st_global_v4_hint(orow + 8 * g8, u, stream_pol);
                }
            }
            continue;
        }
        if (half >= nchunk) {   // no columns for this warp in this tile
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_remote(tempty_leader + 8 * acc);
        }
        float dg_acc = 0.f;   // EPI_DGELU_BF16: this thread's share of its row's dot
        for (int ch = half; ch < nchunk; ch += 2) {
            const int c0 = ch * 32;
            if constexpr (ECLS == ECLS_ADD) {   // the y-accumulator reductions
                uint32_t v[32];
                tmem_ld_32x32b_x32(tbase + c0, v);
                tmem_wait_ld();
                if (ch + 2 >= nchunk) {   // this warp's last read of the accumulator
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive_remote(tempty_leader + 8 * acc);
                }
                const int n = t.n0 + c0;
                const int64_t my_yoff = ok_row ? t.ks * p.y_split_stride + tok * p.ldy : -1;
                reduce_chunk<STG_ROWS>(p, sm.stg, warp, lane, v, sc, my_yoff, n, TRAIN && t.store);
                continue;
            }
            uint32_t v[32];
            tmem_ld_32x32b_x32(tbase + c0, v);
            tmem_wait_ld();
            if (ch + 2 >= nchunk) {   // this warp's last read of the accumulator
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive_remote(tempty_leader + 8 * acc);
            }
            if (!ok_row) continue;
            const int n = t.n0 + c0;
            if constexpr (!to_f32) {
                __nv_bfloat16* orow = p.out + (int64_t)gr * p.ldo + n;
                if (TRAIN && p.epi == EPI_DSWIGLU_BF16) {   // SwiGLU: du, dv and the dot acc . a
                    const __nv_bfloat16* urow = p.epi_u + (int64_t)gr * p.ldo + n;
                    const __nv_bfloat16* vrow = p.epi_v + (int64_t)gr * p.ldo + n;
                    const __nv_bfloat16* arow = p.epi_a + (int64_t)gr * p.ldo + n;
#pragma unroll
                    for (int g8 = 0; g8 < 4; ++g8) {
                        if (n + 8 * g8 >= p.N) break;
                        float uf[8], vf[8], af[8], fu[8], fv[8];
                        unpack_bf16x8(*reinterpret_cast<const uint4*>(urow + 8 * g8), uf);
                        unpack_bf16x8(*reinterpret_cast<const uint4*>(vrow + 8 * g8), vf);
                        unpack_bf16x8(*reinterpret_cast<const uint4*>(arow + 8 * g8), af);
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const float a = __uint_as_float(v[8 * g8 + i]);
                            const bool in = n + 8 * g8 + i < p.N;   // columns past N: padding
                            dg_acc += in ? a * af[i] : 0.f;
                            const float sg = __fdividef(1.0f, 1.0f + __expf(-uf[i]));   // SiLU(u) = u sg
                            fu[i] = in ? sc * a * vf[i] * sg * (1.0f + uf[i] * (1.0f - sg)) : 0.f;
                            fv[i] = in ? sc * a * uf[i] * sg : 0.f;
                        }
                        uint4 u, w;
                        u.x = pack_bf16x2(fu[0], fu[1]);
                        u.y = pack_bf16x2(fu[2], fu[3]);
                        u.z = pack_bf16x2(fu[4], fu[5]);
                        u.w = pack_bf16x2(fu[6], fu[7]);
                        w.x = pack_bf16x2(fv[0], fv[1]);
                        w.y = pack_bf16x2(fv[2], fv[3]);
                        w.z = pack_bf16x2(fv[4], fv[5]);
                        w.w = pack_bf16x2(fv[6], fv[7]);
                        *reinterpret_cast<uint4*>(orow + 8 * g8) = u;
                        *reinterpret_cast<uint4*>(p.out2 + (int64_t)gr * p.ldo + n + 8 * g8) = w;
                    }
                    continue;
                }
                if (TRAIN && p.epi == EPI_DGELU_BF16) {   // training path: du = scale acc GELU'(u), dot acc . a
                    const __nv_bfloat16* urow = p.epi_u + (int64_t)gr * p.ldo + n;
                    const __nv_bfloat16* arow = p.epi_a + (int64_t)gr * p.ldo + n;
#pragma unroll
                    for (int g8 = 0; g8 < 4; ++g8) {
                        if (n + 8 * g8 >= p.N) break;
                        float uf[8], af[8], f[8];
                        unpack_bf16x8(*reinterpret_cast<const uint4*>(urow + 8 * g8), uf);
                        unpack_bf16x8(*reinterpret_cast<const uint4*>(arow + 8 * g8), af);
#pragma unroll
                        for (int i = 0; i < 8; i += 2) gelu_grad2(uf[i], uf[i + 1]);   // GELU'(u)
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const float a = __uint_as_float(v[8 * g8 + i]);
                            const bool in = n + 8 * g8 + i < p.N;   // columns past N: padding
                            dg_acc += in ? a * af[i] : 0.f;
                            f[i] = in ? sc * a * uf[i] : 0.f;
                        }
                        uint4 u;
                        u.x = pack_bf16x2(f[0], f[1]);
                        u.y = pack_bf16x2(f[2], f[3]);
                        u.z = pack_bf16x2(f[4], f[5]);
                        u.w = pack_bf16x2(f[6], f[7]);
                        *reinterpret_cast<uint4*>(orow + 8 * g8) = u;
                    }
                    continue;
                }
#pragma unroll
                for (int g8 = 0; g8 < 4; ++g8) {
                    if (n + 8 * g8 >= p.N) break;
                    float f[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) f[i] = __uint_as_float(v[8 * g8 + i]);
                    if (TRAIN && p.epi == EPI_GELU2_BF16) {   // the pre-activation as well
                        uint4 u;
                        u.x = pack_bf16x2(f[0], f[1]);
                        u.y = pack_bf16x2(f[2], f[3]);
                        u.z = pack_bf16x2(f[4], f[5]);
                        u.w = pack_bf16x2(f[6], f[7]);
                        *reinterpret_cast<uint4*>(p.out2 + (int64_t)gr * p.ldo + n + 8 * g8) = u;
                    }
                    if (p.epi == EPI_GELU_BF16 || (TRAIN && p.epi == EPI_GELU2_BF16)) {
#pragma unroll
                        for (int i = 0; i < 8; i += 2) gelu_erf2(f[i], f[i + 1]);
                    }
                    uint4 u;
                    u.x = pack_bf16x2(f[0], f[1]);
                    u.y = pack_bf16x2(f[2], f[3]);
                    u.z = pack_bf16x2(f[4], f[5]);
                    u.w = pack_bf16x2(f[6], f[7]);
                    st_global_v4_hint(orow + 8 * g8, u, stream_pol);
                }
            } else {
                float* yrow = p.yacc + t.ks * p.y_split_stride + tok * p.ldy + n;
#pragma unroll
                for (int q = 0; q < 8; ++q) {
                    if (n + 4 * q >= p.N) break;
                    *reinterpret_cast<float4*>(yrow + 4 * q) =
                        make_float4(sc * __uint_as_float(v[4 * q]), sc * __uint_as_float(v[4 * q + 1]),
                                    sc * __uint_as_float(v[4 * q + 2]), sc * __uint_as_float(v[4 * q + 3]));
                }
            }
        }
        if (TRAIN && !to_f32 && (p.epi == EPI_DGELU_BF16 || p.epi == EPI_DSWIGLU_BF16) && ok_row &&
            p.dg_part)   // row dot (the gates' gradient; none for the shared expert)
            p.dg_part[(int64_t)(2 * (t.n0 / p.n_step) + half) * p.m_total + gr] = dg_acc;
    }
}

// STG_ROWS: rows per warp of the reduction staging buffer (EPI_ADD_F32), one kernel
// instance each so that the epilogue loops have constant trip counts.
template <int STG_ROWS, bool GATHER, int ECLS, bool TRAIN>
__global__ void __launch_bounds__(GM_THREADS, 1) grouped_gemm_kernel(const __grid_constant__ GemmArgs p) {
    extern __shared__ uint8_t gm_smem_raw[];
    uint8_t* smem = reinterpret_cast<uint8_t*>(
        (reinterpret_cast<uintptr_t>(gm_smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    uint8_t* sA = smem;
    const int nst = gm_stages(ECLS == ECLS_ADD ? EPI_ADD_F32 : p.epi, STG_ROWS);
    uint8_t* sB = smem + nst * GM_A_BYTES;
    uint8_t* sStg = sB + nst * GM_B_BYTES;                       // reduction staging (EPI_ADD_F32)
    uint64_t* bars = reinterpret_cast<uint64_t*>(sStg + gm_stg_bytes(ECLS == ECLS_ADD ? EPI_ADD_F32 : p.epi, STG_ROWS));
    uint32_t* tmem_slot = reinterpret_cast<uint32_t*>(bars + 3 * GM_STAGES_MAX + 5);
    volatile int* abort_flag = reinterpret_cast<volatile int*>(tmem_slot + 1);
    uint8_t* sink = reinterpret_cast<uint8_t*>(bars) + 256;   // 16-byte aligned, after the barriers

    Smem sm;
    sm.a0 = smem_u32(sA);
    sm.b0 = smem_u32(sB);
    sm.full = smem_u32(bars);
    sm.empty = sm.full + 8 * GM_STAGES_MAX;
    sm.afull = sm.empty + 8 * GM_STAGES_MAX;
    sm.tfull = sm.afull + 8 * GM_STAGES_MAX;
    sm.tempty = sm.tfull + 16;
    sm.drain = sm.tempty + 16;
    sm.nstages = nst;
    sm.stg = reinterpret_cast<float*>(sStg);
    sm.sink = smem_u32(sink);
    sm.rank = cluster_rank();
    sm.pair = blockIdx.x >> 1;
    sm.npairs = gridDim.x >> 1;

    const int warp = threadIdx.x >> 5;
    constexpr bool gather = GATHER;   // A rows gathered by the gather warps (else TMA)
    if (threadIdx.x == 0) {
        for (int s = 0; s < nst; ++s) {
            // leader's expect_tx arrival (+ the leader's forwarder; the peer's signals
            // are transaction bytes)
            mbar_init(sm.full + 8 * s, 1 + (gather ? 1 : 0));
            mbar_init(sm.empty + 8 * s, 1);         // multicast tcgen05.commit
            mbar_init(sm.afull + 8 * s, GM_GATHER_WARPS * 32);   // gather threads (async arrivals)
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(sm.tfull + 8 * a, 1);         // multicast tcgen05.commit
            mbar_init(sm.tempty + 8 * a, 2 * GM_EPI_WARPS);   // every epilogue warp of the pair
        }
        mbar_init(sm.drain, 1);
        *abort_flag = 0;
        mbar_fence_init();
    }
    if (warp == GM_WARP_MMA) {
        tmem_alloc_pair(smem_u32(tmem_slot), 2 * GM_MAXBN);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    cluster_sync();   // barriers of both CTAs initialised before any remote arrival
    tc_fence_after();
    pdl_wait();       // the previous kernel's outputs (tile tables, A, row maps) are ready
    const uint32_t tmem = *tmem_slot;
    int64_t n_mtiles;
    if (p.tiles) {
        n_mtiles = __ldg(p.n_tiles_dev);
        if (n_mtiles < 0 || n_mtiles > p.max_mtiles) {   // inconsistent offsets: no work
            if (threadIdx.x == 0) report(p.status, MOEVIE_ERR_DEVICE, SITE_GEMM_TILES, (int)n_mtiles, -1);
            n_mtiles = 0;
        }
    } else {
        n_mtiles = (p.m_total + GM_BM - 1) / GM_BM;
    }
    const int64_t n_work = p.item_table ? n_mtiles * p.ksplit : n_mtiles * p.n_ntiles * p.ksplit;

    if (warp < GM_EPI_WARPS) {
        epilogue<STG_ROWS, GATHER, ECLS, TRAIN>(p, sm, tmem, n_work, abort_flag);
    } else if (warp == GM_WARP_MMA) {
        if ((threadIdx.x & 31) == 0 && sm.rank == 0) mma_issuer<TRAIN>(p, sm, tmem, n_work, abort_flag);
    } else if (warp == GM_WARP_LOAD) {
        if ((threadIdx.x & 31) == 0) producer_tma<GATHER, TRAIN>(p, sm, n_work, abort_flag);
    } else if (warp == GM_WARP_FWD) {
        if constexpr (GATHER) {
            if ((threadIdx.x & 31) == 0) gather_forwarder(p, sm, n_work, abort_flag);
        }
    } else if constexpr (GATHER) {
        producer_gather(p, sm, n_work, abort_flag);
    } else if (!GATHER && ECLS == ECLS_F32 && (p.zero || p.nrm_out || p.wn_out) &&
               warp >= GM_WARP_GATHER && warp < GM_WARP_FWD) {
        // Side jobs for the gather warps of a dense-A GEMM, while the MMAs run.
        // 1. Row norms of the A rows of this CTA's items (the router's |x_t|, read while
        //    the TMA brings the same rows in): one warp per row, lanes over 16-byte chunks;
        //    the K splits of an m-tile share its rows.
        if (p.nrm_out) {
            const int q = warp - GM_WARP_GATHER, lane = threadIdx.x & 31;
            for (int64_t w = sm.pair; w < n_work; w += sm.npairs) {
                const Tile t = decode_tile(p, w);
                if (t.n0 != 0) continue;
                const int nh = rows_half(t, sm.rank);
                // the K splits of an m-tile share its rows: split ks takes rows ks mod ksplit
                for (int r = t.ks + q * p.ksplit; r < nh; r += GM_GATHER_WARPS * p.ksplit) {
                    const int64_t row = t.row0 + (int64_t)sm.rank * GM_HALF + r;
                    const uint4* v = reinterpret_cast<const uint4*>(p.nrm_x + row * p.nrm_ld);
                    float acc = 0.f;
                    for (int c = lane; c < p.nrm_cols / 8; c += 32) {
                        const uint4 u = v[c];
                        float f[8];
                        unpack_bf16x8(u, f);
#pragma unroll
                        for (int i = 0; i < 8; ++i) acc = fmaf(f[i], f[i], acc);
                    }
#pragma unroll
                    for (int o = 16; o; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
                    if (lane == 0) p.nrm_out[row] = sqrtf(acc);
                }
            }
        }
        // 2. Column norms from per-CTA partial sums of squares (wn_sets sets of wn_nparts
        //    parts): one warp per column, lanes over the parts, then a fixed shuffle tree
        //    (deterministic).
        if (p.wn_out) {
            const int q = warp - GM_WARP_GATHER, lane = threadIdx.x & 31;
            for (int j = blockIdx.x * GM_GATHER_WARPS + q; j < p.wn_sets * p.wn_E;
                 j += gridDim.x * GM_GATHER_WARPS) {
                const int set = j / p.wn_E, e = j - set * p.wn_E;
                const float* part = p.wn_part + (int64_t)set * p.wn_nparts * p.wn_Ep;
                float v = 0.f;
                for (int pp = lane; pp < p.wn_nparts; pp += 32) v += part[(int64_t)pp * p.wn_Ep + e];
#pragma unroll
                for (int o = 16; o; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
                if (lane == 0) p.wn_out[j] = sqrtf(v);
            }
        }
        // 3. Clear another buffer (the y accumulator) with 16-byte stores, grid-strided
        //    (evict-first: the zeros must not push the GEMM's re-read operands out of L2).
        if (p.zero) {
            const uint4 z = make_uint4(0u, 0u, 0u, 0u);
            const uint64_t pol = l2_policy_evict_first();
            const int64_t per = (int64_t)GM_GATHER_WARPS * 32;
            for (int64_t i = (int64_t)blockIdx.x * per + (threadIdx.x - GM_WARP_GATHER * 32);
                 i < p.zero_n; i += (int64_t)gridDim.x * per)
                st_global_v4_hint(p.zero + i, z, pol);
        }
    }

    tc_fence_before();
    __syncthreads();
    cluster_sync();   // the leader's MMAs have drained; both CTAs are done with TMEM
    if (warp == GM_WARP_MMA) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, 2 * GM_MAXBN);
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

bool make_weight_tmap_strided(CUtensorMap* tm, const void* base, int64_t N, int64_t K, int64_t G,
                              int64_t k_ld, int64_t g_ld) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[3] = {(cuuint64_t)N, (cuuint64_t)K, (cuuint64_t)G};
    cuuint64_t strides[2] = {(cuuint64_t)k_ld * 2, (cuuint64_t)g_ld * 2};
    cuuint32_t box[3] = {64, GM_BK, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims,
                     strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_weight_tmap(CUtensorMap* tm, const void* base, int64_t N, int64_t K, int64_t G) {
    return make_weight_tmap_strided(tm, base, N, K, G, N, N * K);
}

bool make_kmajor_tmap(CUtensorMap* tm, const void* base, int64_t K, int64_t N, int64_t G, int64_t k_ld,
                      int64_t g_ld, int box_n) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
    if (!enc || box_n < 8 || box_n > 256) return false;
    cuuint64_t dims[3] = {(cuuint64_t)K, (cuuint64_t)N, (cuuint64_t)G};
    cuuint64_t strides[2] = {(cuuint64_t)k_ld * 2, (cuuint64_t)g_ld * 2};
    cuuint32_t box[3] = {GM_BK, (cuuint32_t)box_n, 1};
    cuuint32_t estr[3] = {1, 1, 1};
    CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 3, const_cast<void*>(base), dims, strides, box,
                     estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_rows_tmap(CUtensorMap* tm, const void* base, int64_t cols, int64_t rows, int64_t ld) {
    PFN_cuTensorMapEncodeTiled_v12000 enc = get_encode_fn();
    if (!enc) return false;
    cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    cuuint64_t strides[1] = {(cuuint64_t)ld * 2};
    cuuint32_t box[2] = {64, (cuuint32_t)GM_HALF};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = enc(tm, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void*>(base), dims, strides,
                     box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
                     CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

void choose_bn(int N, int* BN, int* n_ntiles) {
    const int nt = (N + GM_MAXBN - 1) / GM_MAXBN;
    int bn = (N + nt - 1) / nt;
    bn = (bn + 31) / 32 * 32;   // each CTA of a pair holds BN / 2 columns, a multiple of 16
    *BN = bn;
    *n_ntiles = (N + bn - 1) / bn;
}

cudaError_t launch_grouped_gemm(const GemmArgs& a, int grid, cudaStream_t s) {
    if (a.stg_rows != 32 && a.stg_rows != 16) return cudaErrorInvalidValue;
    // one instance per (staging rows, A path, epilogue class, training-path layouts): each
    // holds only the code its launches run (constant trip counts, no other epilogue or
    // operand layout to crowd its registers)
    using Kern = void (*)(GemmArgs);
    static const Kern kerns[8] = {
        grouped_gemm_kernel<32, false, ECLS_ADD, false>, grouped_gemm_kernel<16, false, ECLS_ADD, false>,
        grouped_gemm_kernel<32, false, ECLS_F32, false>, grouped_gemm_kernel<32, false, ECLS_BF16, false>,
        grouped_gemm_kernel<32, true, ECLS_BF16, false>,
        // the training path: K-major B, M-major A, weight-gradient items, backward epilogues
        grouped_gemm_kernel<32, true, ECLS_BF16, true>, grouped_gemm_kernel<32, false, ECLS_ADD, true>,
        grouped_gemm_kernel<16, false, ECLS_ADD, true>};
    const bool gathered = a.a_rows || a.a_ident;   // A rows through the gather warps
    const bool train = a.b_kmajor || a.a_mn || a.item_table == 2 || a.epi == EPI_GELU2_BF16 ||
                       a.epi == EPI_DGELU_BF16 || a.epi == EPI_DSWIGLU_BF16 || a.out2 != nullptr;
    const bool bf16_out = a.epi == EPI_GELU_BF16 || a.epi == EPI_STORE_BF16 || a.epi == EPI_SWIGLU_BF16 ||
                          a.epi == EPI_GELU2_BF16 || a.epi == EPI_DGELU_BF16 || a.epi == EPI_DSWIGLU_BF16;
    if (gathered && !bf16_out) return cudaErrorInvalidValue;
    if (!gathered && a.epi == EPI_SWIGLU_BF16) return cudaErrorInvalidValue;
    Kern kern;
    if (train) {
        if (gathered) kern = kerns[5];
        else if (a.epi == EPI_ADD_F32) kern = a.stg_rows == 32 ? kerns[6] : kerns[7];
        else return cudaErrorInvalidValue;
    } else if (gathered) kern = kerns[4];
    else if (a.epi == EPI_ADD_F32) kern = a.stg_rows == 32 ? kerns[0] : kerns[1];
    else if (a.epi == EPI_STORE_F32 || a.epi == EPI_SUM2_F32) kern = kerns[2];
    else kern = kerns[3];
    static bool attr_set[64] = {};
    int dev = 0;
    cudaGetDevice(&dev);
    if (dev >= 0 && dev < 64 && !attr_set[dev]) {
        for (Kern k : kerns) {
            cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                                 GM_SMEM_BYTES_MAX);
            if (e != cudaSuccess) return e;
        }
        attr_set[dev] = true;
    }
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((grid + 1) & ~1));   // whole pairs
    cfg.blockDim = dim3(GM_THREADS);
    cfg.dynamicSmemBytes = gm_smem_bytes(a.epi, a.stg_rows);
    cfg.stream = s;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 2;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;   // see launch_pdl
    attr[1].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    cudaError_t e = cudaLaunchKernelEx(&cfg, kern, a);
    count_launches(1);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace mv
