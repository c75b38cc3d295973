/*
 * moevie_testing.h -- test hooks of the MoE-ViE layer library.
 *
 * These entry points are not part of the layer.  They expose single steps of
 * moevie_moe_forward so that each can be compared with the oracle on its own,
 * and they exercise the device error path without faulting or hanging a GPU.
 * Conventions (device memory, alignment, workspace, status block) are those of
 * moevie.h.
 */
#ifndef MOEVIE_TESTING_H
#define MOEVIE_TESTING_H

#include "moevie.h"

#ifdef __cplusplus
extern "C" {
#endif

/* Router logits as the fast path computes them (Eq. 1 on the tensor cores): W_r is
 * split into bf16 pieces hi = bf16(w), mid = bf16(w - hi), and s[t, e] = sum_i x[t, i]
 * (hi + mid)[i, e] with fp32 accumulation (for E <= 128 the two pieces' products are
 * accumulated separately and added hi + mid).  The left-out lo = w - hi - mid is part of
 * the certified error bound, not of these logits.  s fp32 [T, E32] with E32 = E rounded
 * up to a multiple of 32 (the extra columns are zero). */
moevie_status moevie_test_route_logits(const void* x, const float* W_r, int64_t T, int64_t d,
                                       int64_t E, float* s, void* ws, size_t ws_bytes,
                                       void* stream);

/* Synchronise `stream`; *out = number of tokens that the last moevie_route /
 * moevie_moe_forward on this workspace re-decided with exact logits. */
moevie_status moevie_test_fallback_count(const void* ws, void* stream, int32_t* out);

/* The up-projection step alone (App. B, Algorithm 1, Kernel 1 with GELU):
 * hidden[r, :] = bf16(GELU(x[perm[r] / k] W1[e])) for r in expert e's segment.
 * hidden bf16 [T*k, h] with row stride h rounded up to a multiple of 8 (as W1). */
moevie_status moevie_test_expert_hidden(const void* x, const int32_t* perm, const int32_t* offsets,
                                        const void* W1, int64_t T, int64_t d, int64_t h, int64_t E,
                                        int64_t k, void* hidden, void* ws, size_t ws_bytes,
                                        void* stream);

/* moevie_moe_forward (routing by-products not returned) that also records 7 CUDA
 * events (cudaEvent_t passed as void*) on `stream`: before the router, then after
 * the router, the expert-major order, the y-accumulator set-up (shared expert or
 * zero fill), the grouped up-projection, the grouped down-projection with the
 * combine epilogue, and the final bf16 conversion.  n_events must be 7. */
moevie_status moevie_test_moe_forward_events(const moevie_layer* layer, const void* x, int64_t T,
                                             void* y, void* ws, size_t ws_bytes, void* stream,
                                             void* const* events, int n_events);

/* Launch one CTA that waits on a shared-memory barrier nobody arrives at.  The
 * wait gives up after limit_ns nanoseconds of device time, records
 * MOEVIE_ERR_TIMEOUT in the workspace status block and the kernel returns.
 * limit_ns must be in (0, 10^10]. */
moevie_status moevie_test_wait_timeout(void* ws, size_t ws_bytes, uint64_t limit_ns, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* MOEVIE_TESTING_H */
