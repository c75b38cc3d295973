/*
 * moevie.h -- C ABI of the GB300 (sm_103a) MoE-ViE fine-grained MoE FFN layer.
 *
 * The layer (paper "MoE-ViE", Sec. 2.1-2.2 and App. B, Algorithm 1) maps tokens
 * x[T, d] to y[T, d]:
 *
 *   s      = x . W_r                                  (Eq. 1; W_r stored [d, E])
 *   T(x)   = the k experts with the largest sigmoid(s_e) + b_e      (Eq. 7)
 *   g'_e   = sigmoid(s_e) / sum_{i in T(x)} sigmoid(s_i)            (Eqs. 4-5)
 *   y      = sum_{e in T(x)} g'_e E_e(x) + lambda * S(x)             (Eq. 6)
 *   E_e(x) = GELU(x W1[e]) W2[e],   S(x) = GELU(x Ws1) Ws2 (optional shared expert)
 *
 * GELU is the erf form u/2 (1 + erf(u / sqrt 2)).  The bias b only selects; it
 * never enters a gate.  Ties in the selection key go to the lower expert id.  A
 * token's k ids are stored in ascending order.  The expert-major row order is the
 * stable sort of the flat slots t*k + j by expert id (Algorithm 1, phase 1).
 *
 * Conventions for every entry point
 *  - Every array argument is DEVICE memory owned by the caller, unless a comment
 *    says otherwise.  The library never allocates, frees or synchronises on these
 *    calls (moevie_get_device_status excepted); all work is enqueued on `stream`
 *    (a cudaStream_t passed as void*; NULL is the legacy default stream) and runs
 *    asynchronously.
 *  - bf16 tensors are passed as void* pointing at __nv_bfloat16 data.  Matrices are
 *    row-major: x[T, d], W1[E, d, h], W2[E, h, d], Ws1[d, h_s], Ws2[h_s, d],
 *    y[T, d]; W_r[d, E] and b[E] are fp32.  Rows start 16 bytes apart: a matrix
 *    whose rows hold h values has row stride hp = h rounded up to a multiple of 8
 *    elements.  This matters only for W1 and W3 (stored [E][d][hp], expert stride
 *    d*hp) and Ws1 and Ws3 ([d][h_s rounded up to 8]) when h or h_s is not a
 *    multiple of 8 (the paper's L and H models: h = 684, 854); the pad columns are
 *    never read.  Every other matrix is dense.
 *  - Device pointers must be 16-byte aligned.  Sizes must satisfy d % 8 == 0,
 *    1 <= k <= E <= 1024 and T * k < 2^31; otherwise MOEVIE_ERR_UNSUPPORTED.
 *    T == 0 is valid and launches nothing.
 *  - Argument errors are reported synchronously, before anything is enqueued.
 *    A failed kernel launch returns MOEVIE_ERR_CUDA.  Errors found on the device
 *    (an out-of-range expert id, a pipeline wait that ran past its time limit) are
 *    written to a status block at the start of the workspace and read back with
 *    moevie_get_device_status; kernels never trap.
 *  - `ws` is caller-owned device scratch of `ws_bytes` bytes.  A workspace of
 *    moevie_workspace_size(T_max, d, E, k, h, h_s) bytes serves every entry point
 *    for any T <= T_max with the same sizes.  It must be set up once with
 *    moevie_workspace_init before first use.  Calls that share one workspace must
 *    be ordered on one stream.
 */
#ifndef MOEVIE_H
#define MOEVIE_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef int moevie_status;
#define MOEVIE_OK 0
#define MOEVIE_ERR_INVALID_ARG 1   /* null / misaligned pointer, negative size      */
#define MOEVIE_ERR_UNSUPPORTED 2   /* sizes outside the supported set above         */
#define MOEVIE_ERR_WORKSPACE 3     /* ws_bytes smaller than the entry point needs   */
#define MOEVIE_ERR_CUDA 4          /* a CUDA runtime call or kernel launch failed   */
#define MOEVIE_ERR_TIMEOUT 5       /* device: a bounded wait gave up (see status)   */
#define MOEVIE_ERR_DEVICE 6        /* device: a bounds check failed (see status)    */

/* Human-readable name of a status code (static string). */
const char* moevie_status_string(moevie_status s);

/* Library ABI version (major * 10000 + minor * 100 + patch). */
int moevie_version(void);

/* Bytes of workspace needed by moevie_moe_forward for up to T_max tokens (h_s = 0:
 * no shared expert).  Host-only; no device query.  Monotone in T_max. */
moevie_status moevie_workspace_size(int64_t T_max, int64_t d, int64_t E, int64_t k, int64_t h,
                                    int64_t h_s, size_t* bytes);

/* Zero the workspace's device status block (enqueued on stream).  Call once per
 * workspace before its first use; the status is sticky until cleared again. */
moevie_status moevie_workspace_init(void* ws, size_t ws_bytes, void* stream);

/* Router (Eqs. 1, 7, 4-5).  x bf16 [T, d], W_r fp32 [d, E], b fp32 [E].
 * Out: idx int32 [T, k] (ascending ids per token), gate fp32 [T, k] (same order).
 * Logits are fp32 (tensor cores); a token whose selection the fp32 logits cannot
 * certify (its k-th and (k+1)-th keys closer than their error bounds) is re-decided
 * from exact logits of the experts near its boundary -- an integer long accumulator
 * of the bf16 x fp32 products, within d 2^-64 sum|x_i w_i| of the exact dot product --
 * with the keys sigmoid(s) + b then formed in fp64, so idx equals the
 * exact-arithmetic selection. */
moevie_status moevie_route(const void* x, const float* W_r, const float* b, int64_t T, int64_t d,
                           int64_t E, int64_t k, int32_t* idx, float* gate, void* ws,
                           size_t ws_bytes, void* stream);

/* Expert-major order (App. B, Algorithm 1, phase 1: Sort, index = pos // K,
 * BinCount, CumSum).  idx int32 [T, k].  Out: counts int32 [E], offsets int32
 * [E + 1] (exclusive prefix; offsets[E] = the number of valid slots, T*k when every
 * id is valid), perm int32 [T*k] (row -> flat slot t*k + j, stable), inv int32 [T*k]
 * (flat slot -> row).  An id outside [0, E) is a device error (MOEVIE_ERR_DEVICE in
 * the status block): that slot is dropped, its inv entry is -1, it is not counted in
 * counts / offsets, and perm rows from offsets[E] to T*k are left unwritten. */
moevie_status moevie_permute(const int32_t* idx, int64_t T, int64_t k, int64_t E, int32_t* counts,
                             int32_t* offsets, int32_t* perm, int32_t* inv, void* ws,
                             size_t ws_bytes, void* stream);

/* Un-gated expert outputs in expert-major row order (App. B, Algorithm 1, Kernels
 * 1 and 2 without the routing weight): out_rows[r, :] = GELU(x[perm[r] / k] W1[e])
 * W2[e] for r in [offsets[e], offsets[e+1]).  out_rows bf16 [T*k, d]; fp32
 * accumulation, the hidden activation is rounded to bf16. */
moevie_status moevie_expert_ffn(const void* x, const int32_t* perm, const int32_t* offsets,
                                const void* W1, const void* W2, int64_t T, int64_t d, int64_t h,
                                int64_t E, int64_t k, void* out_rows, void* ws, size_t ws_bytes,
                                void* stream);

/* Shared expert (Sec. 2.2.1, Eq. 6, second term, without lambda):
 * out[t, :] = GELU(x[t] Ws1) Ws2, out bf16 [T, d]. */
moevie_status moevie_shared_expert(const void* x, const void* Ws1, const void* Ws2, int64_t T,
                                   int64_t d, int64_t h_s, void* out, void* ws, size_t ws_bytes,
                                   void* stream);

/* Gate-weighted combine (Eq. 6): y[t] = sum_j gate[t, j] out_rows[inv[t*k + j]]
 * + lambda * shared_out[t]   (shared_out bf16 [T, d] or NULL).  fp32 sums, y bf16. */
moevie_status moevie_combine(const void* out_rows, const int32_t* inv, const float* gate,
                             const void* shared_out, float lambda, int64_t T, int64_t k, int64_t d,
                             void* y, void* stream);

/* Layer description for moevie_moe_forward.  Weights are device pointers. */
typedef struct moevie_layer {
    int64_t d, E, k, h;
    int64_t h_s;            /* 0: no shared expert (Ws1, Ws2 ignored) */
    const float* W_r;       /* fp32 [d, E] */
    const float* b;         /* fp32 [E]    */
    const void* W1;         /* bf16 [E, d, h], rows h rounded up to 8 apart */
    const void* W2;         /* bf16 [E, h, d] */
    const void* Ws1;        /* bf16 [d, h_s], rows h_s rounded up to 8 apart */
    const void* Ws2;        /* bf16 [h_s, d]  */
    float lambda;           /* weight of the shared expert */
    const void* W3;         /* bf16 [E, d, h] (rows as W1) or NULL.  NULL: GELU experts GELU(x W1[e]) W2[e].
                             * Else SwiGLU experts (App. B): (SiLU(x W1[e]) * (x W3[e])) W2[e],
                             * W1 the gate and W3 the up projection. */
    const void* Ws3;        /* bf16 [d, h_s] (rows as Ws1): with W3, the shared expert's up projection
                             * (SwiGLU shared expert (SiLU(x Ws1) * (x Ws3)) Ws2); ignored
                             * without W3 or without a shared expert. */
} moevie_layer;

/* Optional routing by-products of moevie_moe_forward; any member may be NULL. */
typedef struct moevie_routing {
    int32_t* idx;       /* [T, k]   */
    float* gate;        /* [T, k]   */
    int32_t* counts;    /* [E]      */
    int32_t* offsets;   /* [E + 1]  */
    int32_t* perm;      /* [T * k]  */
    int32_t* inv;       /* [T * k]  */
} moevie_routing;

/* The whole layer forward (Eqs. 1, 4-7; Algorithm 1): router, expert-major
 * order, grouped up-projection with GELU fused into its epilogue and the token
 * gather fused into its operand load, grouped down-projection whose epilogue
 * scales each row by its gate and adds it into an fp32 accumulator of y (the
 * scatter-add of Algorithm 1), and the shared expert.  x bf16 [T, d] -> y bf16
 * [T, d].  `routing` may be NULL. */
moevie_status moevie_moe_forward(const moevie_layer* layer, const void* x, int64_t T, void* y,
                                 const moevie_routing* routing, void* ws, size_t ws_bytes,
                                 void* stream);

/* The layer from host memory to host memory, the copies overlapped with the compute.
 * Every token's output depends on that token alone (Eqs. 4-7: routing, gates and the
 * experts act per token), so the layer runs piece by piece over contiguous token ranges
 * of at most Tc = ceil(T / chunks) tokens: one piece with chunks = 1; otherwise a first
 * piece of ceil(Tc / 2) tokens, then pieces of Tc, the last one what is left (so the first
 * copy in and the last copy out, which no layer hides, are short).  A piece's rows of x
 * go from x_host to x_dev on the library's copy-in stream, moevie_moe_forward runs it on
 * `stream`, and its rows of y go from y_dev to y_host on the copy-out stream, so each
 * piece's layer overlaps the copies of its neighbours.  `stream` completes after the last
 * copy out: synchronise it (or wait on it) before reading y_host.
 * x_host, y_host: host memory [T, d] bf16 (pinned, for the copies to be asynchronous);
 * x_dev, y_dev: caller-owned device buffers [T, d] bf16, 16-byte aligned; ws:
 * moevie_workspace_size(Tc, ...) bytes at least, set up with moevie_workspace_init;
 * 1 <= chunks <= MOEVIE_HOST_MAX_CHUNKS, else MOEVIE_ERR_UNSUPPORTED.  The first call in a
 * context creates the two copy streams and their events (make it before any stream
 * capture); calls on one device share them, so calls from several host threads must
 * not overlap.  Errors as for moevie_moe_forward; device errors land in ws's status. */
#define MOEVIE_HOST_MAX_CHUNKS 16
moevie_status moevie_moe_forward_host(const moevie_layer* layer, const void* x_host, int64_t T, void* y_host,
                                      void* x_dev, void* y_dev, int64_t chunks, void* ws, size_t ws_bytes,
                                      void* stream);

/* moevie_permute without a workspace (the paper has no counterpart: this is a
 * calling convention, not part of the method).  Same inputs, outputs, ordering and
 * validation as moevie_permute, and bit-identical results.
 *
 * Who it is for: callers that cannot give the library scratch memory and cannot let
 * it allocate any -- e.g. code running inside another framework's operator that
 * only hands over its input and output buffers, or a process whose device memory
 * is all reserved up front by its own pool, where a cudaMalloc would fail or would
 * synchronise the device at a bad moment.  This entry point makes no cudaMalloc or
 * cudaFree and calls no allocating library: its scratch is one fixed array of
 * 2,179,584 bytes in the library's device image, one copy per device.
 *
 * Limits: T * k <= 1048576 (2^20) flat slots, plus the limits of moevie_permute
 * (1 <= k <= E <= 1024); larger inputs return MOEVIE_ERR_UNSUPPORTED before
 * anything is enqueued.
 *
 * Set-up: the first call on a device (with that device current) looks up the
 * array's device address, which may load the library's device code; make that
 * first call before any stream capture.  Later calls reuse the address as long as
 * the device's context is the same; after cudaDeviceReset the next call looks it up
 * again in the new context (again, before any capture).
 *
 * Concurrency: all calls on one device share the one array.  Two calls whose GPU
 * work overlaps (different streams, or several host threads without ordering) race
 * on it and give undefined results; order them on one stream or with events.
 *
 * Device-side errors: each call clears the array's status block; an expert id
 * outside [0, E) drops its slot (inv = -1, not counted in counts / offsets) and is
 * recorded there, but no entry point reads that status back -- check inv for -1
 * where ids are untrusted. */
moevie_status moevie_permute_static(const int32_t* idx, int64_t T, int64_t k, int64_t E,
                                    int32_t* counts, int32_t* offsets, int32_t* perm,
                                    int32_t* inv, void* stream);

/* Number of kernels this library has launched since it was loaded (all
 * threads, all devices).  Host-only. */
uint64_t moevie_launch_count(void);

/* Loss-free balancing (Sec. 2.2.2): update the selection bias b[E] (fp32, device,
 * in place) from one step's expert loads counts[E] (int32, device; e.g. the counts
 * moevie_permute / moevie_moe_forward return), E <= 1024.  With mu the mean load and
 * sigma the population standard deviation of the loads over the E experts:
 *   rule 0, z-score (Eq. 9):  b_e <- b_e - alpha (t_e - mu) / sigma
 *                              (all loads equal, sigma = 0: b unchanged)
 *   rule 1, sign (Eq. 8):     b_e <- b_e - alpha sign(t_e - mu), sign(0) = 0.
 * Arithmetic in fp64, each new b_e rounded to fp32.  One tiny kernel on `stream`;
 * `ws` (>= 256 bytes, the workspace of the other entry points will do) receives the
 * device status: a negative load leaves b unchanged and records MOEVIE_ERR_DEVICE.
 * Argument errors (E outside [1, 1024], rule not 0 or 1, null or misaligned
 * pointers) return before anything is enqueued. */
moevie_status moevie_update_bias(const int32_t* counts, int64_t E, float alpha, int rule, float* b,
                                 void* ws, size_t ws_bytes, void* stream);

/* Launch plan of moevie_moe_forward for these sizes, GELU or SwiGLU experts alike
 * (host-only, no GPU work; the paper has no counterpart -- it describes how this
 * library schedules Eq. 6's shared term).  Returns the number S of always-on groups of
 * width h that carry the shared expert inside the routed up- and down-projection
 * launches (its hidden units in S = h_s / h chunks, every token with gate lambda), or 0
 * when it runs as its own GEMMs (no shared expert, h not dividing h_s, several chunks
 * of a width h that is not a multiple of 8, or a band-ordered down-projection).
 * Invalid sizes return 0. */
int64_t moevie_shared_groups(int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t h_s);

/* ---------------------------------------------------------------- training path
 *
 * Backward pass of the layer, GELU or SwiGLU experts, with or without a shared expert (App. B:
 * the paper trains with grouped GEMMs and applies the activation as its own step).  Given
 * the forward's selection idx (held fixed: top-k is piecewise constant in the logits, so
 * it has no gradient) and the output gradient dy, it returns the gradients of
 * L = sum_t dy_t . y_t:
 *   through each selected expert e of token t, with gate g (Eqs. 4-5) and the hidden
 *   activation a (GELU(u), u = x_t W1[e]; SwiGLU: SiLU(u) v, v = x_t W3[e]):
 *     dW2[e] += a^T (g dy_t),   da = g dy_t W2[e]^T,
 *     GELU:   du = da GELU'(u);   SwiGLU: du = da v SiLU'(u), dv = da SiLU(u),
 *     dW1[e] += x_t^T du,  dW3[e] += x_t^T dv,  dx_t += du W1[e]^T + dv W3[e]^T;
 *   through the gates (Eqs. 4-5), with sigma_j = sigmoid(s_{e_j}), S = sum_j sigma_j and
 *   dg_j = dy_t . E_{e_j}(x_t):
 *     ds_{e_j} = sigma_j (1 - sigma_j) (dg_j - sum_l g_l dg_l) / S,
 *     dW_r[:, e_j] += x_t ds_{e_j},   dx_t += ds_{e_j} W_r[:, e_j];
 *   through the shared expert (Eq. 6, second term; h_s > 0), every token with the
 *   constant weight lambda, the expert's rules with g = lambda and Ws1, Ws2, Ws3 in place
 *   of W1[e], W2[e], W3[e] (lambda gets no gradient).
 * The bias b gets no gradient (it only selects; moevie_update_bias moves it).
 *
 * Inputs: the layer (W_r, W1, W2, for SwiGLU experts W3, and the shared expert's Ws1, Ws2,
 * Ws3 and lambda when h_s > 0, as for moevie_moe_forward), x bf16 [T, d], dy bf16 [T, d],
 * idx int32 [T, k] (the forward's selection, e.g. moevie_routing.idx; ids in [0, E)).
 * Outputs, fp32, all overwritten: dx [T, d], dW_r [d, E], dW1 [E, d, h] with rows h
 * rounded up to 8 apart (as W1; the pad columns hold zeros), dW2 [E, h, d], for SwiGLU
 * experts dW3 laid out as dW1 (NULL otherwise); with a shared expert dWs1 [d, h_s] with
 * rows h_s rounded up to 8 apart (as Ws1), dWs2 [h_s, d] and, for SwiGLU, dWs3 laid out as
 * dWs1 (all three NULL without one).  The gates are recomputed from x and W_r in fp32.
 * Arithmetic: bf16 GEMM operands with fp32 accumulation (the recomputed pre-activations,
 * activations, their gradients, g dy and ds are rounded to bf16 as GEMM operands); dx,
 * and every weight gradient summed over more than 4096 rows (an expert's rows padded to
 * 64; all T tokens for dW_r and the shared expert's), take fp32 reductions over chunks of
 * rows, so their last bits depend on the order in which the GEMM's work items finish;
 * the other weight gradients are written once.  Sizes: k <= 32, d and h <=
 * 65535 (h_s too), plus the limits of moevie_moe_forward.  `ws`:
 * moevie_backward_workspace_size(T_max, d, E, k, h, h_s, swiglu) bytes (swiglu nonzero for
 * SwiGLU experts), set up with moevie_workspace_init; device errors land in its status
 * block. */
moevie_status moevie_backward_workspace_size(int64_t T_max, int64_t d, int64_t E, int64_t k, int64_t h,
                                             int64_t h_s, int swiglu, size_t* bytes);
moevie_status moevie_moe_backward(const moevie_layer* layer, const void* x, const void* dy, int64_t T,
                                  const int32_t* idx, float* dx, float* dW_r, float* dW1, float* dW2,
                                  float* dW3, float* dWs1, float* dWs2, float* dWs3, void* ws,
                                  size_t ws_bytes, void* stream);

/* Synchronise `stream`, then read the workspace's device status into *out
 * (MOEVIE_OK when no device-side error was recorded).  `detail` (host, may be
 * NULL) receives 4 ints: code, site, and two values describing the failure. */
moevie_status moevie_get_device_status(const void* ws, void* stream, moevie_status* out,
                                       int32_t* detail);

#ifdef __cplusplus
}
#endif

#endif /* MOEVIE_H */
