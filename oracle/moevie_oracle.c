/*
 * moevie_oracle.c -- plain, slow, fp64 CPU oracle of the MoE-ViE fine-grained
 * mixture-of-experts FFN layer: forward pass, bias update and backward pass.
 *
 * TEST INFRASTRUCTURE, NOT PRODUCT CODE.  This file exists only so that the
 * CUDA library can be checked against an independent statement of the method.
 * Only the tests, the smoke check and the benchmark's CPU-baseline leg may load
 * it.  It shares no code, header, table or helper with the CUDA library.
 *
 * What it computes (paper: "MoE-ViE", Sec. 2.1-2.2, App. B):
 *   Eq. (1)      s = W_r x                     router logits, here x.W_r with
 *                                              W_r stored [d, E]
 *   Eq. (7)      selection by top-k(Sigmoid(s) + b)
 *   Eq. (4)-(5)  gates: Sigmoid(s) of the selected experts, renormalised to
 *                sum to one (the bias b only selects; it is not part of g)
 *   Eq. (3)/(6)  y = sum_{e in T(x)} g'_e E_e(x) + lambda * sum_shared E_s(x)
 *   expert       E_e(x) = GELU(x W1[e]) W2[e], GELU(u) = u/2 (1 + erf(u/sqrt 2)),
 *                or the SwiGLU expert of App. B: (SiLU(x W1[e]) * (x W3[e])) W2[e],
 *                SiLU(v) = v / (1 + exp(-v))
 *   App. B, Algorithm 1 phase 1: the sort of the flattened routing indices by
 *                expert, its histogram and exclusive prefix sum (offsets).
 *
 * Readings of points the paper leaves open (each is listed in the design notes):
 *   - ties in the selection key go to the lower expert id;
 *   - a token's k selected ids are stored in ascending id order;
 *   - the sort of Algorithm 1 is stable: inside one expert's segment, rows keep
 *     ascending flat-slot order t*k + j;
 *   - the shared expert has its own width h_s, its weight lambda multiplies it,
 *     and it is not renormalised together with the routed gates.
 *
 * Arithmetic: every input is widened exactly to double (bf16 and fp32 values
 * are exact doubles, and so is every product x_i * w_i of a bf16 and an fp32
 * number, since 8 + 24 mantissa bits fit in 53).  Sums run in ascending index
 * order in double.  exp() and erf() are the C library's.  Nothing is blocked,
 * fused or reordered beyond that.  Build with -ffp-contract=off so that no
 * compiler contracts a*b+c into a fused multiply-add, which keeps the results
 * the same on x86-64 and aarch64.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_OK 0
#define ORACLE_ERR_ARG 1
#define ORACLE_ERR_NOMEM 2

/* ---------------------------------------------------------------- helpers */

/* A bf16 value is the upper half of an IEEE fp32 value. */
static double bf16_to_double(uint16_t v) {
    uint32_t bits = ((uint32_t)v) << 16;
    float f;
    memcpy(&f, &bits, sizeof f);
    return (double)f;
}

static double sigmoid(double s) { return 1.0 / (1.0 + exp(-s)); }

static double gelu(double u) { return 0.5 * u * (1.0 + erf(u / sqrt(2.0))); }

/* Parallel-for over [0, n) with plain pthreads; each worker takes a contiguous
 * block of items.  Work items never share output memory. */
typedef void (*item_fn)(void* ctx, int64_t begin, int64_t end);
typedef struct { item_fn fn; void* ctx; int64_t begin, end; } worker_arg;

static void* worker_main(void* p) {
    worker_arg* a = (worker_arg*)p;
    a->fn(a->ctx, a->begin, a->end);
    return NULL;
}

static void parallel_for(int64_t n, int nthreads, item_fn fn, void* ctx) {
    if (n <= 0) return;
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 256) nthreads = 256;
    if ((int64_t)nthreads > n) nthreads = (int)n;
    if (nthreads == 1) { fn(ctx, 0, n); return; }
    pthread_t th[256];
    worker_arg args[256];
    int started[256];
    int64_t chunk = (n + nthreads - 1) / nthreads;
    for (int i = 0; i < nthreads; ++i) {
        args[i].fn = fn; args[i].ctx = ctx;
        args[i].begin = (int64_t)i * chunk;
        args[i].end = args[i].begin + chunk < n ? args[i].begin + chunk : n;
        started[i] = 0;
        if (args[i].begin >= args[i].end) continue;
        if (pthread_create(&th[i], NULL, worker_main, &args[i]) == 0) started[i] = 1;
        else worker_main(&args[i]);   /* could not spawn: run it here */
    }
    for (int i = 0; i < nthreads; ++i)
        if (started[i]) pthread_join(th[i], NULL);
}

/* ------------------------------------------------------ Eq. (1): logits */

/* s[t, e] = sum_i x[t, i] * W_r[i, e]   (x bf16 [T, d], W_r fp32 [d, E]).
 * The loop over i is outermost so that W_r is read row by row; each s[t, e]
 * is still one sum taken in ascending i. */
static void logits_row(const uint16_t* xt, const float* Wr, int64_t d, int64_t E, double* st) {
    for (int64_t e = 0; e < E; ++e) st[e] = 0.0;
    for (int64_t i = 0; i < d; ++i) {
        double xi = bf16_to_double(xt[i]);
        const float* wi = Wr + i * E;
        for (int64_t e = 0; e < E; ++e) st[e] += xi * (double)wi[e];
    }
}

typedef struct { const uint16_t* x; const float* Wr; int64_t d, E; double* s; } logits_ctx;

static void logits_items(void* p, int64_t t0, int64_t t1) {
    logits_ctx* c = (logits_ctx*)p;
    for (int64_t t = t0; t < t1; ++t)
        logits_row(c->x + t * c->d, c->Wr, c->d, c->E, c->s + t * c->E);
}

int oracle_logits(const uint16_t* x, const float* Wr, int64_t T, int64_t d, int64_t E,
                  double* s, int nthreads) {
    if (T < 0 || d <= 0 || E <= 0 || (T > 0 && (!x || !Wr || !s))) return ORACLE_ERR_ARG;
    logits_ctx c = { x, Wr, d, E, s };
    parallel_for(T, nthreads, logits_items, &c);
    return ORACLE_OK;
}

/* ------------------------------------------- Eqs. (7), (4), (5): routing */

/* Select the k experts with the largest key_e = Sigmoid(s_e) + b_e (Eq. 7).
 * Repeated arg-max over the experts not yet chosen; a tie goes to the lower id
 * because the scan keeps the first maximum it meets.  The chosen ids are then
 * sorted ascending.  Gates are Sigmoid(s) of the chosen experts divided by their
 * sum (Eqs. 4-5); the bias does not enter them.  margin = (smallest chosen key)
 * - (largest key left out), +inf when k == E. */
static void select_one(const double* st, const float* b, int64_t E, int64_t k,
                       int32_t* idx, double* gate, double* margin, unsigned char* taken,
                       double* key) {
    for (int64_t e = 0; e < E; ++e) { key[e] = sigmoid(st[e]) + (double)b[e]; taken[e] = 0; }
    double min_chosen = INFINITY;
    for (int64_t j = 0; j < k; ++j) {
        int64_t best = -1;
        for (int64_t e = 0; e < E; ++e) {
            if (taken[e]) continue;
            if (best < 0 || key[e] > key[best]) best = e;
        }
        taken[best] = 1;
        idx[j] = (int32_t)best;
        if (key[best] < min_chosen) min_chosen = key[best];
    }
    /* ascending id order (insertion sort: k is small) */
    for (int64_t j = 1; j < k; ++j) {
        int32_t v = idx[j];
        int64_t i = j - 1;
        while (i >= 0 && idx[i] > v) { idx[i + 1] = idx[i]; --i; }
        idx[i + 1] = v;
    }
    double sum = 0.0;
    for (int64_t j = 0; j < k; ++j) sum += sigmoid(st[idx[j]]);
    for (int64_t j = 0; j < k; ++j) gate[j] = sigmoid(st[idx[j]]) / sum;
    double max_left = -INFINITY;
    for (int64_t e = 0; e < E; ++e)
        if (!taken[e] && key[e] > max_left) max_left = key[e];
    if (margin) *margin = (k == E) ? INFINITY : (min_chosen - max_left);
}

typedef struct {
    const double* s; const float* b; int64_t E, k;
    int32_t* idx; double* gate; double* margin; int err;
} select_ctx;

static void select_items(void* p, int64_t t0, int64_t t1) {
    select_ctx* c = (select_ctx*)p;
    unsigned char* taken = (unsigned char*)malloc((size_t)c->E);
    double* key = (double*)malloc((size_t)c->E * sizeof(double));
    if (!taken || !key) { c->err = ORACLE_ERR_NOMEM; free(taken); free(key); return; }
    for (int64_t t = t0; t < t1; ++t)
        select_one(c->s + t * c->E, c->b, c->E, c->k, c->idx + t * c->k, c->gate + t * c->k,
                   c->margin ? c->margin + t : NULL, taken, key);
    free(taken); free(key);
}

int oracle_select(const double* s, const float* b, int64_t T, int64_t E, int64_t k,
                  int32_t* idx, double* gate, double* margin, int nthreads) {
    if (T < 0 || E <= 0 || k < 1 || k > E) return ORACLE_ERR_ARG;
    if (T > 0 && (!s || !b || !idx || !gate)) return ORACLE_ERR_ARG;
    select_ctx c = { s, b, E, k, idx, gate, margin, ORACLE_OK };
    parallel_for(T, nthreads, select_items, &c);
    return c.err;
}

/* ------------------------------- Algorithm 1, phase 1: expert-major order */

/* counts[e] = number of flat slots (t, j) with idx[t*k + j] == e (BinCount);
 * offsets = exclusive prefix sum of counts, E + 1 entries (CumSum);
 * perm[r] = flat slot placed at row r by a stable counting sort on the expert
 * id (rows of one expert keep ascending slot order); inv[perm[r]] = r.
 * The token of row r is perm[r] / k, the "index" of Algorithm 1. */
int oracle_permute(const int32_t* idx, int64_t T, int64_t k, int64_t E,
                   int32_t* counts, int32_t* offsets, int32_t* perm, int32_t* inv) {
    if (T < 0 || k < 1 || E <= 0 || !counts || !offsets) return ORACLE_ERR_ARG;
    if (T > 0 && (!idx || !perm || !inv)) return ORACLE_ERR_ARG;
    int64_t n = T * k;
    for (int64_t e = 0; e < E; ++e) counts[e] = 0;
    for (int64_t i = 0; i < n; ++i) {
        if (idx[i] < 0 || idx[i] >= E) return ORACLE_ERR_ARG;
        counts[idx[i]] += 1;
    }
    offsets[0] = 0;
    for (int64_t e = 0; e < E; ++e) offsets[e + 1] = offsets[e] + counts[e];
    int64_t* cursor = (int64_t*)malloc((size_t)E * sizeof(int64_t));
    if (!cursor) return ORACLE_ERR_NOMEM;
    for (int64_t e = 0; e < E; ++e) cursor[e] = offsets[e];
    for (int64_t i = 0; i < n; ++i) {
        int64_t r = cursor[idx[i]]++;
        perm[r] = (int32_t)i;
        inv[i] = (int32_t)r;
    }
    free(cursor);
    return ORACLE_OK;
}

/* ------------------------------------------------ one expert on one token */

/* hidden[n] = GELU(sum_i x[i] W1[e, i, n])  for n < h   (W1 bf16 [E, d, h]).
 * i is the outer loop (W1 read row by row); each pre-activation is still one
 * sum in ascending i, and GELU is applied once it is complete. */
static void expert_hidden(const uint16_t* xt, const uint16_t* W1e, int64_t d, int64_t h, double* hidden) {
    for (int64_t n = 0; n < h; ++n) hidden[n] = 0.0;
    for (int64_t i = 0; i < d; ++i) {
        double xi = bf16_to_double(xt[i]);
        const uint16_t* wi = W1e + i * h;
        for (int64_t n = 0; n < h; ++n) hidden[n] += xi * bf16_to_double(wi[n]);
    }
    for (int64_t n = 0; n < h; ++n) hidden[n] = gelu(hidden[n]);
}

static double silu(double v) { return v / (1.0 + exp(-v)); }

/* SwiGLU expert (the paper's own FFN, App. B):
 * hidden[n] = SiLU(sum_i x[i] W1[e, i, n]) * (sum_i x[i] W3[e, i, n]),
 * both sums in ascending i, the product formed once both are complete. */
static void expert_hidden_swiglu(const uint16_t* xt, const uint16_t* W1e, const uint16_t* W3e,
                                 int64_t d, int64_t h, double* hidden, double* up) {
    for (int64_t n = 0; n < h; ++n) hidden[n] = up[n] = 0.0;
    for (int64_t i = 0; i < d; ++i) {
        double xi = bf16_to_double(xt[i]);
        const uint16_t* wi = W1e + i * h;
        const uint16_t* vi = W3e + i * h;
        for (int64_t n = 0; n < h; ++n) {
            hidden[n] += xi * bf16_to_double(wi[n]);
            up[n] += xi * bf16_to_double(vi[n]);
        }
    }
    for (int64_t n = 0; n < h; ++n) hidden[n] = silu(hidden[n]) * up[n];
}

/* out[c] = sum_n hidden[n] W2[e, n, c]  for c < d   (W2 bf16 [E, h, d]);
 * n outermost, each out[c] one sum in ascending n. */
static void expert_down(const double* hidden, const uint16_t* W2e, int64_t h, int64_t d, double* out) {
    for (int64_t c = 0; c < d; ++c) out[c] = 0.0;
    for (int64_t n = 0; n < h; ++n) {
        double a = hidden[n];
        const uint16_t* wn = W2e + n * d;
        for (int64_t c = 0; c < d; ++c) out[c] += a * bf16_to_double(wn[c]);
    }
}

static int64_t expert_of_row(const int32_t* offsets, int64_t E, int64_t r) {
    for (int64_t e = 0; e < E; ++e)
        if (r >= offsets[e] && r < offsets[e + 1]) return e;
    return -1;
}

typedef struct {
    const uint16_t* x; const int32_t* perm; const int32_t* offsets;
    const uint16_t* W1; const uint16_t* W2; int64_t T, d, h, E, k;
    const int32_t* rows; double* out; int want_hidden; int err;
} rows_ctx;

static void rows_items(void* p, int64_t i0, int64_t i1) {
    rows_ctx* c = (rows_ctx*)p;
    double* hidden = (double*)malloc((size_t)c->h * sizeof(double));
    if (!hidden) { c->err = ORACLE_ERR_NOMEM; return; }
    for (int64_t i = i0; i < i1; ++i) {
        int64_t r = c->rows[i];
        int64_t e = expert_of_row(c->offsets, c->E, r);
        int64_t t = c->perm[r] / c->k;
        if (e < 0 || t < 0 || t >= c->T) { c->err = ORACLE_ERR_ARG; continue; }
        expert_hidden(c->x + t * c->d, c->W1 + e * c->d * c->h, c->d, c->h, hidden);
        if (c->want_hidden) memcpy(c->out + i * c->h, hidden, (size_t)c->h * sizeof(double));
        else expert_down(hidden, c->W2 + e * c->h * c->d, c->h, c->d, c->out + i * c->d);
    }
    free(hidden);
}

/* Un-gated expert output of selected expert-major rows:
 * out[i, :] = E_e(x_t) with r = rows[i], e the expert whose segment holds r,
 * t = perm[r] / k.  want_hidden != 0 returns GELU(x_t W1[e]) ([nrows, h]) instead. */
int oracle_expert_rows(const uint16_t* x, const int32_t* perm, const int32_t* offsets,
                       const uint16_t* W1, const uint16_t* W2, int64_t T, int64_t d, int64_t h,
                       int64_t E, int64_t k, const int32_t* rows, int64_t nrows, int want_hidden,
                       double* out, int nthreads) {
    if (T < 0 || d <= 0 || h <= 0 || E <= 0 || k < 1 || nrows < 0) return ORACLE_ERR_ARG;
    if (nrows > 0 && (!x || !perm || !offsets || !W1 || (!want_hidden && !W2) || !rows || !out))
        return ORACLE_ERR_ARG;
    rows_ctx c = { x, perm, offsets, W1, W2, T, d, h, E, k, rows, out, want_hidden, ORACLE_OK };
    parallel_for(nrows, nthreads, rows_items, &c);
    return c.err;
}

/* ------------------------------------------------------ Eq. (6): combine */

/* y[t] = sum_j gate[t*k+j] * rows_out[inv[t*k+j]] + lambda * shared[t]
 * (shared may be NULL).  All arrays are double. */
int oracle_combine(const double* rows_out, const int32_t* inv, const double* gate,
                   const double* shared, double lambda, int64_t T, int64_t k, int64_t d, double* y) {
    if (T < 0 || k < 1 || d <= 0) return ORACLE_ERR_ARG;
    if (T > 0 && (!rows_out || !inv || !gate || !y)) return ORACLE_ERR_ARG;
    for (int64_t t = 0; t < T; ++t)
        for (int64_t c = 0; c < d; ++c) {
            double acc = 0.0;
            for (int64_t j = 0; j < k; ++j)
                acc += gate[t * k + j] * rows_out[(int64_t)inv[t * k + j] * d + c];
            if (shared) acc += lambda * shared[t * d + c];
            y[t * d + c] = acc;
        }
    return ORACLE_OK;
}

/* ------------------------------------- the whole layer, token by token */

typedef struct {
    const uint16_t* x; const float* Wr; const float* b; const uint16_t* W1; const uint16_t* W2;
    const uint16_t* W3; const uint16_t* Ws1; const uint16_t* Ws2; const uint16_t* Ws3; double lambda;
    int64_t T, d, E, k, h, hs;
    const int32_t* tokens; double* y; int32_t* idx; double* gate; double* margin;
    double* shared_out; int err;
} fwd_ctx;

static void fwd_items(void* p, int64_t i0, int64_t i1) {
    fwd_ctx* c = (fwd_ctx*)p;
    int64_t hmax = c->h > c->hs ? c->h : c->hs;
    double* s = (double*)malloc((size_t)c->E * sizeof(double));
    double* key = (double*)malloc((size_t)c->E * sizeof(double));
    unsigned char* taken = (unsigned char*)malloc((size_t)c->E);
    double* hidden = (double*)malloc((size_t)hmax * sizeof(double));
    double* up = (double*)malloc((size_t)hmax * sizeof(double));
    double* o = (double*)malloc((size_t)c->d * sizeof(double));
    int32_t* sel = (int32_t*)malloc((size_t)c->k * sizeof(int32_t));
    double* g = (double*)malloc((size_t)c->k * sizeof(double));
    if (!s || !key || !taken || !hidden || !up || !o || !sel || !g) {
        c->err = ORACLE_ERR_NOMEM;
        goto done;
    }
    for (int64_t i = i0; i < i1; ++i) {
        int64_t t = c->tokens ? c->tokens[i] : i;
        if (t < 0 || t >= c->T) { c->err = ORACLE_ERR_ARG; continue; }
        const uint16_t* xt = c->x + t * c->d;
        logits_row(xt, c->Wr, c->d, c->E, s);                                              /* Eq. 1 */
        double m;
        select_one(s, c->b, c->E, c->k, sel, g, &m, taken, key);                          /* Eqs. 7, 4, 5 */
        double* yt = c->y + i * c->d;
        for (int64_t col = 0; col < c->d; ++col) yt[col] = 0.0;
        for (int64_t j = 0; j < c->k; ++j) {                                               /* Eq. 6, routed */
            int64_t e = sel[j];
            if (c->W3)
                expert_hidden_swiglu(xt, c->W1 + e * c->d * c->h, c->W3 + e * c->d * c->h, c->d, c->h,
                                     hidden, up);
            else
                expert_hidden(xt, c->W1 + e * c->d * c->h, c->d, c->h, hidden);
            expert_down(hidden, c->W2 + e * c->h * c->d, c->h, c->d, o);
            for (int64_t col = 0; col < c->d; ++col) yt[col] += g[j] * o[col];
        }
        if (c->hs > 0) {                                                                    /* Eq. 6, shared */
            if (c->Ws3) expert_hidden_swiglu(xt, c->Ws1, c->Ws3, c->d, c->hs, hidden, up);
            else expert_hidden(xt, c->Ws1, c->d, c->hs, hidden);
            expert_down(hidden, c->Ws2, c->hs, c->d, o);
            for (int64_t col = 0; col < c->d; ++col) yt[col] += c->lambda * o[col];
            if (c->shared_out)
                for (int64_t col = 0; col < c->d; ++col) c->shared_out[i * c->d + col] = o[col];
        }
        if (c->idx) for (int64_t j = 0; j < c->k; ++j) c->idx[i * c->k + j] = sel[j];
        if (c->gate) for (int64_t j = 0; j < c->k; ++j) c->gate[i * c->k + j] = g[j];
        if (c->margin) c->margin[i] = m;
    }
done:
    free(s); free(key); free(taken); free(hidden); free(up); free(o); free(sel); free(g);
}

/* y[i, :] for token tokens[i] (tokens may be NULL: all T tokens in order).
 * W3 NULL: GELU experts GELU(x W1[e]) W2[e]; else SwiGLU experts
 * (SiLU(x W1[e]) * (x W3[e])) W2[e], W3 bf16 [E, d, h].
 * hs == 0 means no shared expert (Ws1, Ws2, Ws3 ignored); Ws3 NULL: a GELU shared
 * expert, else a SwiGLU one (SiLU(x Ws1) * (x Ws3)) Ws2, Ws3 bf16 [d, hs].
 * idx, gate, margin and shared_out ([ntok, d], the un-weighted shared expert
 * output) may be NULL. */
int oracle_forward_tokens(const uint16_t* x, const float* Wr, const float* b,
                          const uint16_t* W1, const uint16_t* W2, const uint16_t* W3,
                          const uint16_t* Ws1, const uint16_t* Ws2, const uint16_t* Ws3, double lambda,
                          int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t hs,
                          const int32_t* tokens, int64_t ntok,
                          double* y, int32_t* idx, double* gate, double* margin,
                          double* shared_out, int nthreads) {
    if (T < 0 || d <= 0 || E <= 0 || k < 1 || k > E || h <= 0 || hs < 0 || ntok < 0) return ORACLE_ERR_ARG;
    if (ntok > 0 && (!x || !Wr || !b || !W1 || !W2 || !y)) return ORACLE_ERR_ARG;
    if (hs > 0 && ntok > 0 && (!Ws1 || !Ws2)) return ORACLE_ERR_ARG;
    fwd_ctx c = { x, Wr, b, W1, W2, W3, Ws1, Ws2, Ws3, lambda, T, d, E, k, h, hs,
                  tokens, y, idx, gate, margin, shared_out, ORACLE_OK };
    parallel_for(ntok, nthreads, fwd_items, &c);
    return c.err;
}

/* ------------------------------------------------------- bias update */

/* Loss-free balancing bias update from one step's expert loads (Sec. 2.2.2):
 * t_e = counts[e] (tokens routed to expert e), mu = their mean, sigma their
 * (population) standard deviation over the E experts.
 *   rule 0, z-score (Eq. 9):  b_e <- b_e - alpha (t_e - mu) / sigma
 *                             (sigma == 0, all loads equal: b unchanged)
 *   rule 1, sign (Eq. 8):     b_e <- b_e - alpha sign(t_e - mu), sign(0) = 0
 * mu = (sum of t_e, an exact integer) / E; sigma = sqrt(sum_e (t_e - mu)^2 / E),
 * summed in ascending e; each new b_e is computed in double and rounded to float. */
int oracle_update_bias(const int32_t* counts, int64_t E, float alpha, int rule, float* b) {
    if (E <= 0 || !counts || !b || (rule != 0 && rule != 1)) return ORACLE_ERR_ARG;
    int64_t sum = 0;
    for (int64_t e = 0; e < E; ++e) {
        if (counts[e] < 0) return ORACLE_ERR_ARG;
        sum += counts[e];
    }
    const double mu = (double)sum / (double)E;
    double ss = 0.0;
    for (int64_t e = 0; e < E; ++e) {
        const double dev = (double)counts[e] - mu;
        ss += dev * dev;
    }
    const double sigma = sqrt(ss / (double)E);
    for (int64_t e = 0; e < E; ++e) {
        const double dev = (double)counts[e] - mu;
        double step;
        if (rule == 0) {
            if (sigma == 0.0) continue;
            step = dev / sigma;
        } else {
            step = (double)((dev > 0.0) - (dev < 0.0));
        }
        b[e] = (float)((double)b[e] - (double)alpha * step);
    }
    return ORACLE_OK;
}

/* ------------------------------------------- backward of the layer (training) */

/* The training path of the layer (App. B: grouped GEMMs for training, the activation
 * a separate operator between the up- and down-projections): the gradients of
 * L = sum_t dy[t] . y[t] with respect to the inputs and weights, given dy[T, d].
 *
 * Readings (listed in the design notes):
 *   - the top-k selection is held fixed: it is piecewise constant in s, so it has no
 *     gradient; the gradient reaches W_r and x through the gates of Eqs. 4-5 only;
 *   - the bias b gets no gradient (it only selects; Sec. 2.2.2 updates it from the
 *     expert loads, Eqs. 8-9, not by back-propagation).
 *
 * Per token t with selected experts e_j, sigma_j = Sigmoid(s_{e_j}), S = sum_j sigma_j,
 * gates g_j = sigma_j / S, expert outputs o_j = E_{e_j}(x_t):
 *   dg_j      = dy . o_j
 *   dsigma_j  = (dg_j - sum_l g_l dg_l) / S            (derivative of sigma_j / S)
 *   ds_{e_j}  = dsigma_j sigma_j (1 - sigma_j)           (Sigmoid' = sigma (1 - sigma))
 *   dW_r[:, e_j] += x_t ds_{e_j},   dx_t += ds_{e_j} W_r[:, e_j]
 * and through each selected expert with output weight g_j (and the shared expert
 * with weight lambda), with a the hidden activation, u = x W1[e] (and v = x W3[e]):
 *   dW2[e] += a^T (g dy),  da = (g dy) W2[e]^T,
 *   GELU:   du = da GELU'(u),  GELU'(u) = Phi(u) + u phi(u)
 *   SwiGLU: du = da v SiLU'(u), dv = da SiLU(u),  SiLU'(u) = sigma(u) (1 + u (1 - sigma(u)))
 *   dW1[e] += x^T du,  dW3[e] += x^T dv,  dx += du W1[e]^T + dv W3[e]^T.
 * Tokens are taken one after another in ascending t (one thread: the weight
 * gradients are sums over tokens, accumulated in that order).  A token whose dy row
 * is all zero adds exact zeros to every gradient -- every term it contributes is a
 * product with an element of dy_t -- as long as the other factor is finite, which
 * holds when its input row x_t and every weight of the layer are finite; such a token
 * is skipped, so a sampled check (dy nonzero on a few tokens) costs only those tokens.
 * With a non-finite x_t or weight it is not skipped, so 0 * inf gives NaN exactly as
 * the unskipped sum does.  All outputs are
 * double and are overwritten: dx [T, d], dWr [d, E], dW1 [E, d, h], dW2 [E, h, d],
 * dW3 [E, d, h] (with W3), dWs1 [d, hs], dWs2 [hs, d], dWs3 [d, hs] (with Ws3). */

static double gelu_grad(double u) {
    const double Phi = 0.5 * (1.0 + erf(u / sqrt(2.0)));
    const double phi = exp(-0.5 * u * u) / sqrt(2.0 * 3.14159265358979323846);
    return Phi + u * phi;
}

/* One expert (or the shared expert) on one token: forward to its output o, then
 * the gradient pieces for the output weight w (g_j or lambda).  W3 NULL: GELU. */
static void expert_backward(const uint16_t* xt, const uint16_t* W1e, const uint16_t* W3e,
                            const uint16_t* W2e, int64_t d, int64_t h, double w, const double* dyt,
                            double* dW1e, double* dW3e, double* dW2e, double* dxt, double* o,
                            double* u, double* v, double* a, double* da) {
    for (int64_t n = 0; n < h; ++n) { u[n] = 0.0; v[n] = 0.0; }
    for (int64_t i = 0; i < d; ++i) {
        const double xi = bf16_to_double(xt[i]);
        for (int64_t n = 0; n < h; ++n) {
            u[n] += xi * bf16_to_double(W1e[i * h + n]);
            if (W3e) v[n] += xi * bf16_to_double(W3e[i * h + n]);
        }
    }
    for (int64_t n = 0; n < h; ++n) a[n] = W3e ? silu(u[n]) * v[n] : gelu(u[n]);
    expert_down(a, W2e, h, d, o);
    /* dW2[e] += a^T (w dy);  da = (w dy) W2[e]^T */
    for (int64_t n = 0; n < h; ++n) {
        double acc = 0.0;
        for (int64_t c = 0; c < d; ++c) {
            const double dO = w * dyt[c];
            dW2e[n * d + c] += a[n] * dO;
            acc += dO * bf16_to_double(W2e[n * d + c]);
        }
        da[n] = acc;
    }
    /* du (in u), dv (in v) */
    for (int64_t n = 0; n < h; ++n) {
        if (W3e) {
            const double sg = sigmoid(u[n]);
            const double du = da[n] * v[n] * sg * (1.0 + u[n] * (1.0 - sg));
            const double dv = da[n] * u[n] * sg;   /* SiLU(u) = u sigma(u) */
            u[n] = du;
            v[n] = dv;
        } else {
            u[n] = da[n] * gelu_grad(u[n]);
        }
    }
    for (int64_t i = 0; i < d; ++i) {
        const double xi = bf16_to_double(xt[i]);
        double acc = 0.0;
        for (int64_t n = 0; n < h; ++n) {
            dW1e[i * h + n] += xi * u[n];
            acc += u[n] * bf16_to_double(W1e[i * h + n]);
            if (W3e) {
                dW3e[i * h + n] += xi * v[n];
                acc += v[n] * bf16_to_double(W3e[i * h + n]);
            }
        }
        dxt[i] += acc;
    }
}

/* 1 when every value of the n bf16 values v is finite (exponent field not all ones). */
static int bf16_all_finite(const uint16_t* v, int64_t n) {
    for (int64_t i = 0; i < n; ++i)
        if ((v[i] & 0x7f80u) == 0x7f80u) return 0;
    return 1;
}

static int f32_all_finite(const float* v, int64_t n) {
    for (int64_t i = 0; i < n; ++i)
        if (!isfinite(v[i])) return 0;
    return 1;
}

int oracle_backward(const uint16_t* x, const float* Wr, const float* b,
                    const uint16_t* W1, const uint16_t* W2, const uint16_t* W3,
                    const uint16_t* Ws1, const uint16_t* Ws2, const uint16_t* Ws3, double lambda,
                    int64_t T, int64_t d, int64_t E, int64_t k, int64_t h, int64_t hs,
                    const double* dy, double* dx, double* dWr, double* dW1, double* dW2,
                    double* dW3, double* dWs1, double* dWs2, double* dWs3) {
    if (T < 0 || d <= 0 || E <= 0 || k < 1 || k > E || h <= 0 || hs < 0) return ORACLE_ERR_ARG;
    if (!x || !Wr || !b || !W1 || !W2 || !dy || !dx || !dWr || !dW1 || !dW2) return ORACLE_ERR_ARG;
    if (W3 && !dW3) return ORACLE_ERR_ARG;
    if (hs > 0 && (!Ws1 || !Ws2 || !dWs1 || !dWs2 || (Ws3 && !dWs3))) return ORACLE_ERR_ARG;
    memset(dx, 0, (size_t)(T * d) * sizeof(double));
    memset(dWr, 0, (size_t)(d * E) * sizeof(double));
    memset(dW1, 0, (size_t)(E * d * h) * sizeof(double));
    memset(dW2, 0, (size_t)(E * h * d) * sizeof(double));
    if (W3) memset(dW3, 0, (size_t)(E * d * h) * sizeof(double));
    if (hs > 0) {
        memset(dWs1, 0, (size_t)(d * hs) * sizeof(double));
        memset(dWs2, 0, (size_t)(hs * d) * sizeof(double));
        if (Ws3) memset(dWs3, 0, (size_t)(d * hs) * sizeof(double));
    }
    const int64_t hmax = h > hs ? h : hs;
    double* s = (double*)malloc((size_t)E * sizeof(double));
    double* key = (double*)malloc((size_t)E * sizeof(double));
    unsigned char* taken = (unsigned char*)malloc((size_t)E);
    int32_t* sel = (int32_t*)malloc((size_t)k * sizeof(int32_t));
    double* g = (double*)malloc((size_t)k * sizeof(double));
    double* dg = (double*)malloc((size_t)k * sizeof(double));
    double* o = (double*)malloc((size_t)d * sizeof(double));
    double* u = (double*)malloc((size_t)hmax * sizeof(double));
    double* v = (double*)malloc((size_t)hmax * sizeof(double));
    double* a = (double*)malloc((size_t)hmax * sizeof(double));
    double* da = (double*)malloc((size_t)hmax * sizeof(double));
    int err = ORACLE_OK;
    if (!s || !key || !taken || !sel || !g || !dg || !o || !u || !v || !a || !da) {
        err = ORACLE_ERR_NOMEM;
        goto done;
    }
    /* zero-cotangent tokens may be skipped only when the factors they multiply are finite */
    const int weights_finite =
        f32_all_finite(Wr, d * E) && f32_all_finite(b, E) && bf16_all_finite(W1, E * d * h) &&
        bf16_all_finite(W2, E * h * d) && (!W3 || bf16_all_finite(W3, E * d * h)) &&
        (hs == 0 || (bf16_all_finite(Ws1, d * hs) && bf16_all_finite(Ws2, hs * d) &&
                     (!Ws3 || bf16_all_finite(Ws3, d * hs))));
    for (int64_t t = 0; t < T; ++t) {
        const uint16_t* xt = x + t * d;
        const double* dyt = dy + t * d;
        double* dxt = dx + t * d;
        int64_t nz = 0;
        while (nz < d && dyt[nz] == 0.0) ++nz;
        if (nz == d && weights_finite && bf16_all_finite(xt, d)) continue;   /* dy_t = 0: adds zeros */
        logits_row(xt, Wr, d, E, s);                                                        /* Eq. 1 */
        double m;
        select_one(s, b, E, k, sel, g, &m, taken, key);                                    /* Eqs. 7, 4, 5 */
        for (int64_t j = 0; j < k; ++j) {                                                   /* routed experts */
            const int64_t e = sel[j];
            expert_backward(xt, W1 + e * d * h, W3 ? W3 + e * d * h : NULL, W2 + e * h * d, d, h, g[j],
                            dyt, dW1 + e * d * h, W3 ? dW3 + e * d * h : NULL, dW2 + e * h * d, dxt,
                            o, u, v, a, da);
            double acc = 0.0;
            for (int64_t c = 0; c < d; ++c) acc += dyt[c] * o[c];
            dg[j] = acc;                                                                    /* dy . o_j */
        }
        double S = 0.0, gdg = 0.0;                                                          /* Eqs. 4-5 */
        for (int64_t j = 0; j < k; ++j) S += sigmoid(s[sel[j]]);
        for (int64_t j = 0; j < k; ++j) gdg += g[j] * dg[j];
        for (int64_t j = 0; j < k; ++j) {
            const int64_t e = sel[j];
            const double sg = sigmoid(s[e]);
            const double ds = (dg[j] - gdg) / S * sg * (1.0 - sg);
            for (int64_t i = 0; i < d; ++i) {
                dWr[i * E + e] += bf16_to_double(xt[i]) * ds;
                dxt[i] += ds * (double)Wr[i * E + e];
            }
        }
        if (hs > 0)                                                                         /* Eq. 6, shared */
            expert_backward(xt, Ws1, Ws3, Ws2, d, hs, lambda, dyt, dWs1, Ws3 ? dWs3 : NULL, dWs2, dxt,
                            o, u, v, a, da);
    }
done:
    free(s); free(key); free(taken); free(sel); free(g); free(dg); free(o); free(u); free(v);
    free(a); free(da);
    return err;
}

/* Staged backward of the routed experts, row by row in expert-major order (the rows of
 * Algorithm 1): for row r of expert e (the segment holding r), token t = perm[r] / k and
 * its gate g = gate_rows[r] (the gate of slot perm[r]):
 *   du[i, :] = (g dy[t] W2[e]^T) * GELU'(u)      (GELU experts), or for SwiGLU experts
 *   du[i, :] = (g dy[t] W2[e]^T) * v * SiLU'(u),  dv[i, :] = (g dy[t] W2[e]^T) * SiLU(u)
 *   dg[i]    = dy[t] . E_e(x_t)                    (the un-gated expert output)
 * with u = x_t W1[e], v = x_t W3[e], for r = rows[i].  These are the intermediate
 * gradients from which dW1 = sum x^T du, dW3 = sum x^T dv, dx and the gate gradients
 * of oracle_backward are formed.  du, dv: double [nrows, h] (dv only with W3); dg:
 * double [nrows]. */
int oracle_backward_rows(const uint16_t* x, const int32_t* perm, const int32_t* offsets,
                         const double* gate_rows, const uint16_t* W1, const uint16_t* W2,
                         const uint16_t* W3, const double* dy, int64_t T, int64_t d, int64_t h,
                         int64_t E, int64_t k, const int32_t* rows, int64_t nrows,
                         double* du, double* dv, double* dg) {
    if (T < 0 || d <= 0 || h <= 0 || E <= 0 || k < 1 || nrows < 0) return ORACLE_ERR_ARG;
    if (nrows > 0 && (!x || !perm || !offsets || !gate_rows || !W1 || !W2 || !dy || !rows || !du ||
                      !dg || (W3 && !dv)))
        return ORACLE_ERR_ARG;
    double* u = (double*)malloc((size_t)h * sizeof(double));
    double* v = (double*)malloc((size_t)h * sizeof(double));
    double* a = (double*)malloc((size_t)h * sizeof(double));
    double* da = (double*)malloc((size_t)h * sizeof(double));
    double* o = (double*)malloc((size_t)d * sizeof(double));
    int err = ORACLE_OK;
    if (!u || !v || !a || !da || !o) { err = ORACLE_ERR_NOMEM; goto done; }
    for (int64_t i = 0; i < nrows; ++i) {
        const int64_t r = rows[i];
        const int64_t e = expert_of_row(offsets, E, r);
        const int64_t t = (e < 0) ? -1 : perm[r] / k;
        if (e < 0 || t < 0 || t >= T) { err = ORACLE_ERR_ARG; continue; }
        const uint16_t* xt = x + t * d;
        const uint16_t* W1e = W1 + e * d * h;
        const uint16_t* W3e = W3 ? W3 + e * d * h : NULL;
        const uint16_t* W2e = W2 + e * h * d;
        for (int64_t n = 0; n < h; ++n) { u[n] = 0.0; v[n] = 0.0; }
        for (int64_t c = 0; c < d; ++c) {
            const double xc = bf16_to_double(xt[c]);
            for (int64_t n = 0; n < h; ++n) {
                u[n] += xc * bf16_to_double(W1e[c * h + n]);
                if (W3e) v[n] += xc * bf16_to_double(W3e[c * h + n]);
            }
        }
        for (int64_t n = 0; n < h; ++n) a[n] = W3e ? silu(u[n]) * v[n] : gelu(u[n]);
        expert_down(a, W2e, h, d, o);
        double acc = 0.0;
        for (int64_t c = 0; c < d; ++c) acc += dy[t * d + c] * o[c];
        dg[i] = acc;
        for (int64_t n = 0; n < h; ++n) {
            double s = 0.0;
            for (int64_t c = 0; c < d; ++c) s += gate_rows[r] * dy[t * d + c] * bf16_to_double(W2e[n * d + c]);
            da[n] = s;
        }
        for (int64_t n = 0; n < h; ++n) {
            if (W3e) {
                const double sg = sigmoid(u[n]);
                du[i * h + n] = da[n] * v[n] * sg * (1.0 + u[n] * (1.0 - sg));
                dv[i * h + n] = da[n] * u[n] * sg;
            } else {
                du[i * h + n] = da[n] * gelu_grad(u[n]);
            }
        }
    }
done:
    free(u); free(v); free(a); free(da); free(o);
    return err;
}
