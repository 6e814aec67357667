/*
 * pmpe_oracle.c -- plain CPU oracle for the policy-masked sparse-MoE layer
 * forward of "Policy-Masked Private Experts" (arXiv 2608.06690).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously-correct
 * definition that the GPU path is checked against.  Only the test suite,
 * the smoke check and the benchmark's CPU-baseline leg may load it.  It
 * shares no code, header, table or helper with the CUDA library; the two
 * only meet in the seeded input generator, which holds none of the method's
 * arithmetic.
 *
 * Arithmetic: every dot product accumulates in double (fp64) from the BF16
 * operands.  Three rounding points are part of the reading of the method, not
 * of any kernel:
 *   - router logits are rounded to fp32 before the top-k decision (the
 *     routing decision is taken on fp32 logits on both sides);
 *   - the SwiGLU activation silu(g)*u is rounded to BF16, because it is the
 *     BF16 operand of the down projection in a BF16 model;
 *   - the layer output is rounded once to BF16 (round to nearest even).
 * Everything else (g, u, y, the weighted sum) stays in double.
 *
 * Parity status: the values are pinned by closed forms, special cases that
 * reduce to a textbook SwiGLU MLP / softmax / sort, brute force on tiny
 * inputs and the audit invariants of Sec. 2.2 (Eq. 1, G1).  The paper prints
 * no worked numeric example of the layer, so no printed value pins it; the
 * hand-worked fixtures under tests/golden/ are derived from the definitions.
 *
 * Method passages followed (paper sections / equations):
 *   - Sec. 2.1 (threat model) and App. B.1 (policy resolution): missing,
 *     malformed or non-Boolean authorisation resolves to tau = 0.  As a byte
 *     per token: only 0x01 is ALLOW; NULL means every token is DENY.
 *   - Sec. 3.1, Eq. 4 (the mask m_{l,e}(tau)) and the sentence after it: top-k
 *     is taken over z_l(h) + m_l(tau), m = 0 on the eligible pool and -inf on
 *     the other one; public ids 0..E_pub-1, private ids E_pub..E_pub+E_priv-1
 *     (the concatenated public/private pool of Sec. 4.2).
 *   - App. B.1 fail-closed procedure, steps 2, 4, 5: resolve, mask then
 *     top-k, record the route.
 *   - Sec. 3.1 / Sec. 4.2: private experts copy the public expert
 *     architecture (gate, up, down projections: a SwiGLU MLP).
 *   - Sec. 5.2 / App. F.1: independent execution counts observed at the
 *     expert modules themselves, separate from the route log.
 *   - Sec. 4.2 (matched adaptation and controls) and App. E (the complete
 *     Qwen control matrix), the soft-router-only arm: routing over the concatenated public/private pool
 *     without the hard mask.  With `unmasked` set, m(tau) = 0 for every
 *     expert; this is a negative control, not the method (G1 does not hold).
 *   - Sec. 2.2 (G2) and Sec. 3.2 (training of the private branch): the two
 *     backward functions -- the gradients of the private parameters, and the
 *     gradient of the layer's input that the layer below needs -- by the chain
 *     rule through the forward as computed (rounding points as the identity;
 *     `exact` drops them so that finite differences can pin the functions).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

typedef struct {
    int T, H, I, E_pub, E_priv, E_sh, k;
    int renormalize;                 /* 1: softmax renormalised over the top-k; 0: pool softmax probs */
    const uint16_t *hidden;          /* [T][H] BF16 bits */
    const uint8_t *policy;           /* [T] bytes, or NULL */
    const uint16_t *router_pub;      /* [E_pub][H] */
    const uint16_t *router_priv;     /* [E_priv][H] */
    const uint16_t *gate_pub, *up_pub, *down_pub;     /* [E_pub][I][H], [E_pub][I][H], [E_pub][H][I] */
    const uint16_t *gate_priv, *up_priv, *down_priv;  /* [E_priv][I][H], ..., [E_priv][H][I] */
    const uint16_t *gate_sh, *up_sh, *down_sh;        /* [E_sh][I][H], ..., [E_sh][H][I]; NULL if E_sh == 0 */
    int unmasked;                    /* 1: the soft-router control, no hard mask (all E experts eligible) */
    int exact;                       /* 1: no rounding of logits (fp32) or activations (BF16): the smooth
                                        function that finite-difference pins of the backward differentiate */
} oracle_layer;

/* ---------------------------------------------------------------- BF16 -- */

static double bf16_value(uint16_t b)
{
    uint32_t u = (uint32_t)b << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Round a double to the nearest BF16 value, ties to even.  BF16 keeps
 * 8 significant bits; for |x| in [2^(e-1), 2^e) the spacing is 2^(e-8),
 * and below the smallest normal (2^-126) it is 2^-133. */
uint16_t oracle_bf16_round(double x)
{
    if (isnan(x)) return 0x7FC0;
    uint16_t sign = signbit(x) ? 0x8000 : 0;
    double a = fabs(x);
    if (a == 0.0) return sign;
    if (isinf(a)) return sign | 0x7F80;
    int e;
    frexp(a, &e);                     /* a = m * 2^e with m in [0.5, 1) */
    int q_exp = (e - 1 < -126) ? -133 : e - 8;
    double q = nearbyint(ldexp(a, -q_exp));   /* default mode: ties to even */
    double r = ldexp(q, q_exp);
    if (r > 0x1.FEp127) return sign | 0x7F80; /* beyond the largest finite BF16 */
    float f = (float)r;               /* exact: r is a BF16 value */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return sign | (uint16_t)(u >> 16);
}

double oracle_bf16_value(uint16_t b) { return bf16_value(b); }

/* ------------------------------------------------------ policy resolve -- */

/* tau_t = 1 only for the trusted byte 0x01; NULL policy -> all 0. */
void oracle_resolve(const uint8_t *policy, int T, uint8_t *tau)
{
    for (int t = 0; t < T; ++t)
        tau[t] = (policy != NULL && policy[t] == 0x01) ? 1 : 0;
}

/* Per-request policy (one trusted byte per request, requests given by the
 * cumulative token offsets cu[0..n]) expanded to one byte per token.  Any
 * malformed offset list (cu[0] != 0, a decreasing step, or cu[n] > T) is
 * malformed metadata: every token becomes DENY (0x00).  Tokens after cu[n]
 * belong to no request and are DENY.  Sec. 2.1 / App. B.1: missing or
 * malformed authorisation resolves to DENY. */
void oracle_policy_from_requests(const uint8_t *req_policy, const int32_t *cu, int n, int T, uint8_t *out)
{
    int valid = (n >= 0 && cu != NULL && (n == 0 || req_policy != NULL) && cu[0] == 0 && cu[n] <= T);
    for (int r = 0; valid && r < n; ++r)
        if (cu[r + 1] < cu[r]) valid = 0;
    for (int t = 0; t < T; ++t) out[t] = 0x00;
    if (!valid) return;
    for (int r = 0; r < n; ++r)
        for (int t = cu[r]; t < cu[r + 1]; ++t) out[t] = req_policy[r];
}

/* ------------------------------------------------------------- routing -- */

/* The row of the concatenated router for global expert id e. */
static const uint16_t *router_row(const oracle_layer *L, int e)
{
    return e < L->E_pub ? L->router_pub + (size_t)e * L->H
                        : L->router_priv + (size_t)(e - L->E_pub) * L->H;
}

/* The masked logits of one token: s_e = z_e + m_e(tau), with z_e = h . W_e
 * accumulated in double and rounded to fp32 (the routing decision is taken on
 * fp32 logits), m = 0 on the pool tau selects and -inf on the other pool
 * (Sec. 3.1 Eq. 4).  In the unmasked control m = 0 for every expert. */
static void masked_logits(const oracle_layer *L, int t, double *s /* [E] */)
{
    const int E = L->E_pub + L->E_priv;
    const int tau = (L->policy != NULL && L->policy[t] == 0x01);
    const uint16_t *h = L->hidden + (size_t)t * L->H;
    for (int e = 0; e < E; ++e) {
        const uint16_t *wr = router_row(L, e);
        double z = 0.0;
        for (int c = 0; c < L->H; ++c) z += bf16_value(h[c]) * bf16_value(wr[c]);
        const int eligible = L->unmasked ? 1 : (tau ? (e >= L->E_pub) : (e < L->E_pub));
        s[e] = eligible ? (L->exact ? z : (double)(float)z) : -INFINITY;   /* z + m(tau), z rounded to fp32 */
    }
}

/* Routing weights of the selected ids idx[k] from the masked logits s: the
 * softmax over the visible pool (shifted by its largest logit; exp(-inf) = 0
 * drops the other pool), then, for the renormalised variant, divided by
 * their sum over the selection. */
static void route_weights(const oracle_layer *L, const double *s, const int32_t *idx, double *w)
{
    const int E = L->E_pub + L->E_priv;
    double smax = -INFINITY;
    for (int e = 0; e < E; ++e) smax = s[e] > smax ? s[e] : smax;
    double denom_pool = 0.0;
    for (int e = 0; e < E; ++e) denom_pool += exp(s[e] - smax);
    double sel = 0.0;
    for (int j = 0; j < L->k; ++j) {
        w[j] = exp(s[idx[j]] - smax) / denom_pool;     /* p_e of the pool softmax */
        sel += w[j];
    }
    if (L->renormalize)
        for (int j = 0; j < L->k; ++j) w[j] /= sel;     /* renormalise over the top-k */
}

/* Route one token: s = z + m(tau), top-k of s (descending, ties to the lower
 * id), weights from the softmax of s.  In the unmasked control m = 0, so the
 * top-k and the softmax run over all E.  Writes idx[k], w[k], and the gap
 * s_(k) - s_(k+1) inside the visible pool (+inf when k equals the pool size). */
static void route_token(const oracle_layer *L, int t, int32_t *idx, double *w, double *gap,
                        double *s /* scratch [E] */, char *taken /* scratch [E] */)
{
    const int E = L->E_pub + L->E_priv;
    masked_logits(L, t, s);
    for (int e = 0; e < E; ++e) taken[e] = 0;
    /* top-k by repeated selection: largest s, lower id on ties */
    for (int j = 0; j < L->k; ++j) {
        int best = -1;
        for (int e = 0; e < E; ++e) {
            if (taken[e] || s[e] == -INFINITY) continue;
            if (best < 0 || s[e] > s[best]) best = e;
        }
        idx[j] = best;
        taken[best] = 1;
    }
    /* (k+1)-th best in the visible pool, for the gap rule */
    int next = -1;
    for (int e = 0; e < E; ++e) {
        if (taken[e] || s[e] == -INFINITY) continue;
        if (next < 0 || s[e] > s[next]) next = e;
    }
    *gap = next < 0 ? INFINITY : s[idx[L->k - 1]] - s[next];
    route_weights(L, s, idx, w);
}

/* ------------------------------------------------------------- experts -- */

/* One SwiGLU expert on one token: g = Wg h, u = Wu h, a = bf16(silu(g) u),
 * y = Wd a.  Wg, Wu: [I][H]; Wd: [H][I].  Every call adds one row to
 * *exec_counter: the execution count is observed here, where the expert
 * runs, not copied from the route log. */
static void swiglu_expert(const uint16_t *Wg, const uint16_t *Wu, const uint16_t *Wd, int H, int I,
                          const double *h, double *y, double *a, uint32_t *exec_counter, int exact)
{
    for (int i = 0; i < I; ++i) {
        const uint16_t *rg = Wg + (size_t)i * H, *ru = Wu + (size_t)i * H;
        double g = 0.0, u = 0.0;
        for (int c = 0; c < H; ++c) {
            g += h[c] * bf16_value(rg[c]);
            u += h[c] * bf16_value(ru[c]);
        }
        const double silu = g / (1.0 + exp(-g));
        a[i] = exact ? silu * u : bf16_value(oracle_bf16_round(silu * u));
    }
    for (int o = 0; o < H; ++o) {
        const uint16_t *rd = Wd + (size_t)o * I;
        double acc = 0.0;
        for (int i = 0; i < I; ++i) acc += a[i] * bf16_value(rd[i]);
        y[o] = acc;
    }
    *exec_counter += 1;
}

static void routed_expert_weights(const oracle_layer *L, int e, const uint16_t **g, const uint16_t **u,
                                  const uint16_t **d)
{
    const size_t ih = (size_t)L->I * L->H;
    if (e < L->E_pub) {
        *g = L->gate_pub + e * ih; *u = L->up_pub + e * ih; *d = L->down_pub + e * ih;
    } else {
        const int p = e - L->E_pub;
        *g = L->gate_priv + p * ih; *u = L->up_priv + p * ih; *d = L->down_priv + p * ih;
    }
}

/* ---------------------------------------------------------- public API -- */

static int check_layer(const oracle_layer *L)
{
    if (!L || L->T < 0 || L->H <= 0 || L->I <= 0 || L->E_pub < 0 || L->E_priv < 0 || L->E_sh < 0) return -1;
    if (L->k < 1 || L->k > L->E_pub || L->k > L->E_priv) return -1;
    if (L->T > 0 && !L->hidden) return -1;
    if (!L->router_pub || !L->router_priv) return -1;
    return 0;
}

/* Routing only, for the tokens in `tokens` (NULL = all T).  Outputs are
 * indexed by position in the list. */
int oracle_route(const oracle_layer *L, const int32_t *tokens, int n, int32_t *idx, double *w, double *gap,
                 int nthreads)
{
    if (check_layer(L)) return -1;
    const int E = L->E_pub + L->E_priv;
    if (!tokens) n = L->T;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel
    {
        double *s = (double *)malloc(sizeof(double) * E);
        char *taken = (char *)malloc(E);
#pragma omp for schedule(dynamic, 4)
        for (int p = 0; p < n; ++p) {
            const int t = tokens ? tokens[p] : p;
            route_token(L, t, idx + (size_t)p * L->k, w + (size_t)p * L->k, gap + p, s, taken);
        }
        free(s);
        free(taken);
    }
    return 0;
}

/* One routed expert (global id e) or, with shared = 1, shared expert e, on a
 * single BF16 hidden row.  y: [H] doubles. */
int oracle_expert(const oracle_layer *L, int e, int shared, const uint16_t *h_row, double *y)
{
    if (!L || !h_row || !y) return -1;
    const uint16_t *g, *u, *d;
    if (shared) {
        if (e < 0 || e >= L->E_sh) return -1;
        const size_t ih = (size_t)L->I * L->H;
        g = L->gate_sh + e * ih; u = L->up_sh + e * ih; d = L->down_sh + e * ih;
    } else {
        if (e < 0 || e >= L->E_pub + L->E_priv) return -1;
        routed_expert_weights(L, e, &g, &u, &d);
    }
    double *h = (double *)malloc(sizeof(double) * L->H);
    double *a = (double *)malloc(sizeof(double) * L->I);
    for (int c = 0; c < L->H; ++c) h[c] = bf16_value(h_row[c]);
    uint32_t dummy = 0;
    swiglu_expert(g, u, d, L->H, L->I, h, y, a, &dummy, L->exact);
    free(h);
    free(a);
    return 0;
}

/* Full layer forward for the tokens in `tokens` (NULL = all T).
 *   out_bf16 [n][H], out_f64 [n][H] (may be NULL), idx [n][k], w [n][k], gap [n]
 *   route_count [E], route_priv_rows [n]      -- the route log
 *   exec_rows [E], exec_priv_rows [n]         -- counted where the experts run
 *   shared_rows [1]                           -- shared-expert executions
 * Counters are overwritten (not accumulated). */
int oracle_forward(const oracle_layer *L, const int32_t *tokens, int n, uint16_t *out_bf16, double *out_f64,
                   int32_t *idx, double *w, double *gap, uint32_t *route_count, uint32_t *route_priv_rows,
                   uint32_t *exec_rows, uint32_t *exec_priv_rows, uint32_t *shared_rows, int nthreads)
{
    if (check_layer(L)) return -1;
    if (L->E_sh > 0 && (!L->gate_sh || !L->up_sh || !L->down_sh)) return -1;
    const int E = L->E_pub + L->E_priv, H = L->H, I = L->I, k = L->k;
    if (!tokens) n = L->T;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
    const int nt = omp_get_max_threads();
#else
    (void)nthreads;
    const int nt = 1;
#endif
    /* per-thread execution counters, reduced in a fixed order afterwards */
    uint32_t *exec_local = (uint32_t *)calloc((size_t)nt * (E + 1), sizeof(uint32_t));
    uint32_t *exec_priv_local = (uint32_t *)calloc((size_t)n > 0 ? (size_t)n : 1, sizeof(uint32_t));

#pragma omp parallel
    {
#ifdef _OPENMP
        const int tid = omp_get_thread_num();
#else
        const int tid = 0;
#endif
        uint32_t *my_exec = exec_local + (size_t)tid * (E + 1);
        double *s = (double *)malloc(sizeof(double) * E);
        char *taken = (char *)malloc(E);
        double *h = (double *)malloc(sizeof(double) * H);
        double *y = (double *)malloc(sizeof(double) * H);
        double *acc = (double *)malloc(sizeof(double) * H);
        double *a = (double *)malloc(sizeof(double) * I);
#pragma omp for schedule(dynamic, 1)
        for (int p = 0; p < n; ++p) {
            const int t = tokens ? tokens[p] : p;
            int32_t *ti = idx + (size_t)p * k;
            double *tw = w + (size_t)p * k;
            route_token(L, t, ti, tw, gap + p, s, taken);

            const uint16_t *hr = L->hidden + (size_t)t * H;
            for (int c = 0; c < H; ++c) { h[c] = bf16_value(hr[c]); acc[c] = 0.0; }
            for (int j = 0; j < k; ++j) {
                const int e = ti[j];
                const uint16_t *g, *u, *d;
                routed_expert_weights(L, e, &g, &u, &d);
                uint32_t before = my_exec[e];
                swiglu_expert(g, u, d, H, I, h, y, a, &my_exec[e], L->exact);
                if (e >= L->E_pub) exec_priv_local[p] += my_exec[e] - before;
                for (int c = 0; c < H; ++c) acc[c] += tw[j] * y[c];
            }
            const size_t ih = (size_t)I * H;
            for (int sidx = 0; sidx < L->E_sh; ++sidx) {
                swiglu_expert(L->gate_sh + sidx * ih, L->up_sh + sidx * ih, L->down_sh + sidx * ih, H, I, h, y, a,
                              &my_exec[E], L->exact);
                for (int c = 0; c < H; ++c) acc[c] += y[c];
            }
            for (int c = 0; c < H; ++c) {
                out_bf16[(size_t)p * H + c] = oracle_bf16_round(acc[c]);
                if (out_f64) out_f64[(size_t)p * H + c] = acc[c];
            }
        }
        free(s); free(taken); free(h); free(y); free(acc); free(a);
    }

    /* route log, from the routing decisions */
    for (int e = 0; e < E; ++e) route_count[e] = 0;
    for (int p = 0; p < n; ++p) {
        route_priv_rows[p] = 0;
        for (int j = 0; j < k; ++j) {
            const int e = idx[(size_t)p * k + j];
            route_count[e] += 1;
            if (e >= L->E_pub) route_priv_rows[p] += 1;
        }
    }
    /* execution log, from the expert calls */
    for (int e = 0; e < E; ++e) exec_rows[e] = 0;
    *shared_rows = 0;
    for (int tid = 0; tid < nt; ++tid) {
        for (int e = 0; e < E; ++e) exec_rows[e] += exec_local[(size_t)tid * (E + 1) + e];
        *shared_rows += exec_local[(size_t)tid * (E + 1) + E];
    }
    for (int p = 0; p < n; ++p) exec_priv_rows[p] = exec_priv_local[p];
    free(exec_local);
    free(exec_priv_local);
    return 0;
}

/* The masked logits s = z + m(tau) of the tokens in `tokens` (NULL = all T),
 * fp32-rounded as the routing decision sees them, -inf outside the visible
 * pool: s [n][E]. */
int oracle_logits(const oracle_layer *L, const int32_t *tokens, int n, double *s, int nthreads)
{
    if (check_layer(L)) return -1;
    const int E = L->E_pub + L->E_priv;
    if (!tokens) n = L->T;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel for schedule(dynamic, 4)
    for (int p = 0; p < n; ++p) masked_logits(L, tokens ? tokens[p] : p, s + (size_t)p * E);
    return 0;
}

/* The layer forward of the tokens in `tokens` for a GIVEN routing idx_in
 * [n][k] (global expert ids, in rank order) instead of the top-k the layer
 * would pick: the weights come from the masked logits as in route_weights,
 * then out = bf16(sum_j w_j y_{idx_j}(h) + shared).  It serves the tokens at
 * a routing near-tie, where another selection than the oracle's own is also
 * a valid top-k: their output is checked against the selection actually
 * made.  Writes out_bf16 [n][H] and w_out [n][k].  An id outside the visible
 * pool gets weight 0 (exp(-inf)); -1 for an id outside [0, E). */
int oracle_forward_forced(const oracle_layer *L, const int32_t *tokens, int n, const int32_t *idx_in,
                          uint16_t *out_bf16, double *w_out, int nthreads)
{
    if (check_layer(L)) return -1;
    if (L->E_sh > 0 && (!L->gate_sh || !L->up_sh || !L->down_sh)) return -1;
    const int E = L->E_pub + L->E_priv, H = L->H, I = L->I, k = L->k;
    if (!tokens) n = L->T;
    for (size_t q = 0; q < (size_t)n * k; ++q)
        if (idx_in[q] < 0 || idx_in[q] >= E) return -1;
#ifdef _OPENMP
    if (nthreads > 0) omp_set_num_threads(nthreads);
#else
    (void)nthreads;
#endif
#pragma omp parallel
    {
        double *s = (double *)malloc(sizeof(double) * E);
        double *h = (double *)malloc(sizeof(double) * H);
        double *y = (double *)malloc(sizeof(double) * H);
        double *acc = (double *)malloc(sizeof(double) * H);
        double *a = (double *)malloc(sizeof(double) * I);
        uint32_t dummy = 0;
#pragma omp for schedule(dynamic, 1)
        for (int p = 0; p < n; ++p) {
            const int t = tokens ? tokens[p] : p;
            const int32_t *ti = idx_in + (size_t)p * k;
            double *tw = w_out + (size_t)p * k;
            masked_logits(L, t, s);
            route_weights(L, s, ti, tw);
            const uint16_t *hr = L->hidden + (size_t)t * H;
            for (int c = 0; c < H; ++c) { h[c] = bf16_value(hr[c]); acc[c] = 0.0; }
            for (int j = 0; j < k; ++j) {
                const uint16_t *g, *u, *d;
                routed_expert_weights(L, ti[j], &g, &u, &d);
                swiglu_expert(g, u, d, H, I, h, y, a, &dummy, L->exact);
                for (int c = 0; c < H; ++c) acc[c] += tw[j] * y[c];
            }
            const size_t ih = (size_t)I * H;
            for (int sidx = 0; sidx < L->E_sh; ++sidx) {
                swiglu_expert(L->gate_sh + sidx * ih, L->up_sh + sidx * ih, L->down_sh + sidx * ih, H, I, h, y, a,
                              &dummy, L->exact);
                for (int c = 0; c < H; ++c) acc[c] += y[c];
            }
            for (int c = 0; c < H; ++c) out_bf16[(size_t)p * H + c] = oracle_bf16_round(acc[c]);
        }
        free(s); free(h); free(y); free(acc); free(a);
    }
    return 0;
}

/* Dispatch order of the routed rows (the permutation any grouped expert
 * execution needs): rows are grouped by expert id, and inside an expert by
 * token then rank.  counts[e] = #{(t,j): idx[t][j] = e}; offsets = exclusive
 * prefix sum of counts (E+1 entries); slot_of[t][j] = the row's position;
 * tok_of_slot[slot] = t.  Returns -1 on an id outside [0, E). */
/* ------------------------------------------------------------ backward -- */

/* Gradients of  L = sum_t dout_t . out_t  with respect to the PRIVATE
 * parameters only -- the private router rows and the private experts' gate,
 * up and down projections -- for the routing the forward takes (the top-k
 * choice is piecewise constant).  The public parameters are frozen and get no
 * gradient (G2, Sec. 2.2 and Sec. 3.2: only the private branch is trained).
 * Chain rule through the forward as computed, with its rounding points
 * (fp32 logits, BF16 activation) taken as the identity:
 *   y'_j = W_down a_j,  a = silu(g) u,  out_t = sum_j w_j y'_j (+ shared)
 *   dL/dw_j = dout_t . y'_j
 *   private e = idx[j]:  dW_down[e] += (w_j dout_t) a_j^T,  da = W_down^T (w_j dout_t),
 *     dg = da u silu'(g),  du = da silu(g),  dW_gate[e] += dg h^T,  dW_up[e] += du h^T
 *   router (softmax over the eligible pool p, or renormalised over the top-k w):
 *     renorm:     dz_j = w_j (dL/dw_j - sum_i w_i dL/dw_i) on the selected ids
 *     pool:       dz_e = p_e (dL/dp_e - sum_e' p_e' dL/dp_e') on the pool, dL/dp_e = dL/dw_j if selected
 *     dW_router[e] += dz_e h^T for private e
 * dout [T][H]; outputs (overwritten): d_router [E_priv][H], d_gate / d_up
 * [E_priv][I][H], d_down [E_priv][H][I].  Serial (test sizes). */
int oracle_backward_private(const oracle_layer *L, const double *dout, double *d_router, double *d_gate,
                            double *d_up, double *d_down)
{
    if (check_layer(L)) return -1;
    const int E = L->E_pub + L->E_priv, H = L->H, I = L->I, k = L->k, Ep = L->E_pub;
    memset(d_router, 0, sizeof(double) * L->E_priv * H);
    memset(d_gate, 0, sizeof(double) * L->E_priv * I * H);
    memset(d_up, 0, sizeof(double) * L->E_priv * I * H);
    memset(d_down, 0, sizeof(double) * L->E_priv * H * I);
    double *s = (double *)malloc(sizeof(double) * E), *h = (double *)malloc(sizeof(double) * H);
    double *a = (double *)malloc(sizeof(double) * I), *g = (double *)malloc(sizeof(double) * I);
    double *u = (double *)malloc(sizeof(double) * I), *dy = (double *)malloc(sizeof(double) * H);
    double *da = (double *)malloc(sizeof(double) * I), *dz = (double *)malloc(sizeof(double) * E);
    double *gw = (double *)malloc(sizeof(double) * k), *w = (double *)malloc(sizeof(double) * k);
    char *taken = (char *)malloc(E);
    int32_t *idx = (int32_t *)malloc(sizeof(int32_t) * k);
    for (int t = 0; t < L->T; ++t) {
        const double *dt = dout + (size_t)t * H;
        /* every gradient term is linear in dout_t: a zero row contributes exactly zero */
        int nonzero = 0;
        for (int o = 0; o < H && !nonzero; ++o) nonzero = dt[o] != 0.0;
        if (!nonzero) continue;
        double gap;
        route_token(L, t, idx, w, &gap, s, taken);
        const uint16_t *hr = L->hidden + (size_t)t * H;
        for (int c = 0; c < H; ++c) h[c] = bf16_value(hr[c]);
        for (int j = 0; j < k; ++j) {
            const int e = idx[j];
            const uint16_t *Wg, *Wu, *Wd;
            routed_expert_weights(L, e, &Wg, &Wu, &Wd);
            for (int i = 0; i < I; ++i) {
                double gi = 0.0, ui = 0.0;
                for (int c = 0; c < H; ++c) {
                    gi += h[c] * bf16_value(Wg[(size_t)i * H + c]);
                    ui += h[c] * bf16_value(Wu[(size_t)i * H + c]);
                }
                g[i] = gi;
                u[i] = ui;
                const double silu = gi / (1.0 + exp(-gi));
                a[i] = L->exact ? silu * ui : bf16_value(oracle_bf16_round(silu * ui));
            }
            double gwj = 0.0;  /* dout_t . y'_j */
            for (int o = 0; o < H; ++o) {
                double yo = 0.0;
                for (int i = 0; i < I; ++i) yo += a[i] * bf16_value(Wd[(size_t)o * I + i]);
                gwj += dt[o] * yo;
            }
            gw[j] = gwj;
            if (e < Ep) continue;  /* public expert: frozen */
            const int q = e - Ep;
            for (int o = 0; o < H; ++o) dy[o] = w[j] * dt[o];
            double *Dd = d_down + (size_t)q * H * I, *Dg = d_gate + (size_t)q * I * H, *Du = d_up + (size_t)q * I * H;
            for (int o = 0; o < H; ++o)
                for (int i = 0; i < I; ++i) Dd[(size_t)o * I + i] += dy[o] * a[i];
            for (int i = 0; i < I; ++i) {
                double acc = 0.0;
                for (int o = 0; o < H; ++o) acc += bf16_value(Wd[(size_t)o * I + i]) * dy[o];
                da[i] = acc;
            }
            for (int i = 0; i < I; ++i) {
                const double sg = 1.0 / (1.0 + exp(-g[i]));
                const double dg = da[i] * u[i] * sg * (1.0 + g[i] * (1.0 - sg));
                const double du = da[i] * g[i] * sg;
                for (int c = 0; c < H; ++c) {
                    Dg[(size_t)i * H + c] += dg * h[c];
                    Du[(size_t)i * H + c] += du * h[c];
                }
            }
        }
        /* router: dz over the eligible pool */
        for (int e = 0; e < E; ++e) dz[e] = 0.0;
        if (L->renormalize) {
            double sum = 0.0;
            for (int j = 0; j < k; ++j) sum += w[j] * gw[j];
            for (int j = 0; j < k; ++j) dz[idx[j]] = w[j] * (gw[j] - sum);
        } else {
            const double smax = s[idx[0]];
            double denom = 0.0;
            for (int e = 0; e < E; ++e) denom += exp(s[e] - smax);
            double sum = 0.0;
            for (int j = 0; j < k; ++j) sum += w[j] * gw[j];  /* w_j = p_{idx[j]} */
            for (int e = 0; e < E; ++e) {
                if (s[e] == -INFINITY) continue;
                const double pe = exp(s[e] - smax) / denom;
                double dpe = 0.0;
                for (int j = 0; j < k; ++j)
                    if (idx[j] == e) dpe = gw[j];
                dz[e] = pe * (dpe - sum);
            }
        }
        for (int e = Ep; e < E; ++e)
            if (dz[e] != 0.0)
                for (int c = 0; c < H; ++c) d_router[(size_t)(e - Ep) * H + c] += dz[e] * h[c];
    }
    free(s); free(h); free(a); free(g); free(u); free(dy); free(da); free(dz); free(gw); free(w); free(taken); free(idx);
    return 0;
}

/* Gradient of L = sum_t dout_t . out_t with respect to the layer's input h
 * (the hidden states), for the routing the forward takes: what the layer
 * below needs when its own private branch is trained (Sec. 3.2 trains the
 * private experts of two wrapped layers).  Every parameter is held fixed
 * here -- public, private and shared alike -- and none gets a gradient; the
 * input gradient still flows through the frozen ones (Sec. 2.2: G2 is a
 * claim about the optimizer state, not about the derivative).  Chain rule
 * through the forward as computed, rounding points as the identity:
 *   per pick j (expert e, weight w_j):  da = W_down,e^T (w_j dout_t),
 *     dg = da u silu'(g),  du = da silu(g),  dh += W_gate,e^T dg + W_up,e^T du
 *   per shared expert (weight 1): the same with da = W_down,s^T dout_t
 *   router, over the token's eligible pool (the unmasked control: all E):
 *     dz as in oracle_backward_private,  dh += sum_e dz_e W_router,e
 * A token whose dout row is zero contributes nothing and is skipped.
 * dout [T][H]; d_hidden [T][H] (overwritten).  Serial (test sizes). */
int oracle_backward_input(const oracle_layer *L, const double *dout, double *d_hidden)
{
    if (check_layer(L)) return -1;
    const int E = L->E_pub + L->E_priv, H = L->H, I = L->I, k = L->k;
    memset(d_hidden, 0, sizeof(double) * (size_t)L->T * H);
    double *s = (double *)malloc(sizeof(double) * E), *h = (double *)malloc(sizeof(double) * H);
    double *a = (double *)malloc(sizeof(double) * I), *g = (double *)malloc(sizeof(double) * I);
    double *u = (double *)malloc(sizeof(double) * I), *da = (double *)malloc(sizeof(double) * I);
    double *dz = (double *)malloc(sizeof(double) * E);
    double *gw = (double *)malloc(sizeof(double) * k), *w = (double *)malloc(sizeof(double) * k);
    char *taken = (char *)malloc(E);
    int32_t *idx = (int32_t *)malloc(sizeof(int32_t) * k);
    for (int t = 0; t < L->T; ++t) {
        const double *dt = dout + (size_t)t * H;
        int nonzero = 0;
        for (int o = 0; o < H && !nonzero; ++o) nonzero = dt[o] != 0.0;
        if (!nonzero) continue;
        double gap;
        route_token(L, t, idx, w, &gap, s, taken);
        const uint16_t *hr = L->hidden + (size_t)t * H;
        for (int c = 0; c < H; ++c) h[c] = bf16_value(hr[c]);
        double *dh = d_hidden + (size_t)t * H;
        /* routed experts (j < k) and shared experts (j >= k, weight 1) */
        for (int j = 0; j < k + L->E_sh; ++j) {
            const uint16_t *Wg, *Wu, *Wd;
            double wj = 1.0;
            if (j < k) {
                routed_expert_weights(L, idx[j], &Wg, &Wu, &Wd);
                wj = w[j];
            } else {
                const size_t ih = (size_t)I * H;
                Wg = L->gate_sh + (j - k) * ih; Wu = L->up_sh + (j - k) * ih; Wd = L->down_sh + (j - k) * ih;
            }
            for (int i = 0; i < I; ++i) {
                double gi = 0.0, ui = 0.0;
                for (int c = 0; c < H; ++c) {
                    gi += h[c] * bf16_value(Wg[(size_t)i * H + c]);
                    ui += h[c] * bf16_value(Wu[(size_t)i * H + c]);
                }
                g[i] = gi;
                u[i] = ui;
                const double silu = gi / (1.0 + exp(-gi));
                a[i] = L->exact ? silu * ui : bf16_value(oracle_bf16_round(silu * ui));
            }
            if (j < k) {  /* dL/dw_j = dout_t . y'_j */
                double gwj = 0.0;
                for (int o = 0; o < H; ++o) {
                    double yo = 0.0;
                    for (int i = 0; i < I; ++i) yo += a[i] * bf16_value(Wd[(size_t)o * I + i]);
                    gwj += dt[o] * yo;
                }
                gw[j] = gwj;
            }
            for (int i = 0; i < I; ++i) {
                double acc = 0.0;
                for (int o = 0; o < H; ++o) acc += bf16_value(Wd[(size_t)o * I + i]) * dt[o];
                da[i] = wj * acc;
            }
            for (int i = 0; i < I; ++i) {
                const double sg = 1.0 / (1.0 + exp(-g[i]));
                const double dg = da[i] * u[i] * sg * (1.0 + g[i] * (1.0 - sg));
                const double du = da[i] * g[i] * sg;
                for (int c = 0; c < H; ++c)
                    dh[c] += dg * bf16_value(Wg[(size_t)i * H + c]) + du * bf16_value(Wu[(size_t)i * H + c]);
            }
        }
        /* router: dz over the eligible pool, dh += sum_e dz_e W_router,e */
        for (int e = 0; e < E; ++e) dz[e] = 0.0;
        double sum = 0.0;
        for (int j = 0; j < k; ++j) sum += w[j] * gw[j];
        if (L->renormalize) {
            for (int j = 0; j < k; ++j) dz[idx[j]] = w[j] * (gw[j] - sum);
        } else {
            const double smax = s[idx[0]];
            double denom = 0.0;
            for (int e = 0; e < E; ++e) denom += exp(s[e] - smax);
            for (int e = 0; e < E; ++e) {
                if (s[e] == -INFINITY) continue;
                const double pe = exp(s[e] - smax) / denom;
                double dpe = 0.0;
                for (int j = 0; j < k; ++j)
                    if (idx[j] == e) dpe = gw[j];
                dz[e] = pe * (dpe - sum);
            }
        }
        for (int e = 0; e < E; ++e)
            if (dz[e] != 0.0) {
                const uint16_t *wr = router_row(L, e);
                for (int c = 0; c < H; ++c) dh[c] += dz[e] * bf16_value(wr[c]);
            }
    }
    free(s); free(h); free(a); free(g); free(u); free(da); free(dz); free(gw); free(w); free(taken); free(idx);
    return 0;
}

int oracle_permute(const int32_t *idx, int T, int k, int E, uint32_t *counts, uint32_t *offsets, int32_t *slot_of,
                   int32_t *tok_of_slot)
{
    for (int e = 0; e < E; ++e) counts[e] = 0;
    for (size_t r = 0; r < (size_t)T * k; ++r) {
        if (idx[r] < 0 || idx[r] >= E) return -1;
        counts[idx[r]] += 1;
    }
    offsets[0] = 0;
    for (int e = 0; e < E; ++e) offsets[e + 1] = offsets[e] + counts[e];
    uint32_t next = 0;
    for (int e = 0; e < E; ++e)
        for (int t = 0; t < T; ++t)
            for (int j = 0; j < k; ++j)
                if (idx[(size_t)t * k + j] == e) {
                    slot_of[(size_t)t * k + j] = (int32_t)next;
                    tok_of_slot[next] = t;
                    next += 1;
                }
    return 0;
}
