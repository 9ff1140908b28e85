/*
 * hybrid_oracle.c -- plain fp64 CPU oracle for block-hybrid attention.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the independent reference that the
 * CUDA path is checked against.  Only the test suite, the smoke check and the
 * CPU-baseline leg of the benchmark may load it.  It shares no code, header,
 * table or helper with the CUDA library, and it never reads anything the
 * CUDA library produced except where a caller passes such data in explicitly.
 *
 * Source: "Retrofitting Linear Attention into Diffusion Language Models",
 * Section 3.1 (block-hybrid attention) and Section 2.2 (linear attention,
 * Eq. 1).  Every routine below writes a definition of that section out
 * literally, in double precision, with no blocking, fusion or reordering:
 *
 *   phi(x)   = [softmax(x W), softmax(-x W)]            (Sec. 3.1, Hedgehog map)
 *   a_j      = exp(q . k_j / sqrt(d)),  j in active block (Sec. 3.1)
 *   sm_num   = sum_j a_j v_j,   sm_den = sum_j a_j       (Sec. 3.1)
 *   S_n      = S_{n-1} + sum_t phi(k_t) v_t^T            (Sec. 3.1, commit)
 *   Z_n      = Z_{n-1} + sum_t phi(k_t)                  (Sec. 3.1, commit)
 *   lin_num  = phi(q)^T S_{n-1},  lin_den = phi(q)^T Z_{n-1}   (Sec. 3.1)
 *   w        = sigmoid(alpha)                            (Sec. 3.1, gate)
 *   out      = (w sm_num + lin_num) / (w sm_den + lin_den)      (Sec. 3.1)
 *
 * The training form (Sec. 3.2, Stage 1) applies the same definitions to every
 * block of a sequence (oracle_train_forward) and writes out, by the chain
 * rule, the gradient of sum(dO * O) with respect to W and alpha
 * (oracle_train_backward).
 *
 * A second route (oracle_block_attn_prefix) never forms S or Z: it sums the
 * linear branch token by token over the explicit prefix, the left-hand form
 * of Eq. 1.  The two routes are a mutual check (state = explicit sum).
 *
 * Readings of points the paper leaves open (each is listed in the design
 * notes as well):
 *   - W is indexed per state (key/value) head; query head h of a GQA group of
 *     size G = Hq / Hkv uses the W and the state of head h / G.  With
 *     Hq == Hkv this is the paper's "per query head" design.
 *   - The gate alpha is per query head.
 *   - No scale or temperature inside phi; 1/sqrt(d) only in the softmax branch.
 *   - No mask inside the active block (bidirectional, all B x B pairs).
 *   - The softmax inside phi and the exponentials of the softmax branch are
 *     evaluated unshifted, exactly as defined; the routines refuse inputs whose
 *     exponent arguments leave [-700, 700] (fp64 would overflow).
 *
 * Logical layouts (all row-major, double):
 *   Q, O     [n_req][B][Hq][d]
 *   K, V     [n_req][T][Hkv][d]      (T = B for the active block)
 *   W        [Hkv][d][F]
 *   alpha    [Hq]
 *   S        [n_req][Hkv][2F][d]     (the paper's S in R^{2F x d})
 *   z        [n_req][Hkv][2F]        (the paper's Z)
 *
 * phi_kind 0 = Hedgehog (the paper's map), 1 = identity (phi(x) = x, 2F := d;
 * used only to pin the oracle against the plain linear-attention formula).
 *
 * Return value of every entry point: 0 on success, -1 on a bad argument,
 * -2 if an exponent argument left [-700, 700].
 */
#include <math.h>
#include <pthread.h>
#include <stdlib.h>
#include <string.h>

#define ORACLE_EXP_LIMIT 700.0

enum { PHI_HEDGEHOG = 0, PHI_IDENTITY = 1 };

/* Width of phi(x): 2F for the Hedgehog map, d for the identity map. */
static int phi_width(int phi_kind, int d, int F)
{
    return phi_kind == PHI_IDENTITY ? d : 2 * F;
}

/*
 * phi(x) for one vector x in R^d with W in R^{d x F} (Sec. 3.1):
 *   u      = x W                     (u_f = sum_e x_e W[e][f])
 *   out[f]     = exp(u_f)  / sum_g exp(u_g)      f = 0..F-1   (softmax(xW))
 *   out[F + f] = exp(-u_f) / sum_g exp(-u_g)     f = 0..F-1   (softmax(-xW))
 * Returns -2 if some |u_f| exceeds the fp64 exponent limit.
 */
static int phi_one(int phi_kind, const double *x, const double *W, int d, int F,
                   double *u /* scratch, F */, double *out)
{
    if (phi_kind == PHI_IDENTITY) {
        for (int e = 0; e < d; ++e) out[e] = x[e];
        return 0;
    }
    for (int f = 0; f < F; ++f) {
        double acc = 0.0;
        for (int e = 0; e < d; ++e) acc += x[e] * W[(size_t)e * F + f];
        if (fabs(acc) > ORACLE_EXP_LIMIT) return -2;
        u[f] = acc;
    }
    double sum_pos = 0.0, sum_neg = 0.0;
    for (int f = 0; f < F; ++f) {
        sum_pos += exp(u[f]);
        sum_neg += exp(-u[f]);
    }
    for (int f = 0; f < F; ++f) {
        out[f] = exp(u[f]) / sum_pos;
        out[F + f] = exp(-u[f]) / sum_neg;
    }
    return 0;
}

/* ---------------------------------------------------------------------------
 * The definitions of Sec. 3.1 that every route below shares, one routine each.
 * ------------------------------------------------------------------------- */

/* Gate w = sigma(alpha) = 1 / (1 + exp(-alpha)); alpha = -inf gives 0, +inf gives 1. */
static double gate(double alpha)
{
    return 1.0 / (1.0 + exp(-alpha));
}

/* GQA: query head h reads the state (and W) of state head h / G, G = Hq / Hkv. */
static int group_of(int h, int Hq, int Hkv)
{
    const int G = Hq / Hkv;
    return h / G;
}

/* Within-block softmax branch for one query q over the B keys / values of
 * its block (row j at K + j*stride, V + j*stride):
 *   a_j = exp(q . k_j / sqrt(d)),  sm_num = sum_j a_j v_j,  sm_den = sum_j a_j. */
static int softmax_branch(const double *q, const double *K, const double *V, size_t stride, int B,
                          int d, double *sm_num, double *sm_den_out)
{
    double sm_den = 0.0;
    for (int e = 0; e < d; ++e) sm_num[e] = 0.0;
    for (int j = 0; j < B; ++j) {
        const double *k = K + (size_t)j * stride;
        const double *v = V + (size_t)j * stride;
        double s = 0.0;
        for (int e = 0; e < d; ++e) s += q[e] * k[e];
        s /= sqrt((double)d);
        if (fabs(s) > ORACLE_EXP_LIMIT) return -2;
        const double a = exp(s);
        for (int e = 0; e < d; ++e) sm_num[e] += a * v[e];
        sm_den += a;
    }
    *sm_den_out = sm_den;
    return 0;
}

/* Cross-block branch read from the state: lin_num = phi(q)^T S, lin_den = phi(q)^T z. */
static void linear_branch(const double *phi_q, const double *S, const double *z, int P2, int d,
                          double *lin_num, double *lin_den_out)
{
    double lin_den = 0.0;
    for (int e = 0; e < d; ++e) lin_num[e] = 0.0;
    for (int f = 0; f < P2; ++f) {
        for (int e = 0; e < d; ++e) lin_num[e] += phi_q[f] * S[(size_t)f * d + e];
        lin_den += phi_q[f] * z[f];
    }
    *lin_den_out = lin_den;
}

/* Gated shared normaliser: out = (w sm_num + lin_num) / (w sm_den + lin_den);
 * returns the denominator. */
static double merge(double w, const double *sm_num, double sm_den, const double *lin_num,
                    double lin_den, int d, double *o)
{
    const double den = w * sm_den + lin_den;
    for (int e = 0; e < d; ++e) o[e] = (w * sm_num[e] + lin_num[e]) / den;
    return den;
}

/* Commit of one token: S += phi(k) v^T, z += phi(k). */
static void commit_token(const double *phi, const double *v, int P2, int d, double *S, double *z)
{
    for (int f = 0; f < P2; ++f) {
        for (int e = 0; e < d; ++e) S[(size_t)f * d + e] += phi[f] * v[e];
        z[f] += phi[f];
    }
}

/* ---------------------------------------------------------------------------
 * Feature map on a batch of rows.
 *   X   [n_rows][n_heads_x][d],  W [Hkv][d][F],  Phi [n_rows][n_heads_x][2F]
 * Row head h uses W[h / (n_heads_x / Hkv)] (queries: h / G; keys: h).
 * ------------------------------------------------------------------------- */
int oracle_feature_map(long n_rows, int n_heads_x, int n_kv_heads, int d, int F,
                       const double *X, const double *W, double *Phi)
{
    if (n_rows < 0 || n_heads_x <= 0 || n_kv_heads <= 0 || d <= 0 || F <= 0) return -1;
    if (n_heads_x % n_kv_heads != 0) return -1;
    const int group = n_heads_x / n_kv_heads;
    double *u = (double *)malloc(sizeof(double) * (size_t)F);
    if (!u) return -1;
    int rc = 0;
    for (long r = 0; r < n_rows && rc == 0; ++r) {
        for (int h = 0; h < n_heads_x && rc == 0; ++h) {
            const double *x = X + ((size_t)r * n_heads_x + h) * d;
            const double *Wg = W + (size_t)(h / group) * d * F;
            rc = phi_one(PHI_HEDGEHOG, x, Wg, d, F, u, Phi + ((size_t)r * n_heads_x + h) * 2 * F);
        }
    }
    free(u);
    return rc;
}

/* ---------------------------------------------------------------------------
 * Simple static fan-out of independent (request, head) units over threads.
 * Units never share an output element, so the split changes no result.
 * ------------------------------------------------------------------------- */
typedef int (*unit_fn)(void *ctx, long unit, double *scratch);

typedef struct {
    unit_fn fn;
    void *ctx;
    long n_units;
    int n_threads;
    int tid;
    size_t scratch_doubles;
    int rc;
} fanout_arg;

static void *fanout_worker(void *p)
{
    fanout_arg *a = (fanout_arg *)p;
    double *scratch = (double *)malloc(sizeof(double) * (a->scratch_doubles ? a->scratch_doubles : 1));
    if (!scratch) { a->rc = -1; return NULL; }
    a->rc = 0;
    for (long u = a->tid; u < a->n_units; u += a->n_threads) {
        int rc = a->fn(a->ctx, u, scratch);
        if (rc != 0) { a->rc = rc; break; }
    }
    free(scratch);
    return NULL;
}

static int fanout(unit_fn fn, void *ctx, long n_units, int n_threads, size_t scratch_doubles)
{
    if (n_threads < 1) n_threads = 1;
    if (n_threads > 1024) n_threads = 1024;
    if ((long)n_threads > n_units) n_threads = n_units > 0 ? (int)n_units : 1;
    fanout_arg *args = (fanout_arg *)calloc((size_t)n_threads, sizeof(fanout_arg));
    pthread_t *th = (pthread_t *)calloc((size_t)n_threads, sizeof(pthread_t));
    if (!args || !th) { free(args); free(th); return -1; }
    for (int t = 0; t < n_threads; ++t) {
        args[t].fn = fn; args[t].ctx = ctx; args[t].n_units = n_units;
        args[t].n_threads = n_threads; args[t].tid = t;
        args[t].scratch_doubles = scratch_doubles;
    }
    int started = 0;
    for (int t = 1; t < n_threads; ++t) {
        if (pthread_create(&th[t], NULL, fanout_worker, &args[t]) != 0) break;
        started = t;
    }
    fanout_worker(&args[0]);
    for (int t = 1; t <= started; ++t) pthread_join(th[t], NULL);
    int rc = 0;
    for (int t = 0; t < n_threads; ++t) if (args[t].rc != 0) rc = args[t].rc;
    if (started != n_threads - 1) rc = -1;
    free(args); free(th);
    return rc;
}

/* ---------------------------------------------------------------------------
 * Block commit (Sec. 3.1):  S += sum_t phi(k_t) v_t^T,   z += sum_t phi(k_t)
 * for every (request, state head), over the T given tokens, in token order.
 * ------------------------------------------------------------------------- */
typedef struct {
    int n_req, T, Hkv, d, F, phi_kind;
    const double *K, *V, *W;
    double *S, *z;
} commit_ctx;

static int commit_unit(void *p, long unit, double *scratch)
{
    const commit_ctx *c = (const commit_ctx *)p;
    const int r = (int)(unit / c->Hkv), g = (int)(unit % c->Hkv);
    const int d = c->d, F = c->F, P2 = phi_width(c->phi_kind, d, F);
    double *u = scratch, *phi = scratch + F;
    double *S = c->S + ((size_t)r * c->Hkv + g) * P2 * d;
    double *z = c->z + ((size_t)r * c->Hkv + g) * P2;
    const double *Wg = c->W ? c->W + (size_t)g * d * F : NULL;
    for (int t = 0; t < c->T; ++t) {
        const double *k = c->K + (((size_t)r * c->T + t) * c->Hkv + g) * d;
        const double *v = c->V + (((size_t)r * c->T + t) * c->Hkv + g) * d;
        int rc = phi_one(c->phi_kind, k, Wg, d, F, u, phi);
        if (rc) return rc;
        commit_token(phi, v, P2, d, S, z);
    }
    return 0;
}

int oracle_commit(int n_req, int T, int Hkv, int d, int F, int phi_kind,
                  const double *K, const double *V, const double *W,
                  double *S, double *z, int n_threads)
{
    if (n_req < 0 || T < 0 || Hkv <= 0 || d <= 0 || F <= 0) return -1;
    if (phi_kind != PHI_HEDGEHOG && phi_kind != PHI_IDENTITY) return -1;
    if (phi_kind == PHI_HEDGEHOG && !W) return -1;
    commit_ctx c = { n_req, T, Hkv, d, F, phi_kind, K, V, W, S, z };
    const int P2 = phi_width(phi_kind, d, F);
    return fanout(commit_unit, &c, (long)n_req * Hkv, n_threads, (size_t)F + (size_t)P2);
}

/* ---------------------------------------------------------------------------
 * One active block, both branches, gated shared normaliser (Sec. 3.1).
 * The cross-block branch comes either from the state (S, z) or, in the
 * second route, from the explicit prefix tokens (Eq. 1 summed directly).
 * ------------------------------------------------------------------------- */
typedef struct {
    int n_req, B, Hq, Hkv, d, F, phi_kind;
    const double *Q, *K, *V, *W, *alpha;
    /* route 1: state */
    const double *S, *z;
    /* route 2: explicit prefix */
    const double *Kp, *Vp;
    const int *prefix_len;
    int P_max;
    double *O;
} attn_ctx;

static int attn_unit(void *p, long unit, double *scratch)
{
    const attn_ctx *c = (const attn_ctx *)p;
    const int r = (int)(unit / c->Hq), h = (int)(unit % c->Hq);
    const int d = c->d, F = c->F, B = c->B;
    const int g = group_of(h, c->Hq, c->Hkv);
    const int P2 = phi_width(c->phi_kind, d, F);
    const double *Wg = c->W ? c->W + (size_t)g * d * F : NULL;

    double *u = scratch;                 /* F      */
    double *phi_q = u + F;               /* P2     */
    double *phi_k = phi_q + P2;          /* P2     */
    double *sm_num = phi_k + P2;         /* d      */
    double *lin_num = sm_num + d;        /* d      */

    const double w = gate(c->alpha[h]);

    for (int i = 0; i < B; ++i) {
        const double *q = c->Q + (((size_t)r * B + i) * c->Hq + h) * d;

        /* within-block softmax branch: a_j = exp(q . k_j / sqrt(d)) over all j of the block */
        double sm_den = 0.0;
        const size_t kv0 = ((size_t)r * B * c->Hkv + g) * d;
        int rc = softmax_branch(q, c->K + kv0, c->V + kv0, (size_t)c->Hkv * d, B, d, sm_num, &sm_den);
        if (rc) return rc;

        /* cross-block linear branch */
        rc = phi_one(c->phi_kind, q, Wg, d, F, u, phi_q);
        if (rc) return rc;
        double lin_den = 0.0;
        if (c->S) {
            /* route 1: lin_num = phi(q)^T S, lin_den = phi(q)^T z */
            const double *S = c->S + ((size_t)r * c->Hkv + g) * P2 * d;
            const double *z = c->z + ((size_t)r * c->Hkv + g) * P2;
            linear_branch(phi_q, S, z, P2, d, lin_num, &lin_den);
        } else {
            for (int e = 0; e < d; ++e) lin_num[e] = 0.0;
            /* route 2: lin_num = sum_t (phi(q) . phi(k_t)) v_t over the prefix tokens (Eq. 1) */
            const int P = c->prefix_len[r];
            for (int t = 0; t < P; ++t) {
                const double *kt = c->Kp + (((size_t)r * c->P_max + t) * c->Hkv + g) * d;
                const double *vt = c->Vp + (((size_t)r * c->P_max + t) * c->Hkv + g) * d;
                rc = phi_one(c->phi_kind, kt, Wg, d, F, u, phi_k);
                if (rc) return rc;
                double kern = 0.0;
                for (int f = 0; f < P2; ++f) kern += phi_q[f] * phi_k[f];
                for (int e = 0; e < d; ++e) lin_num[e] += kern * vt[e];
                lin_den += kern;
            }
        }

        /* gated merge through the shared normaliser */
        merge(w, sm_num, sm_den, lin_num, lin_den, d, c->O + (((size_t)r * B + i) * c->Hq + h) * d);
    }
    return 0;
}

static int attn_check(int n_req, int B, int Hq, int Hkv, int d, int F, int phi_kind,
                      const double *W)
{
    if (n_req < 0 || B <= 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || F <= 0) return -1;
    if (Hq % Hkv != 0) return -1;
    if (phi_kind != PHI_HEDGEHOG && phi_kind != PHI_IDENTITY) return -1;
    if (phi_kind == PHI_HEDGEHOG && !W) return -1;
    return 0;
}

int oracle_block_attn(int n_req, int B, int Hq, int Hkv, int d, int F, int phi_kind,
                      const double *Q, const double *K, const double *V,
                      const double *W, const double *alpha,
                      const double *S, const double *z, double *O, int n_threads)
{
    if (attn_check(n_req, B, Hq, Hkv, d, F, phi_kind, W) || !S || !z) return -1;
    attn_ctx c;
    memset(&c, 0, sizeof c);
    c.n_req = n_req; c.B = B; c.Hq = Hq; c.Hkv = Hkv; c.d = d; c.F = F; c.phi_kind = phi_kind;
    c.Q = Q; c.K = K; c.V = V; c.W = W; c.alpha = alpha; c.S = S; c.z = z; c.O = O;
    const int P2 = phi_width(phi_kind, d, F);
    return fanout(attn_unit, &c, (long)n_req * Hq, n_threads, (size_t)F + 2u * P2 + 2u * d);
}

int oracle_block_attn_prefix(int n_req, int B, int Hq, int Hkv, int d, int F, int phi_kind,
                             const double *Q, const double *K, const double *V,
                             const double *W, const double *alpha,
                             const double *Kp, const double *Vp, const int *prefix_len,
                             int P_max, double *O, int n_threads)
{
    if (attn_check(n_req, B, Hq, Hkv, d, F, phi_kind, W) || !prefix_len || P_max < 0) return -1;
    for (int r = 0; r < n_req; ++r)
        if (prefix_len[r] < 0 || prefix_len[r] > P_max) return -1;
    attn_ctx c;
    memset(&c, 0, sizeof c);
    c.n_req = n_req; c.B = B; c.Hq = Hq; c.Hkv = Hkv; c.d = d; c.F = F; c.phi_kind = phi_kind;
    c.Q = Q; c.K = K; c.V = V; c.W = W; c.alpha = alpha;
    c.Kp = Kp; c.Vp = Vp; c.prefix_len = prefix_len; c.P_max = P_max; c.O = O;
    const int P2 = phi_width(phi_kind, d, F);
    return fanout(attn_unit, &c, (long)n_req * Hq, n_threads, (size_t)F + 2u * P2 + 2u * d);
}

/* ===========================================================================
 * Training form (Sec. 3.2, Stage 1 attention transfer).
 *
 * A training sequence of L = n_blk * B tokens is cut into blocks B_0, B_1, ...
 * of B tokens.  Teacher forcing gives every block its queries, keys and
 * values; block n attends to itself with the exact softmax branch and to the
 * blocks before it through S_{n-1}, Z_{n-1} (Sec. 3.1 applied to each block of
 * the sequence; S_{-1} = 0).  Stage 1 trains only psi = {W, alpha}.
 *
 * Layouts: Q, O, dO [n_seq][L][Hq][d];  K, V [n_seq][L][Hkv][d];
 *          W, dW [Hkv][d][F];  alpha, dalpha [Hq].
 * ------------------------------------------------------------------------- */
typedef struct {
    int n_seq, L, B, Hq, Hkv, d, F;
    const double *Q, *K, *V, *W, *alpha, *dO;
    double *O;
    double *dW_part;       /* [n_seq * Hkv][d][F]  one slot per unit */
    double *dw_part;       /* [n_seq * Hq]          d loss / d w per (sequence, head) */
} train_ctx;

/* Forward for one (sequence, query head): block by block, the outputs of the
 * block's queries against the state of the earlier blocks, then the commit
 * of the block into that state. */
static int train_fwd_unit(void *p, long unit, double *scratch)
{
    const train_ctx *c = (const train_ctx *)p;
    const int s = (int)(unit / c->Hq), h = (int)(unit % c->Hq);
    const int d = c->d, F = c->F, B = c->B, P2 = 2 * F;
    const int g = group_of(h, c->Hq, c->Hkv);
    const double *Wg = c->W + (size_t)g * d * F;
    const size_t q_row = (size_t)c->Hq * d, kv_row = (size_t)c->Hkv * d;
    double *S = scratch;                      /* P2 * d */
    double *z = S + (size_t)P2 * d;           /* P2     */
    double *u = z + P2;                       /* F      */
    double *phi = u + F;                      /* P2     */
    double *sm_num = phi + P2;                /* d      */
    double *lin_num = sm_num + d;             /* d      */
    for (size_t i = 0; i < (size_t)P2 * d + P2; ++i) S[i] = 0.0;
    const double w = gate(c->alpha[h]);
    const int n_blk = c->L / B;
    for (int n = 0; n < n_blk; ++n) {
        const size_t t0 = (size_t)s * c->L + (size_t)n * B;   /* first token of block n */
        const double *Kb = c->K + t0 * kv_row + (size_t)g * d;
        const double *Vb = c->V + t0 * kv_row + (size_t)g * d;
        for (int i = 0; i < B; ++i) {
            const double *q = c->Q + (t0 + i) * q_row + (size_t)h * d;
            double sm_den, lin_den;
            int rc = softmax_branch(q, Kb, Vb, kv_row, B, d, sm_num, &sm_den);
            if (rc) return rc;
            rc = phi_one(PHI_HEDGEHOG, q, Wg, d, F, u, phi);
            if (rc) return rc;
            linear_branch(phi, S, z, P2, d, lin_num, &lin_den);
            merge(w, sm_num, sm_den, lin_num, lin_den, d, c->O + (t0 + i) * q_row + (size_t)h * d);
        }
        /* block n commits after its own readout */
        for (int t = 0; t < B; ++t) {
            int rc = phi_one(PHI_HEDGEHOG, Kb + (size_t)t * kv_row, Wg, d, F, u, phi);
            if (rc) return rc;
            commit_token(phi, Vb + (size_t)t * kv_row, P2, d, S, z);
        }
    }
    return 0;
}

/* Reverse mode through phi(x) = [softmax(u), softmax(-u)], u = x W, for one
 * vector: given g = dL/dphi (2F), add dL/dW[e][f] = x[e] * du[f] into dW, with
 *   du = p+ (g+ - <g+, p+>) - p- (g- - <g-, p->),   p+- = softmax(+-u). */
static void phi_backward_add(const double *x, const double *phi, const double *gphi, int d, int F,
                             double *du /* scratch, F */, double *dW)
{
    double dot_pos = 0.0, dot_neg = 0.0;
    for (int f = 0; f < F; ++f) {
        dot_pos += gphi[f] * phi[f];
        dot_neg += gphi[F + f] * phi[F + f];
    }
    for (int f = 0; f < F; ++f)
        du[f] = phi[f] * (gphi[f] - dot_pos) - phi[F + f] * (gphi[F + f] - dot_neg);
    for (int e = 0; e < d; ++e)
        for (int f = 0; f < F; ++f) dW[(size_t)e * F + f] += x[e] * du[f];
}

/* Backward for one (sequence, state head g): the gradient of sum(dO * O) with
 * respect to W_g and to the gates w_h of the G query heads of the group.
 * Per query row i of block n (N = numerator, D = denominator of the merge):
 *   dN = g / D,   dD = -(g . o) / D,            g = dO row, o = N / D
 *   dw_h    += dN . sm_num + dD sm_den
 *   dphi(q)  = S_{n-1} dN + Z_{n-1} dD,    dS_{n-1} += phi(q) dN^T,  dZ_{n-1} += phi(q) dD
 * and, since S_{n-1} = sum_{m < n} sum_{t in B_m} phi(k_t) v_t^T, a key t of
 * block m receives  dphi(k_t) = (sum_{n > m} dS_{n-1}) v_t + sum_{n > m} dZ_{n-1}. */
static int train_bwd_unit(void *p, long unit, double *scratch)
{
    const train_ctx *c = (const train_ctx *)p;
    const int s = (int)(unit / c->Hkv), g = (int)(unit % c->Hkv);
    const int d = c->d, F = c->F, B = c->B, P2 = 2 * F;
    const int G = c->Hq / c->Hkv, n_blk = c->L / B;
    const size_t st = (size_t)P2 * d + P2;    /* one (S, Z) pair */
    const size_t q_row = (size_t)c->Hq * d, kv_row = (size_t)c->Hkv * d;
    const double *Wg = c->W + (size_t)g * d * F;
    double *Spre = scratch;                   /* n_blk states: S_{n-1}, Z_{n-1} for block n */
    double *dSpre = Spre + (size_t)n_blk * st;/* n_blk gradients of those states */
    double *u = dSpre + (size_t)n_blk * st;   /* F  */
    double *phi = u + F;                      /* P2 */
    double *gphi = phi + P2;                  /* P2 */
    double *sm_num = gphi + P2;               /* d  */
    double *lin_num = sm_num + d;             /* d  */
    double *o = lin_num + d;                  /* d  */
    double *dN = o + d;                       /* d  */
    double *du = dN + d;                      /* F  */
    double *acc = du + F;                     /* st: running sum of dS over later blocks */
    double *dW = c->dW_part + (size_t)unit * d * F;
    for (size_t i = 0; i < (size_t)n_blk * st; ++i) { Spre[i] = 0.0; dSpre[i] = 0.0; }
    for (size_t i = 0; i < (size_t)d * F; ++i) dW[i] = 0.0;

    /* prefix states: S_{n-1} = S_{n-2} + commit(B_{n-1}) */
    for (int n = 1; n < n_blk; ++n) {
        double *Sn = Spre + (size_t)n * st;
        for (size_t i = 0; i < st; ++i) Sn[i] = Sn[i - st];
        const size_t t0 = (size_t)s * c->L + (size_t)(n - 1) * B;
        for (int t = 0; t < B; ++t) {
            const size_t kv = (t0 + t) * kv_row + (size_t)g * d;
            int rc = phi_one(PHI_HEDGEHOG, c->K + kv, Wg, d, F, u, phi);
            if (rc) return rc;
            commit_token(phi, c->V + kv, P2, d, Sn, Sn + (size_t)P2 * d);
        }
    }

    /* query side */
    for (int hl = 0; hl < G; ++hl) {
        const int h = g * G + hl;
        const double w = gate(c->alpha[h]);
        double dw = 0.0;
        for (int n = 0; n < n_blk; ++n) {
            const double *S = Spre + (size_t)n * st, *z = S + (size_t)P2 * d;
            double *dS = dSpre + (size_t)n * st, *dz = dS + (size_t)P2 * d;
            const size_t t0 = (size_t)s * c->L + (size_t)n * B;
            const double *Kb = c->K + t0 * kv_row + (size_t)g * d;
            const double *Vb = c->V + t0 * kv_row + (size_t)g * d;
            for (int i = 0; i < B; ++i) {
                const double *q = c->Q + (t0 + i) * q_row + (size_t)h * d;
                const double *gr = c->dO + (t0 + i) * q_row + (size_t)h * d;
                double sm_den, lin_den;
                int rc = softmax_branch(q, Kb, Vb, kv_row, B, d, sm_num, &sm_den);
                if (rc) return rc;
                rc = phi_one(PHI_HEDGEHOG, q, Wg, d, F, u, phi);
                if (rc) return rc;
                linear_branch(phi, S, z, P2, d, lin_num, &lin_den);
                const double D = merge(w, sm_num, sm_den, lin_num, lin_den, d, o);
                double go = 0.0;
                for (int e = 0; e < d; ++e) go += gr[e] * o[e];
                const double dD = -go / D;
                for (int e = 0; e < d; ++e) dN[e] = gr[e] / D;
                for (int e = 0; e < d; ++e) dw += dN[e] * sm_num[e];
                dw += dD * sm_den;
                for (int f = 0; f < P2; ++f) {
                    double acc_f = z[f] * dD;
                    for (int e = 0; e < d; ++e) acc_f += S[(size_t)f * d + e] * dN[e];
                    gphi[f] = acc_f;
                    for (int e = 0; e < d; ++e) dS[(size_t)f * d + e] += phi[f] * dN[e];
                    dz[f] += phi[f] * dD;
                }
                phi_backward_add(q, phi, gphi, d, F, du, dW);
            }
        }
        c->dw_part[(size_t)s * c->Hq + h] = dw;
    }

    /* key side: block m gets the sum of dS_{n-1} over the later blocks n > m */
    for (size_t i = 0; i < st; ++i) acc[i] = 0.0;
    for (int m = n_blk - 1; m >= 0; --m) {
        if (m + 1 < n_blk) {
            const double *dS = dSpre + (size_t)(m + 1) * st;
            for (size_t i = 0; i < st; ++i) acc[i] += dS[i];
        }
        const double *dz = acc + (size_t)P2 * d;
        const size_t t0 = (size_t)s * c->L + (size_t)m * B;
        for (int t = 0; t < B; ++t) {
            const size_t kv = (t0 + t) * kv_row + (size_t)g * d;
            const double *k = c->K + kv, *v = c->V + kv;
            int rc = phi_one(PHI_HEDGEHOG, k, Wg, d, F, u, phi);
            if (rc) return rc;
            for (int f = 0; f < P2; ++f) {
                double acc_f = dz[f];
                for (int e = 0; e < d; ++e) acc_f += acc[(size_t)f * d + e] * v[e];
                gphi[f] = acc_f;
            }
            phi_backward_add(k, phi, gphi, d, F, du, dW);
        }
    }
    return 0;
}

static int train_check(int n_seq, int L, int B, int Hq, int Hkv, int d, int F)
{
    if (n_seq < 0 || L < 0 || B <= 0 || Hq <= 0 || Hkv <= 0 || d <= 0 || F <= 0) return -1;
    if (Hq % Hkv != 0 || L % B != 0) return -1;
    return 0;
}

int oracle_train_forward(int n_seq, int L, int B, int Hq, int Hkv, int d, int F,
                         const double *Q, const double *K, const double *V,
                         const double *W, const double *alpha, double *O, int n_threads)
{
    if (train_check(n_seq, L, B, Hq, Hkv, d, F) || !W) return -1;
    train_ctx c;
    memset(&c, 0, sizeof c);
    c.n_seq = n_seq; c.L = L; c.B = B; c.Hq = Hq; c.Hkv = Hkv; c.d = d; c.F = F;
    c.Q = Q; c.K = K; c.V = V; c.W = W; c.alpha = alpha; c.O = O;
    const size_t P2 = 2u * (size_t)F;
    return fanout(train_fwd_unit, &c, (long)n_seq * Hq, n_threads,
                  P2 * d + 2 * P2 + (size_t)F + 2 * (size_t)d);
}

/* dW [Hkv][d][F] and dalpha [Hq] of sum(dO * O); dalpha_h = dw_h * w_h (1 - w_h). */
int oracle_train_backward(int n_seq, int L, int B, int Hq, int Hkv, int d, int F,
                          const double *Q, const double *K, const double *V,
                          const double *W, const double *alpha, const double *dO,
                          double *dW, double *dalpha, int n_threads)
{
    if (train_check(n_seq, L, B, Hq, Hkv, d, F) || !W || !dO || !dW || !dalpha) return -1;
    const size_t P2 = 2u * (size_t)F, st = P2 * d + P2;
    const int n_blk = B > 0 ? L / B : 0;
    train_ctx c;
    memset(&c, 0, sizeof c);
    c.n_seq = n_seq; c.L = L; c.B = B; c.Hq = Hq; c.Hkv = Hkv; c.d = d; c.F = F;
    c.Q = Q; c.K = K; c.V = V; c.W = W; c.alpha = alpha; c.dO = dO;
    c.dW_part = (double *)calloc((size_t)n_seq * Hkv * d * F + 1, sizeof(double));
    c.dw_part = (double *)calloc((size_t)n_seq * Hq + 1, sizeof(double));
    if (!c.dW_part || !c.dw_part) { free(c.dW_part); free(c.dw_part); return -1; }
    int rc = fanout(train_bwd_unit, &c, (long)n_seq * Hkv, n_threads,
                    2 * (size_t)n_blk * st + 2 * P2 + 4 * (size_t)d + 2 * (size_t)F + st);
    if (rc == 0) {
        for (int g = 0; g < Hkv; ++g)
            for (size_t i = 0; i < (size_t)d * F; ++i) {
                double a = 0.0;
                for (int s = 0; s < n_seq; ++s) a += c.dW_part[((size_t)s * Hkv + g) * d * F + i];
                dW[(size_t)g * d * F + i] = a;
            }
        for (int h = 0; h < Hq; ++h) {
            const double w = gate(alpha[h]);
            double a = 0.0;
            for (int s = 0; s < n_seq; ++s) a += c.dw_part[(size_t)s * Hq + h];
            dalpha[h] = a * w * (1.0 - w);
        }
    }
    free(c.dW_part);
    free(c.dw_part);
    return rc;
}
