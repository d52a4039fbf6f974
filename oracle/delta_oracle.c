/*
 * delta_oracle.c — fp64 CPU oracle for the Delta Attention prefill.
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the plain, slow, obviously correct
 * statement of what the prefill computes.  It is used by tests/, by
 * __graft_entry__.smoke() and by the CPU-baseline leg of bench.py, and by
 * nothing else.  It shares no code, header, table or helper with the CUDA
 * path in paper_2505_11254_gb300/csrc/.
 *
 * Definitions followed (paper: "Delta Attention: Fast and Accurate Sparse
 * Attention Inference by Delta Correction", arXiv 2505.11254):
 *   - Eq. 1: attention output of row i is softmax(q_i K^T / sqrt(d)) V over the
 *     causal key set C(i) = {0..i} (causality: key j visible iff j <= i).
 *   - Sec. 2/3, StreamingLLM sparse attention f*: the key set is the union of
 *     the first n_sink keys and the last `window` keys ending at i,
 *     W(i) = { j <= i : j < n_sink  or  j >= i - window + 1 }; the softmax is
 *     normalised over W(i) only (the normaliser "T" of Lemma 1).
 *   - Eq. 4: sampled query rows are i = k*gamma (0-based rows, k = 0,1,...).
 *   - Alg. 1 / Eq. 6: A*V for every row, ~AV (dense) for sampled rows,
 *     Delta_k = ~AV_k - (A*V)_{k gamma}, and the output is
 *     A^V_i = (A*V)_i + Delta_{floor(i/gamma)} ("repeat(Delta, gamma)").
 *   - Eq. 5 ("recompute" ablation): only sampled rows are replaced by dense
 *     rows; every other row keeps its sparse output.
 *   - Appendix "Implementation Details": an optional block of final query rows
 *     is computed densely (dense tail); the Delta-corrected part before it is
 *     unchanged.
 *   - Appendix "Restatement and proof of Lemma 1": the error bound, evaluated
 *     here for the actual selected set W(i) (the proof holds for any set).
 *   - Appendix "Interpolation" and Alg. 2: smoothing of the Delta corrections
 *     (linear interpolation, EMA, alpha-beta-gamma filter) before they are
 *     added to the sparse rows.
 *   - Eq. 2: decoding after the prefill, one new query per sequence attending
 *     densely over the cached keys with its own key appended.
 *   - Sec. 2 (positional encodings applied to Q and K before Eq. 1): RoPE in
 *     the rotate-half form, channel c paired with c + d/2, angle
 *     pos * base^(-2c/d).
 *
 * Readings of the paper used here (each also listed in the design notes):
 *   - Rows are 0-based and the sample for row i is row floor(i/gamma)*gamma,
 *     which never lies after i (Eq. 4 / Eq. 6 with the 1-based off-by-one
 *     resolved in favour of Alg. 1's repeat(Delta, gamma)).
 *   - The window is inclusive of the diagonal: keys i-window+1 .. i.
 *   - Sinks and window overlap as a set union (a key is counted once).
 *   - GQA: q-head h reads kv-head floor(h / (Hq/Hkv)).
 *   - Inputs are bf16 bit patterns widened exactly to double; all arithmetic
 *     is double precision.
 *
 * Layout: Q [B,Hq,N,d], K and V [B,Hkv,N,d], row-major, contiguous.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

#define SET_CAUSAL 0
#define SET_SPARSE 1

/* Deliberately broken variants, built only by tests/test_oracle_mutants.py to
 * show that the pins reject each plausible mistake.  0 = the real oracle. */
#ifndef ORACLE_MUTANT
#define ORACLE_MUTANT 0
#endif
#define MUTANT(n) (ORACLE_MUTANT == (n))

typedef struct {
    const uint16_t *Q, *K, *V;
    int B, Hq, Hkv, d, n_sink, gamma;
    int64_t N, window;
} problem;

/* bf16 -> double is exact: the bf16 bits are the high half of an fp32. */
static double bf16_to_double(uint16_t h)
{
    uint32_t u = (uint32_t)h << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Is key j in the key set of query row i?  (Eq. 1 causality; StreamingLLM
 * sink + sliding window for the sparse set.) */
static int member(const problem *p, int set, int64_t i, int64_t j)
{
    if (j > i) return 0;                       /* causal */
    if (set == SET_CAUSAL) return 1;
    return (j < p->n_sink + MUTANT(1)) || (j >= i - p->window + 1 - MUTANT(2));
}

/*
 * One attention row: out[c] = sum_j p_j v_j[c] with p = softmax over the key
 * set of tau * q_i . k_j, tau = 1/sqrt(d).  `prob` holds the explicit softmax
 * vector (length >= i+1).  Returns |sum_j p_j - 1|.
 */
static double attn_row(const problem *p, int b, int h, int64_t i, int set,
                       double *out, double *prob)
{
    const int d = p->d;
    const int g = MUTANT(3) ? h % p->Hkv : h / (p->Hq / p->Hkv);
    const uint16_t *q  = p->Q + (((int64_t)b * p->Hq + h) * p->N + i) * d;
    const uint16_t *Kh = p->K + ((int64_t)b * p->Hkv + g) * p->N * d;
    const uint16_t *Vh = p->V + ((int64_t)b * p->Hkv + g) * p->N * d;
    const double tau = MUTANT(4) ? 1.0 : 1.0 / sqrt((double)d);

    double m = -INFINITY;
    for (int64_t j = 0; j <= i; ++j) {
        if (!member(p, set, i, j)) continue;
        double s = 0.0;
        for (int c = 0; c < d; ++c)
            s += bf16_to_double(q[c]) *
                 bf16_to_double(MUTANT(8) ? Kh[(int64_t)c * p->N + j] : Kh[j * d + c]);
        s *= tau;
        prob[j] = s;
        if (s > m) m = s;
    }
    double Z = 0.0;
    for (int64_t j = 0; j <= i; ++j) {
        if (!member(p, set, i, j)) continue;
        prob[j] = exp(prob[j] - m);
        Z += prob[j];
    }
    double total = 0.0;
    for (int64_t j = 0; j <= i; ++j) {
        if (!member(p, set, i, j)) continue;
        prob[j] /= Z;
        total += prob[j];
    }
    for (int c = 0; c < d; ++c) out[c] = 0.0;
    for (int64_t j = 0; j <= i; ++j) {
        if (!member(p, set, i, j)) continue;
        for (int c = 0; c < d; ++c)
            out[c] += prob[j] * bf16_to_double(Vh[j * d + c]);
    }
    return fabs(total - 1.0);
}

/* ------------------------------------------------------------------------ */
/* A tiny work-sharing pool: items 0..n_items-1 handed out by an atomic      */
/* counter to nthreads pthreads.                                             */

typedef void (*item_fn)(void *ctx, int64_t item, double *prob, double *dev);

typedef struct {
    item_fn fn;
    void *ctx;
    int64_t n_items;
    int64_t next;        /* shared counter */
    int64_t prob_len;
    int d;
    double max_dev;      /* per-thread result, merged under lock */
    pthread_mutex_t lock;
    int failed;
} pool;

static void *pool_worker(void *arg)
{
    pool *P = (pool *)arg;
    double *prob = (double *)malloc(sizeof(double) * (size_t)(P->prob_len > 0 ? P->prob_len : 1));
    double dev = 0.0;
    if (!prob) {
        pthread_mutex_lock(&P->lock);
        P->failed = 1;
        pthread_mutex_unlock(&P->lock);
    } else {
        for (;;) {
            int64_t it = __atomic_fetch_add(&P->next, 1, __ATOMIC_RELAXED);
            if (it >= P->n_items) break;
            P->fn(P->ctx, it, prob, &dev);
        }
    }
    pthread_mutex_lock(&P->lock);
    if (dev > P->max_dev) P->max_dev = dev;
    pthread_mutex_unlock(&P->lock);
    free(prob);
    return NULL;
}

static int run_pool(item_fn fn, void *ctx, int64_t n_items, int64_t prob_len, int d,
                    int nthreads, double *max_dev)
{
    pool P;
    P.fn = fn; P.ctx = ctx; P.n_items = n_items; P.next = 0;
    P.prob_len = prob_len; P.d = d; P.max_dev = 0.0; P.failed = 0;
    pthread_mutex_init(&P.lock, NULL);
    if (nthreads <= 0) nthreads = (int)sysconf(_SC_NPROCESSORS_ONLN);
    if (nthreads < 1) nthreads = 1;
    if (nthreads > 512) nthreads = 512;
    pthread_t tid[512];
    int started = 0;
    for (int t = 0; t < nthreads; ++t) {
        if (pthread_create(&tid[t], NULL, pool_worker, &P) != 0) break;
        ++started;
    }
    if (started == 0) pool_worker(&P);
    for (int t = 0; t < started; ++t) pthread_join(tid[t], NULL);
    pthread_mutex_destroy(&P.lock);
    if (max_dev && P.max_dev > *max_dev) *max_dev = P.max_dev;
    return P.failed ? -1 : 0;
}

static int valid_problem(const problem *p)
{
    if (!p->Q || !p->K || !p->V) return 0;
    if (p->B < 1 || p->Hq < 1 || p->Hkv < 1 || p->d < 1 || p->N < 1) return 0;
    if (p->Hq % p->Hkv != 0) return 0;
    if (p->gamma < 1 || p->window < 1 || p->n_sink < 0) return 0;
    return 1;
}

/* ------------------------------------------------------------------------ */
/* Full prefill over a box of (b, h, rows), in the order of Alg. 1.          */

typedef struct {
    const problem *p;
    int b0, b1, h0, h1;
    int64_t r0, r1;          /* rows [r0, r1) */
    int64_t k0, k1;          /* samples [k0, k1) covering those rows */
    double *S;               /* [nb, nh, r1-r0, d]   sparse output A*V   */
    double *D;               /* [nb, nh, k1-k0, d]   dense output ~AV    */
    double *A;               /* [nb, nh, r1-r0, d]   corrected output    */
    int mode;                /* OUT_DELTA, OUT_RECOMPUTE */
    int64_t tail_dense;      /* rows >= N - tail_dense are dense */
} box_ctx;

#define OUT_DELTA 0
#define OUT_RECOMPUTE 1

static void box_sparse_item(void *vc, int64_t it, double *prob, double *dev)
{
    box_ctx *c = (box_ctx *)vc;
    const int64_t nr = c->r1 - c->r0;
    const int nh = c->h1 - c->h0;
    int64_t r = it % nr;
    int64_t bh = it / nr;
    int b = c->b0 + (int)(bh / nh), h = c->h0 + (int)(bh % nh);
    double *out = c->S + (bh * nr + r) * c->p->d;
    double e = attn_row(c->p, b, h, c->r0 + r, SET_SPARSE, out, prob);
    if (e > *dev) *dev = e;
}

static void box_dense_item(void *vc, int64_t it, double *prob, double *dev)
{
    box_ctx *c = (box_ctx *)vc;
    const int64_t nk = c->k1 - c->k0;
    const int nh = c->h1 - c->h0;
    int64_t k = it % nk;
    int64_t bh = it / nk;
    int b = c->b0 + (int)(bh / nh), h = c->h0 + (int)(bh % nh);
    double *out = c->D + (bh * nk + k) * c->p->d;
    double e = attn_row(c->p, b, h, (c->k0 + k) * c->p->gamma,
                        MUTANT(6) ? SET_SPARSE : SET_CAUSAL, out, prob);
    if (e > *dev) *dev = e;
}

static void box_tail_item(void *vc, int64_t it, double *prob, double *dev)
{
    /* rows of the dense tail block: A^V_i = dense row i */
    box_ctx *c = (box_ctx *)vc;
    const problem *p = c->p;
    const int64_t nr = c->r1 - c->r0;
    const int nh = c->h1 - c->h0;
    int64_t r = it % nr;
    int64_t bh = it / nr;
    int64_t i = c->r0 + r;
    if (i < p->N - c->tail_dense) return;
    int b = c->b0 + (int)(bh / nh), h = c->h0 + (int)(bh % nh);
    double *out = c->A + (bh * nr + r) * p->d;
    double e = attn_row(p, b, h, i, SET_CAUSAL, out, prob);
    if (e > *dev) *dev = e;
}

/*
 * oracle_delta_attn_box — Delta Attention (Alg. 1, Eq. 6) for batches
 * [b0,b1), q-heads [h0,h1) and rows [r0,r1).
 *
 *   S_out  (nullable) [b1-b0, h1-h0, r1-r0, d]: sparse output (A*V)_i
 *   D_out  (nullable) [b1-b0, h1-h0, k1-k0, d]: dense output ~AV_k of the
 *          samples k in [floor(r0/gamma), floor((r1-1)/gamma)]
 *   A_out  (required) [b1-b0, h1-h0, r1-r0, d]: corrected output A^V_i
 *   mode   0 = Delta (Eq. 6), 1 = recompute (Eq. 5)
 *   tail_dense: rows i >= N - tail_dense are replaced by their dense rows
 *          (appendix "Implementation Details"); 0 = none.
 *   max_dev (nullable): max over all softmax vectors of |sum p - 1|.
 * Returns 0, or -1 on invalid arguments / allocation failure.
 */
int oracle_delta_attn_box(const uint16_t *Q, const uint16_t *K, const uint16_t *V,
                          int B, int Hq, int Hkv, int64_t N, int d,
                          int n_sink, int64_t window, int gamma,
                          int b0, int b1, int h0, int h1, int64_t r0, int64_t r1,
                          int mode, int64_t tail_dense,
                          double *S_out, double *D_out, double *A_out,
                          double *max_dev, int nthreads)
{
    problem p = {Q, K, V, B, Hq, Hkv, d, n_sink, gamma, N, window};
    if (!valid_problem(&p) || !A_out) return -1;
    if (b0 < 0 || b1 > B || b0 >= b1 || h0 < 0 || h1 > Hq || h0 >= h1) return -1;
    if (r0 < 0 || r1 > N || r0 >= r1) return -1;
    if (mode != OUT_DELTA && mode != OUT_RECOMPUTE) return -1;
    if (tail_dense < 0) return -1;

    box_ctx c;
    c.p = &p; c.b0 = b0; c.b1 = b1; c.h0 = h0; c.h1 = h1; c.r0 = r0; c.r1 = r1;
    c.k0 = r0 / gamma; c.k1 = (r1 - 1) / gamma + 1;
    c.mode = mode; c.tail_dense = tail_dense;
    const int64_t nbh = (int64_t)(b1 - b0) * (h1 - h0);
    const int64_t nr = r1 - r0, nk = c.k1 - c.k0;

    double *S = S_out ? S_out : (double *)malloc(sizeof(double) * (size_t)(nbh * nr * d));
    double *D = D_out ? D_out : (double *)malloc(sizeof(double) * (size_t)(nbh * nk * d));
    double *Ss = (double *)malloc(sizeof(double) * (size_t)(nbh * nk * d));
    if (!S || !D || !Ss) {
        if (!S_out) free(S);
        if (!D_out) free(D);
        free(Ss);
        return -1;
    }
    c.S = S; c.D = D; c.A = A_out;
    double dev = 0.0;
    int rc = 0;

    /* Alg. 1, step 1: A*V <- f*(Q, K, V) for every row of the box. */
    rc |= run_pool(box_sparse_item, &c, nbh * nr, N, d, nthreads, &dev);
    /* Alg. 1, steps 2-3: ~AV <- f(~Q, K, V), ~Q the rows k*gamma (Eq. 4). */
    rc |= run_pool(box_dense_item, &c, nbh * nk, N, d, nthreads, &dev);

    /* (A*V) at the sampled rows delta = {i : i mod gamma == 0}.  A sample may
     * lie before r0 (the group of row r0 starts there); compute it directly. */
    {
        double *prob = (double *)malloc(sizeof(double) * (size_t)N);
        if (!prob) rc = -1;
        for (int64_t bh = 0; prob && bh < nbh; ++bh) {
            int b = b0 + (int)(bh / (h1 - h0)), h = h0 + (int)(bh % (h1 - h0));
            for (int64_t k = c.k0; k < c.k1; ++k) {
                int64_t i = k * gamma;
                double *dst = Ss + (bh * nk + (k - c.k0)) * d;
                if (i >= r0 && i < r1) {
                    memcpy(dst, S + (bh * nr + (i - r0)) * d, sizeof(double) * (size_t)d);
                } else {
                    double e = attn_row(&p, b, h, i, SET_SPARSE, dst, prob);
                    if (e > dev) dev = e;
                }
            }
        }
        free(prob);
    }

    /* Alg. 1, steps 4-5: Delta <- ~AV - (A*V)_delta, then
     * A^V = A*V + repeat(Delta, gamma) (Eq. 6), or the Eq. 5 recompute form. */
    for (int64_t bh = 0; bh < nbh; ++bh) {
        for (int64_t r = 0; r < nr; ++r) {
            int64_t i = r0 + r;
            int64_t k = i / gamma;
            const double *s  = S  + (bh * nr + r) * d;
            const double *dn = D  + (bh * nk + (k - c.k0)) * d;
            const double *ss = Ss + (bh * nk + (k - c.k0)) * d;
            double *a = A_out + (bh * nr + r) * d;
            int sampled = (i % gamma) == 0;
            for (int e = 0; e < d; ++e) {
                double delta = dn[e] - (MUTANT(7) ? s[e] : ss[e]);
                if (mode == OUT_DELTA)
                    a[e] = MUTANT(5) ? s[e] - delta : s[e] + delta;
                else
                    a[e] = s[e] + (sampled ? delta : 0.0);
            }
        }
    }

    /* Dense tail block (appendix "Implementation Details"). */
    if (tail_dense > 0)
        rc |= run_pool(box_tail_item, &c, nbh * nr, N, d, nthreads, &dev);

    if (max_dev) *max_dev = dev;
    if (!S_out) free(S);
    if (!D_out) free(D);
    free(Ss);
    return rc;
}

/* Whole problem: all batches, heads and rows. */
int oracle_delta_attn(const uint16_t *Q, const uint16_t *K, const uint16_t *V,
                      int B, int Hq, int Hkv, int64_t N, int d,
                      int n_sink, int64_t window, int gamma,
                      double *S_out, double *D_out, double *A_out,
                      double *max_dev, int nthreads)
{
    return oracle_delta_attn_box(Q, K, V, B, Hq, Hkv, N, d, n_sink, window, gamma,
                                 0, B, 0, Hq, 0, N, OUT_DELTA, 0,
                                 S_out, D_out, A_out, max_dev, nthreads);
}

/* ------------------------------------------------------------------------ */
/* Individual rows, for spot checks at sizes where the full oracle is slow.  */

typedef struct {
    const problem *p;
    const int64_t *bhi;          /* n x 3: b, h, i */
    double *S, *Dk, *Sk, *A;     /* each n x d */
} rows_ctx;

static void rows_item(void *vc, int64_t it, double *prob, double *dev)
{
    rows_ctx *c = (rows_ctx *)vc;
    const problem *p = c->p;
    const int d = p->d;
    int b = (int)c->bhi[3 * it], h = (int)c->bhi[3 * it + 1];
    int64_t i = c->bhi[3 * it + 2];
    int64_t ks = (i / p->gamma) * p->gamma;           /* the sample row of i */
    double *s = c->S + it * d, *dk = c->Dk + it * d, *sk = c->Sk + it * d, *a = c->A + it * d;
    double e;
    e = attn_row(p, b, h, i, SET_SPARSE, s, prob);  if (e > *dev) *dev = e;
    e = attn_row(p, b, h, ks, MUTANT(6) ? SET_SPARSE : SET_CAUSAL, dk, prob);
    if (e > *dev) *dev = e;
    e = attn_row(p, b, h, ks, SET_SPARSE, sk, prob);
    if (e > *dev) *dev = e;
    for (int x = 0; x < d; ++x) {                                  /* Eq. 6 */
        double delta = dk[x] - (MUTANT(7) ? s[x] : sk[x]);
        a[x] = MUTANT(5) ? s[x] - delta : s[x] + delta;
    }
}

/*
 * oracle_rows — for each (b, h, i) in bhi[n][3]: the sparse row S_i, the dense
 * row and the sparse row of its sample floor(i/gamma)*gamma, and the Eq. 6
 * output A^V_i.  Each output array is [n, d].
 */
int oracle_rows(const uint16_t *Q, const uint16_t *K, const uint16_t *V,
                int B, int Hq, int Hkv, int64_t N, int d,
                int n_sink, int64_t window, int gamma,
                const int64_t *bhi, int64_t n,
                double *S_row, double *D_sample, double *S_sample, double *A_row,
                double *max_dev, int nthreads)
{
    problem p = {Q, K, V, B, Hq, Hkv, d, n_sink, gamma, N, window};
    if (!valid_problem(&p) || !bhi || n < 0) return -1;
    if (!S_row || !D_sample || !S_sample || !A_row) return -1;
    for (int64_t t = 0; t < n; ++t) {
        if (bhi[3 * t] < 0 || bhi[3 * t] >= B) return -1;
        if (bhi[3 * t + 1] < 0 || bhi[3 * t + 1] >= Hq) return -1;
        if (bhi[3 * t + 2] < 0 || bhi[3 * t + 2] >= N) return -1;
    }
    rows_ctx c = {&p, bhi, S_row, D_sample, S_sample, A_row};
    double dev = 0.0;
    int rc = run_pool(rows_item, &c, n, N, d, nthreads, &dev);
    if (max_dev) *max_dev = dev;
    return rc;
}

/* ------------------------------------------------------------------------ */
/* Lemma 1 (appendix restatement), for the sampled row i = k*gamma and the   */
/* actual selected set W(i).                                                  */
/*   Delta      = a^T v - a*^T v                 (dense minus sparse)        */
/*   head       = sum_{j in C(i) \ W(i)} a_j v_j (the omitted part)          */
/*   lhs[c]     = | Delta[c] - head[c] |                                     */
/*   rhs[c]     = H / (H + T) * max_{j in W(i)} | v_j[c] |                   */
/* with H = sum over omitted keys of e^{s_j}, T = sum over W(i) of e^{s_j}.  */
int oracle_lemma1(const uint16_t *Q, const uint16_t *K, const uint16_t *V,
                  int B, int Hq, int Hkv, int64_t N, int d,
                  int n_sink, int64_t window, int gamma,
                  int b, int h, int64_t k, double *lhs, double *rhs, double *h_frac)
{
    problem p = {Q, K, V, B, Hq, Hkv, d, n_sink, gamma, N, window};
    if (!valid_problem(&p) || !lhs || !rhs) return -1;
    if (b < 0 || b >= B || h < 0 || h >= Hq || k < 0 || k * (int64_t)gamma >= N) return -1;
    const int64_t i = k * (int64_t)gamma;
    const int g = h / (Hq / Hkv);
    const uint16_t *q  = Q + (((int64_t)b * Hq + h) * N + i) * d;
    const uint16_t *Kh = K + ((int64_t)b * Hkv + g) * N * d;
    const uint16_t *Vh = V + ((int64_t)b * Hkv + g) * N * d;
    const double tau = 1.0 / sqrt((double)d);

    double *e = (double *)malloc(sizeof(double) * (size_t)(i + 1));
    double *dense = (double *)calloc((size_t)d, sizeof(double));
    double *sparse = (double *)calloc((size_t)d, sizeof(double));
    double *head = (double *)calloc((size_t)d, sizeof(double));
    double *vmax = (double *)calloc((size_t)d, sizeof(double));
    if (!e || !dense || !sparse || !head || !vmax) {
        free(e); free(dense); free(sparse); free(head); free(vmax);
        return -1;
    }
    double m = -INFINITY;
    for (int64_t j = 0; j <= i; ++j) {
        double s = 0.0;
        for (int c = 0; c < d; ++c)
            s += bf16_to_double(q[c]) * bf16_to_double(Kh[j * d + c]);
        e[j] = s * tau;
        if (e[j] > m) m = e[j];
    }
    double H = 0.0, T = 0.0;
    for (int64_t j = 0; j <= i; ++j) {
        e[j] = exp(e[j] - m);             /* common shift cancels in H/(H+T) */
        if (member(&p, SET_SPARSE, i, j)) T += e[j]; else H += e[j];
    }
    for (int64_t j = 0; j <= i; ++j) {
        const int in_w = member(&p, SET_SPARSE, i, j);
        const double a = e[j] / (H + T);                 /* full softmax   */
        const double as = in_w ? e[j] / T : 0.0;         /* sparse softmax */
        for (int c = 0; c < d; ++c) {
            double v = bf16_to_double(Vh[j * d + c]);
            dense[c] += a * v;
            sparse[c] += as * v;
            if (!in_w) head[c] += a * v;
            if ((in_w || MUTANT(14)) && fabs(v) > vmax[c]) vmax[c] = fabs(v);
        }
    }
    for (int c = 0; c < d; ++c) {
        double delta = dense[c] - sparse[c];
        lhs[c] = fabs(delta - head[c]);
        rhs[c] = H / (H + T) * vmax[c];
    }
    if (h_frac) *h_frac = H / (H + T);
    free(e); free(dense); free(sparse); free(head); free(vmax);
    return 0;
}

/* ------------------------------------------------------------------------ */
/* Delta smoothing (appendix "Interpolation", Alg. 2).                       */
/*                                                                          */
/* With y_i = Delta_{floor(i/gamma)} (Alg. 1's repeat: one vector per row),  */
/* the correction added to row i becomes                                    */
/*   SMOOTH_LINEAR: (1 - b_i) Delta_k + b_i Delta_{k+1}, k = floor(i/gamma),  */
/*       b_i = (i - k gamma) / gamma, rising linearly from 0 at the sample    */
/*       towards 1 at the next one; the last group has no next sample and     */
/*       keeps Delta_k;                                                       */
/*   SMOOTH_EMA (c1 = beta): over the expanded rows, e_0 = y_0 and            */
/*       e_i = (1 - beta) e_{i-1} + beta y_i;                                 */
/*   SMOOTH_ABG (c1, c2, c3 = the filter's alpha, beta, gamma): Alg. 2 run    */
/*       over the Delta vectors themselves (its output has one vector per    */
/*       Delta), elementwise: position p = Delta_0, velocity v = 0,           */
/*       acceleration a = 0, output Delta_0 for sample 0; at each later       */
/*       sample predict p + v + a/2 and v + a, take the residual r = Delta_k  */
/*       minus the predicted position, correct p, v and a by alpha r, beta r  */
/*       and gamma r, and output p; row i then takes the output of its sample */
/*       floor(i/gamma), as in Alg. 1's repeat.                               */
/* SMOOTH_NONE gives y_i itself (Eq. 6).                                     */

#define SMOOTH_NONE 0
#define SMOOTH_LINEAR 1
#define SMOOTH_EMA 2
#define SMOOTH_ABG 3

/*
 * oracle_smooth_seq — the smoothed corrections of rows [r0, r1) of one
 * (batch, head), computed by running the recurrence from row 0.
 *   delta [n_k, d]: Delta_0 .. Delta_{n_k - 1}; n_k must reach the last sample
 *         the rows use (one more for SMOOTH_LINEAR, unless it is the last of
 *         the n_s samples).
 *   corr  [r1 - r0, d].
 * Returns 0, or -1 on invalid arguments.
 */
int oracle_smooth_seq(int kind, double c1, double c2, double c3,
                      const double *delta, int64_t n_k, int d, int64_t n_s, int gamma,
                      int64_t r0, int64_t r1, double *corr)
{
    if (!delta || !corr || d < 1 || gamma < 1 || n_s < 1 || r0 < 0 || r1 <= r0) return -1;
    if (kind < SMOOTH_NONE || kind > SMOOTH_ABG) return -1;
    int64_t last = (r1 - 1) / gamma;                 /* last sample used */
    if (last >= n_s) return -1;
    if (kind == SMOOTH_LINEAR && last + 1 < n_s) last += 1;
    if (n_k <= last) return -1;

    double *filt = NULL;                             /* Alg. 2 output per sample */
    if (kind == SMOOTH_ABG) {
        filt = (double *)malloc(sizeof(double) * (size_t)((last + 1) * d));
        if (!filt) return -1;
        for (int e = 0; e < d; ++e) {
            double p = delta[e], v = 0.0, a = 0.0;
            filt[e] = p;
            for (int64_t k = 1; k <= last; ++k) {
                const double p_pred = p + v + 0.5 * a;
                const double v_pred = v + a;
                const double r = delta[k * d + e] - p_pred;
                p = p_pred + c1 * r;
                v = v_pred + (MUTANT(10) ? c1 : c2) * r;
                a = a + c3 * r;
                filt[k * d + e] = p;
            }
        }
    }
    for (int e = 0; e < d; ++e) {
        double ema = delta[e];                       /* EMA state */
        for (int64_t i = 0; i < r1; ++i) {
            const int64_t k = i / gamma;
            const double y = delta[k * d + e];
            double out;
            if (kind == SMOOTH_NONE) {
                out = y;
            } else if (kind == SMOOTH_LINEAR) {
                const double b = (double)(i - k * gamma + MUTANT(11)) / (double)gamma;
                const double next = (k + 1 < n_s) ? delta[(k + 1) * d + e] : y;
                out = (1.0 - b) * y + b * next;
            } else if (kind == SMOOTH_EMA) {
                if (i > 0)
                    ema = MUTANT(9) ? c1 * ema + (1.0 - c1) * y : (1.0 - c1) * ema + c1 * y;
                out = ema;
            } else {
                out = filt[k * d + e];
            }
            if (i >= r0) corr[(i - r0) * d + e] = out;
        }
    }
    free(filt);
    return 0;
}

typedef struct {
    const problem *p;
    int b0, h0, nh;
    int64_t nk;              /* samples 0..nk-1 per (b, h) */
    double *delta;           /* [nbh, nk, d] */
} smooth_delta_ctx;

static void smooth_delta_item(void *vc, int64_t it, double *prob, double *dev)
{
    /* Delta_k = (dense row k gamma) - (sparse row k gamma), Alg. 1 */
    smooth_delta_ctx *c = (smooth_delta_ctx *)vc;
    const problem *p = c->p;
    const int d = p->d;
    int64_t k = it % c->nk, bh = it / c->nk;
    int b = c->b0 + (int)(bh / c->nh), h = c->h0 + (int)(bh % c->nh);
    double *dst = c->delta + it * d;
    double *sp = (double *)malloc(sizeof(double) * (size_t)d);
    if (!sp) return;
    double e = attn_row(p, b, h, k * p->gamma, SET_CAUSAL, dst, prob);
    if (e > *dev) *dev = e;
    e = attn_row(p, b, h, k * p->gamma, SET_SPARSE, sp, prob);
    if (e > *dev) *dev = e;
    for (int x = 0; x < d; ++x) dst[x] -= sp[x];
    free(sp);
}

/*
 * oracle_delta_attn_smoothed — Eq. 6 with smoothed corrections over a box of
 * batches [b0,b1), q-heads [h0,h1) and rows [r0,r1):
 *   A_out[b, h, i] = S_i + corr_i (corr from oracle_smooth_seq), and rows
 *   i >= N - tail_dense replaced by their dense rows.
 * Returns 0, or -1 on invalid arguments / allocation failure.
 */
int oracle_delta_attn_smoothed(const uint16_t *Q, const uint16_t *K, const uint16_t *V,
                               int B, int Hq, int Hkv, int64_t N, int d,
                               int n_sink, int64_t window, int gamma,
                               int b0, int b1, int h0, int h1, int64_t r0, int64_t r1,
                               int kind, double c1, double c2, double c3, int64_t tail_dense,
                               double *A_out, double *max_dev, int nthreads)
{
    problem p = {Q, K, V, B, Hq, Hkv, d, n_sink, gamma, N, window};
    if (!valid_problem(&p) || !A_out) return -1;
    if (b0 < 0 || b1 > B || b0 >= b1 || h0 < 0 || h1 > Hq || h0 >= h1) return -1;
    if (r0 < 0 || r1 > N || r0 >= r1 || tail_dense < 0) return -1;
    if (kind < SMOOTH_NONE || kind > SMOOTH_ABG) return -1;
    const int64_t n_s = (N + gamma - 1) / gamma;
    int64_t nk = (r1 - 1) / gamma + 1;
    if (kind == SMOOTH_LINEAR && nk < n_s) nk += 1;
    const int nh = h1 - h0;
    const int64_t nbh = (int64_t)(b1 - b0) * nh, nr = r1 - r0;

    double *delta = (double *)malloc(sizeof(double) * (size_t)(nbh * nk * d));
    double *S = (double *)malloc(sizeof(double) * (size_t)(nbh * nr * d));
    double *corr = (double *)malloc(sizeof(double) * (size_t)(nr * d));
    int rc = (delta && S && corr) ? 0 : -1;
    double dev = 0.0;
    if (rc == 0) {
        smooth_delta_ctx dc = {&p, b0, h0, nh, nk, delta};
        rc |= run_pool(smooth_delta_item, &dc, nbh * nk, N, d, nthreads, &dev);
        box_ctx sc;
        memset(&sc, 0, sizeof sc);
        sc.p = &p; sc.b0 = b0; sc.b1 = b1; sc.h0 = h0; sc.h1 = h1; sc.r0 = r0; sc.r1 = r1;
        sc.S = S; sc.A = A_out; sc.tail_dense = tail_dense;
        rc |= run_pool(box_sparse_item, &sc, nbh * nr, N, d, nthreads, &dev);
        for (int64_t bh = 0; rc == 0 && bh < nbh; ++bh) {
            rc |= oracle_smooth_seq(kind, c1, c2, c3, delta + bh * nk * d, nk, d, n_s, gamma, r0, r1, corr);
            for (int64_t x = 0; x < nr * d; ++x) A_out[bh * nr * d + x] = S[bh * nr * d + x] + corr[x];
        }
        if (rc == 0 && tail_dense > 0)
            rc |= run_pool(box_tail_item, &sc, nbh * nr, N, d, nthreads, &dev);
    }
    if (max_dev) *max_dev = dev;
    free(delta);
    free(S);
    free(corr);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* Decoding (Eq. 2): the query of a newly generated token attends densely    */
/* over the cache [K u k_new], [V u v_new].  The cache holds the new token's */
/* key and value at index n_keys[b] - 1, so the keys are 0 .. n_keys[b] - 1. */

typedef struct {
    const uint16_t *q, *K, *V;
    int B, Hq, Hkv, d;
    int64_t L;
    const int64_t *n_keys;
    double *out;
} decode_ctx;

static void decode_item(void *vc, int64_t it, double *prob, double *dev)
{
    decode_ctx *c = (decode_ctx *)vc;
    const int d = c->d;
    const int b = (int)(it / c->Hq), h = (int)(it % c->Hq);
    const int g = h / (c->Hq / c->Hkv);
    const uint16_t *q = c->q + it * d;
    const uint16_t *Kh = c->K + ((int64_t)b * c->Hkv + g) * c->L * d;
    const uint16_t *Vh = c->V + ((int64_t)b * c->Hkv + g) * c->L * d;
    const int64_t n = c->n_keys[b] - MUTANT(12);
    const double tau = 1.0 / sqrt((double)d);
    double *out = c->out + it * d;
    double m = -INFINITY;
    for (int64_t j = 0; j < n; ++j) {
        double s = 0.0;
        for (int x = 0; x < d; ++x) s += bf16_to_double(q[x]) * bf16_to_double(Kh[j * d + x]);
        prob[j] = s * tau;
        if (prob[j] > m) m = prob[j];
    }
    double Z = 0.0;
    for (int64_t j = 0; j < n; ++j) {
        prob[j] = exp(prob[j] - m);
        Z += prob[j];
    }
    for (int x = 0; x < d; ++x) out[x] = 0.0;
    double total = 0.0;
    for (int64_t j = 0; j < n; ++j) {
        const double pj = prob[j] / Z;
        total += pj;
        for (int x = 0; x < d; ++x) out[x] += pj * bf16_to_double(Vh[j * d + x]);
    }
    const double e = n > 0 ? fabs(total - 1.0) : 0.0;
    if (e > *dev) *dev = e;
}

/*
 * oracle_decode — q [B,Hq,d] (one new token per sequence), K and V caches
 * [B,Hkv,L,d], n_keys[b] in [1, L] valid keys of sequence b; writes
 * out [B,Hq,d].  Returns 0, or -1 on invalid arguments.
 */
int oracle_decode(const uint16_t *q, const uint16_t *K, const uint16_t *V, int B, int Hq, int Hkv, int64_t L,
                  int d, const int64_t *n_keys, double *out, double *max_dev, int nthreads)
{
    if (!q || !K || !V || !n_keys || !out || B < 1 || Hq < 1 || Hkv < 1 || d < 1 || L < 1) return -1;
    if (Hq % Hkv != 0) return -1;
    for (int b = 0; b < B; ++b)
        if (n_keys[b] < 1 || n_keys[b] > L) return -1;
    decode_ctx c = {q, K, V, B, Hq, Hkv, d, L, n_keys, out};
    double dev = 0.0;
    int rc = run_pool(decode_item, &c, (int64_t)B * Hq, L, d, nthreads, &dev);
    if (max_dev) *max_dev = dev;
    return rc;
}

/* ------------------------------------------------------------------------ */
/* RoPE (Sec. 2: positional encodings applied to Q and K before attention).  */
/* Rotate-half form: for c < d/2 the pair (x_c, x_{c+d/2}) at position pos   */
/* is rotated by the angle pos * base^(-2c/d):                               */
/*   x'_c       = x_c cos - x_{c+d/2} sin                                    */
/*   x'_{c+d/2} = x_{c+d/2} cos + x_c sin                                    */
/* Row r of X [rows_total = B*H*N, d] has position pos0 + (r mod N).         */

static double rope_angle(int64_t pos, int c, int d, double base)
{
    return (double)pos * pow(base, -2.0 * (double)c / (double)d);
}

/* fp64 result (no rounding): out [B*H*N, d] doubles. */
int oracle_rope_f64(const uint16_t *X, int64_t rows_total, int64_t N, int d, int64_t pos0, double base,
                    double *out)
{
    if (!X || !out || rows_total < 1 || N < 1 || d < 2 || (d & 1) || base <= 0.0) return -1;
    const int h = d / 2;
    for (int64_t r = 0; r < rows_total; ++r) {
        const int64_t pos = pos0 + r % N;
        const uint16_t *x = X + r * d;
        double *o = out + r * d;
        for (int c = 0; c < h; ++c) {
            const double a = rope_angle(pos, c, d, base);
            const double ca = cos(a), sa = sin(a);
            const double x0 = bf16_to_double(x[c]), x1 = bf16_to_double(x[c + h]);
            const double sg = MUTANT(13) ? -1.0 : 1.0;
            o[c] = x0 * ca - sg * x1 * sa;
            o[c + h] = x1 * ca + sg * x0 * sa;
        }
    }
    return 0;
}

/* double -> bf16 bits, rounded once to the nearest 8-significant-bit value,
 * ties to even (the rotated values enter the attention as bf16, as the
 * unrotated inputs do).  For the normal range of bf16. */
static uint16_t double_to_bf16(double v)
{
    if (v == 0.0) return signbit(v) ? 0x8000u : 0u;
    int e;
    const double m = frexp(v, &e);                 /* v = m 2^e, 0.5 <= |m| < 1 */
    const double r = nearbyint(ldexp(m, 8));       /* 8 significant bits, ties to even */
    const float f = (float)ldexp(r, e - 8);        /* exact: 8 bits fit a float */
    uint32_t u;
    memcpy(&u, &f, sizeof u);
    return (uint16_t)(u >> 16);
}

/* bf16 result: out bits [B*H*N, d]. */
int oracle_rope_bf16(const uint16_t *X, int64_t rows_total, int64_t N, int d, int64_t pos0, double base,
                     uint16_t *out)
{
    if (!out) return -1;
    double *tmp = (double *)malloc(sizeof(double) * (size_t)d);
    if (!tmp) return -1;
    int rc = 0;
    for (int64_t r = 0; r < rows_total && rc == 0; ++r) {
        rc = oracle_rope_f64(X + r * d, 1, 1, d, pos0 + r % N, base, tmp);
        for (int c = 0; c < d && rc == 0; ++c) out[r * d + c] = double_to_bf16(tmp[c]);
    }
    free(tmp);
    return rc;
}
