/*
 * acespec_oracle.c -- plain, slow float64 CPU reference of the AceSpec
 * verify / sparsify / state-cache path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  It shares no code,
 * header or constant with the CUDA library; both read their inputs from the
 * seeded generator package and nothing else.
 *
 * Every function restates the definition it follows, step by step and in the
 * paper's order; there is no blocking, fusion or reordering.  Speculative
 * sampling itself is not written out in the paper: it cites Chen et al.'s
 * modified rejection sampling (Sec. II-A) whose output is identical in
 * distribution to the target model, and its roles (cloud accept test, first
 * rejection index pi, residual resample, sparse downlink, branch cache) are
 * described in Sec. III-B, Sec. III-C and Algorithm 1.  The standard form of
 * that scheme is used:
 *
 *   1. warp:      y = z / T,  pi_x = exp(y_x - max y) / sum exp(y - max y)
 *   2. nucleus:   order ids by (z desc, id asc); keep the shortest prefix
 *                 whose cumulative pi-mass reaches top_p (top_p >= 1 keeps
 *                 every id); p_x = pi_x / mass(prefix) inside, 0 outside
 *   3. accept:    a_i = [u_i < min(1, p_i(x~_i) / q_i(x~_i))]
 *   4. pi_b:      first i with a_i = 0, else K           (Sec. III-B)
 *   5. residual:  r = max(0, p_pi - q_pi) (r = p_K when pi = K, the bonus);
 *                 token = smallest j with sum_{x<=j} r_x > u_K * sum r.
 *                 For a valid draft distribution (q >= 0) r is 0 wherever
 *                 p = 0, so q is read, and checked for NaN or negative
 *                 values, only where p > 0.
 *   6. payload:   first k ids of the step-2 order with p > 0, their p, and
 *                 tail = 1 - sum of those p          (Sec. III-B, Sec. V-C)
 *   7. branches:  per depth d, ids != x~_d with q > 0 ordered by
 *                 (q desc, id asc), first F_d, prob q / (1 - q(x~_d))
 *                                                     (Sec. III-C, Alg. 1)
 *   8. lookup:    key w = (pi, token) -> slot, -1 miss, -2 full accept
 *                                                     (Sec. III-B, Alg. 1)
 *   9. sparse resample on the edge from the payload of row pi alone
 *                 (Alg. 1 RESAMPLE; see orc_resample_sparse)
 *
 * Sums use Neumaier compensation in float64; sorting uses the C library's
 * qsort as the sorting primitive.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_ROW_NONFINITE 1 /* NaN / +inf logits, or every logit is -inf */
#define ORC_ROW_BAD_Q 2     /* draft probability invalid where it is read */

/* ---------------------------------------------------------------------- */
/* compensated summation                                                   */
typedef struct {
    double s, c;
} nsum;

static void nadd(nsum *a, double x) {
    double t = a->s + x;
    if (fabs(a->s) >= fabs(x))
        a->c += (a->s - t) + x;
    else
        a->c += (x - t) + a->s;
    a->s = t;
}
static double nval(const nsum *a) { return a->s + a->c; }

/* ---------------------------------------------------------------------- */
/* ordering by (value desc, id asc)                                        */
typedef struct {
    double v;
    int32_t id;
} item;

static int cmp_desc_id_asc(const void *a, const void *b) {
    const item *x = (const item *)a, *y = (const item *)b;
    if (x->v > y->v) return -1;
    if (x->v < y->v) return 1;
    return (x->id > y->id) - (x->id < y->id);
}

/* ---------------------------------------------------------------------- */
/* one target row: steps 1 and 2                                           */
typedef struct {
    int V;
    item *it;      /* scratch for the sort                         */
    int32_t *order;/* ids in (z desc, id asc) order                */
    int32_t *rank; /* rank[id] = position of id in `order`         */
    double *pi;    /* softmax(z / T)                               */
    double *p;     /* nucleus-renormalised distribution            */
} rowbuf;

static int rowbuf_init(rowbuf *rb, int V) {
    rb->V = V;
    rb->it = (item *)malloc(sizeof(item) * (size_t)V);
    rb->order = (int32_t *)malloc(sizeof(int32_t) * (size_t)V);
    rb->rank = (int32_t *)malloc(sizeof(int32_t) * (size_t)V);
    rb->pi = (double *)malloc(sizeof(double) * (size_t)V);
    rb->p = (double *)malloc(sizeof(double) * (size_t)V);
    return rb->it && rb->order && rb->rank && rb->pi && rb->p;
}
static void rowbuf_free(rowbuf *rb) {
    free(rb->it); free(rb->order); free(rb->rank); free(rb->pi); free(rb->p);
}

typedef struct {
    int status;
    int n_nuc;       /* size of the nucleus prefix                 */
    double cum_prev; /* cumulative pi-mass before the crossing id  */
    double cum_at;   /* cumulative pi-mass including it            */
} rowinfo;

/* Steps 1-2 for one row of V logits. */
static rowinfo warp_row(const float *z, int V, double T, double top_p, rowbuf *rb) {
    rowinfo ri = {0, 0, NAN, NAN};
    /* step 1: y = z / T, pi = exp(y - max y) / sum */
    double m = -INFINITY;
    for (int x = 0; x < V; ++x) {
        double zx = (double)z[x];
        if (isnan(zx) || zx == INFINITY) { ri.status = ORC_ROW_NONFINITE; return ri; }
        double y = zx / T;
        if (y > m) m = y;
    }
    if (m == -INFINITY) { ri.status = ORC_ROW_NONFINITE; return ri; }
    nsum s = {0, 0};
    for (int x = 0; x < V; ++x) {
        double e = exp((double)z[x] / T - m);
        rb->pi[x] = e;
        nadd(&s, e);
    }
    double S = nval(&s);
    for (int x = 0; x < V; ++x) rb->pi[x] /= S;

    /* step 2: order by (z desc, id asc), shortest prefix with mass >= top_p */
    for (int x = 0; x < V; ++x) { rb->it[x].v = (double)z[x]; rb->it[x].id = x; }
    qsort(rb->it, (size_t)V, sizeof(item), cmp_desc_id_asc);
    for (int i = 0; i < V; ++i) { rb->order[i] = rb->it[i].id; rb->rank[rb->it[i].id] = i; }
    int n_finite = 0;
    for (int i = 0; i < V; ++i) if ((double)z[rb->order[i]] > -INFINITY) n_finite = i + 1;

    int n = n_finite;
    if (top_p < 1.0) {
        nsum c = {0, 0};
        for (int i = 0; i < n_finite; ++i) {
            double before = nval(&c);
            nadd(&c, rb->pi[rb->order[i]]);
            if (nval(&c) >= top_p) {
                n = i + 1;
                ri.cum_prev = before;
                ri.cum_at = nval(&c);
                break;
            }
        }
    }
    nsum mass = {0, 0};
    for (int i = 0; i < n; ++i) nadd(&mass, rb->pi[rb->order[i]]);
    double M = nval(&mass);
    for (int x = 0; x < V; ++x) rb->p[x] = 0.0;
    for (int i = 0; i < n; ++i) rb->p[rb->order[i]] = rb->pi[rb->order[i]] / M;
    ri.n_nuc = n;
    return ri;
}

/* Step 6: sparse payload of one warped row. */
static void payload_row(const rowbuf *rb, const rowinfo *ri, int k, int32_t *ids, double *probs,
                        double *tail) {
    nsum t = {0, 0};
    int j = 0;
    for (int i = 0; i < ri->n_nuc && j < k; ++i) {
        int32_t x = rb->order[i];
        if (!(rb->p[x] > 0.0)) continue;
        ids[j] = x;
        probs[j] = rb->p[x];
        nadd(&t, rb->p[x]);
        ++j;
    }
    for (; j < k; ++j) { ids[j] = -1; probs[j] = 0.0; }
    *tail = 1.0 - nval(&t);
}

/* ---------------------------------------------------------------------- */
/* Public: sparsify `rows` independent rows (steps 1, 2, 6).               */
int orc_sparsify(const float *z, int rows, int V, double T, double top_p, int k, int32_t *topk_ids,
                 double *topk_probs, double *tail, int32_t *row_status, double *cum_prev,
                 double *cum_at, int32_t *n_nuc) {
    int err = 0;
#pragma omp parallel
    {
        rowbuf rb;
        int ok = rowbuf_init(&rb, V);
        if (!ok) {
#pragma omp atomic write
            err = 1;
        }
#pragma omp for schedule(dynamic, 1)
        for (int r = 0; r < rows; ++r) {
            if (!ok) continue;
            rowinfo ri = warp_row(z + (size_t)r * V, V, T, top_p, &rb);
            row_status[r] = ri.status;
            if (cum_prev) cum_prev[r] = ri.cum_prev;
            if (cum_at) cum_at[r] = ri.cum_at;
            if (n_nuc) n_nuc[r] = ri.n_nuc;
            if (ri.status) {
                for (int j = 0; j < k; ++j) { topk_ids[(size_t)r * k + j] = -1; topk_probs[(size_t)r * k + j] = 0.0; }
                tail[r] = 1.0;
            } else {
                payload_row(&rb, &ri, k, topk_ids + (size_t)r * k, topk_probs + (size_t)r * k, tail + r);
            }
        }
        rowbuf_free(&rb);
    }
    return err;
}

/* ---------------------------------------------------------------------- */
/* Public: verify B sequences (steps 1-6).
 *   z  [B, K+1, V]  target logits (bf16 inputs are widened to float exactly)
 *   q  [B, K, V]    draft probabilities
 *   xt [B, K]       draft tokens,  u [B, K+1] uniforms
 * Outputs: accept_len [B], out_token [B]; when k > 0 the payload
 * [B, K+1, k] ids / probs and tail [B, K+1]; row_status [B, K+1].
 * Diagnostics used by the parity tests to flag near-ties (any may be NULL):
 *   ratio [B, K]       p(x~) / q(x~) at every draft position
 *   cum_prev, cum_at   [B, K+1] cumulative mass around the nucleus crossing
 *   n_nuc [B, K+1]     nucleus sizes
 *   res_target, res_cj, res_cjm1, res_sum  [B]  u_K * sum r, C_j, C_{j-1}, sum r
 */
int orc_verify(const float *z, const float *q, const int32_t *xt, const float *u, int B, int K,
               int V, double T, double top_p, int k, int32_t *accept_len, int32_t *out_token,
               int32_t *topk_ids, double *topk_probs, double *tail, int32_t *row_status,
               double *ratio, double *cum_prev, double *cum_at, int32_t *n_nuc, double *res_target,
               double *res_cj, double *res_cjm1, double *res_sum) {
    int err = 0;
    const int R = K + 1;
#pragma omp parallel
    {
        rowbuf rb;
        int ok = rowbuf_init(&rb, V);
        double *pK = (double *)malloc(sizeof(double) * (size_t)V * (size_t)R);
        double *r = (double *)malloc(sizeof(double) * (size_t)V);
        int *acc = (int *)malloc(sizeof(int) * (size_t)(K > 0 ? K : 1));
        int *st = (int *)malloc(sizeof(int) * (size_t)R);
        if (!ok || !pK || !r || !acc || !st) {
#pragma omp atomic write
            err = 1;
            ok = 0;
        }
#pragma omp for schedule(dynamic, 1)
        for (int b = 0; b < B; ++b) {
            if (!ok) continue;
            const float *zb = z + (size_t)b * R * V;
            const float *qb = q + (size_t)b * K * V;
            /* steps 1-3 on every row of the sequence */
            for (int i = 0; i < R; ++i) {
                size_t row = (size_t)b * R + i;
                rowinfo ri = warp_row(zb + (size_t)i * V, V, T, top_p, &rb);
                st[i] = ri.status;
                if (cum_prev) cum_prev[row] = ri.cum_prev;
                if (cum_at) cum_at[row] = ri.cum_at;
                if (n_nuc) n_nuc[row] = ri.n_nuc;
                memcpy(pK + (size_t)i * V, rb.p, sizeof(double) * (size_t)V);
                if (k > 0) {
                    if (ri.status) {
                        for (int j = 0; j < k; ++j) { topk_ids[row * k + j] = -1; topk_probs[row * k + j] = 0.0; }
                        tail[row] = 1.0;
                    } else {
                        payload_row(&rb, &ri, k, topk_ids + row * k, topk_probs + row * k, tail + row);
                    }
                }
                if (i < K) {
                    int32_t x = xt[(size_t)b * K + i];
                    double px = ri.status ? 0.0 : rb.p[x];
                    double qx = (double)qb[(size_t)i * V + x];
                    double rt;
                    if (!(qx > 0.0)) {
                        st[i] |= ORC_ROW_BAD_Q;
                        rt = 0.0;
                    } else {
                        rt = px / qx;
                    }
                    if (ri.status & ORC_ROW_NONFINITE) rt = 0.0;
                    if (ratio) ratio[(size_t)b * K + i] = rt;
                    double ui = (double)u[(size_t)b * R + i];
                    acc[i] = ui < fmin(1.0, rt);
                }
            }
            /* step 4: first rejection */
            int pi = K;
            for (int i = 0; i < K; ++i) if (!acc[i]) { pi = i; break; }
            accept_len[b] = pi;

            /* step 5: residual (pi < K) or bonus (pi == K) on row pi */
            const double *pp = pK + (size_t)pi * V;
            int32_t tok = -1;
            double tgt = NAN, cj = NAN, cjm1 = NAN, sr = NAN;
            if (!(st[pi] & ORC_ROW_NONFINITE)) {
                int bad = 0;
                if (pi < K) {
                    const float *qr = qb + (size_t)pi * V;
                    for (int x = 0; x < V; ++x) {
                        if (!(pp[x] > 0.0)) { r[x] = 0.0; continue; }  /* max(0, 0 - q), q >= 0 */
                        double qx = (double)qr[x];
                        if (isnan(qx) || qx < 0.0) { bad = 1; break; }
                        double d = pp[x] - qx;
                        r[x] = d > 0.0 ? d : 0.0;
                    }
                } else {
                    for (int x = 0; x < V; ++x) r[x] = pp[x];
                }
                if (bad) {
                    st[pi] |= ORC_ROW_BAD_Q;
                } else {
                    nsum s = {0, 0};
                    for (int x = 0; x < V; ++x) nadd(&s, r[x]);
                    sr = nval(&s);
                    if (!(sr > 0.0)) { /* p <= q everywhere: fall back to p */
                        for (int x = 0; x < V; ++x) r[x] = pp[x];
                        nsum s2 = {0, 0};
                        for (int x = 0; x < V; ++x) nadd(&s2, r[x]);
                        sr = nval(&s2);
                    }
                    tgt = (double)u[(size_t)b * R + K] * sr;
                    nsum c = {0, 0};
                    int last_pos = -1;
                    for (int x = 0; x < V; ++x) {
                        double before = nval(&c);
                        nadd(&c, r[x]);
                        if (r[x] > 0.0) last_pos = x;
                        if (nval(&c) > tgt) { tok = x; cj = nval(&c); cjm1 = before; break; }
                    }
                    if (tok < 0) tok = last_pos;
                }
            }
            out_token[b] = tok;
            if (res_target) res_target[b] = tgt;
            if (res_cj) res_cj[b] = cj;
            if (res_cjm1) res_cjm1[b] = cjm1;
            if (res_sum) res_sum[b] = sr;
            for (int i = 0; i < R; ++i) row_status[(size_t)b * R + i] = st[i];
        }
        rowbuf_free(&rb);
        free(pK); free(r); free(acc); free(st);
    }
    return err;
}

/* ---------------------------------------------------------------------- */
/* Public: probabilistic state cache build (step 7).
 *   q [B, K, V], xt [B, K], F [K] -> branch_tok / branch_prob [B, sum F],
 * depth d occupying columns [off_d, off_d + F_d), off = exclusive prefix of F.
 */
int orc_cache_build(const float *q, const int32_t *xt, const int32_t *F, int B, int K, int V,
                    int32_t *branch_tok, double *branch_prob) {
    int err = 0;
    int total = 0;
    for (int d = 0; d < K; ++d) total += F[d];
#pragma omp parallel
    {
        item *it = (item *)malloc(sizeof(item) * (size_t)V);
        if (!it) {
#pragma omp atomic write
            err = 1;
        }
#pragma omp for schedule(dynamic, 1)
        for (int row = 0; row < B * K; ++row) {
            if (!it) continue;
            int b = row / K, d = row % K;
            int off = 0;
            for (int j = 0; j < d; ++j) off += F[j];
            const float *qr = q + (size_t)row * V;
            int32_t xd = xt[row];
            int n = 0;
            for (int x = 0; x < V; ++x) {
                double qx = (double)qr[x];
                if (x == xd || !(qx > 0.0)) continue;
                it[n].v = qx; it[n].id = x; ++n;
            }
            qsort(it, (size_t)n, sizeof(item), cmp_desc_id_asc);
            double denom = 1.0 - (double)qr[xd];
            int32_t *bt = branch_tok + (size_t)b * total + off;
            double *bp = branch_prob + (size_t)b * total + off;
            for (int j = 0; j < F[d]; ++j) {
                if (j < n && denom > 0.0) { bt[j] = it[j].id; bp[j] = it[j].v / denom; }
                else { bt[j] = -1; bp[j] = 0.0; }
            }
        }
        free(it);
    }
    return err;
}

/* Public: cache lookup (step 8). slot = off[pi] + j when branch j of depth
 * pi holds `token`; -1 on a miss (or an invalid token); -2 when pi == K. */
int orc_cache_lookup(const int32_t *branch_tok, const int32_t *F, int B, int K,
                     const int32_t *accept_len, const int32_t *token, int32_t *slot) {
    int total = 0;
    for (int d = 0; d < K; ++d) total += F[d];
    for (int b = 0; b < B; ++b) {
        int pi = accept_len[b];
        if (pi == K) { slot[b] = -2; continue; }
        slot[b] = -1;
        if (pi < 0 || pi > K || token[b] < 0) continue;
        int off = 0;
        for (int j = 0; j < pi; ++j) off += F[j];
        for (int j = 0; j < F[pi]; ++j)
            if (branch_tok[(size_t)b * total + off + j] == token[b]) { slot[b] = off + j; break; }
    }
    return 0;
}

/* ---------------------------------------------------------------------- */
/* Public: steps 1-2 alone: the nucleus-renormalised target p of `rows`    */
/* rows (used to measure how far the sparse resample is from the exact    */
/* residual).  p_out [rows, V]; row_status [rows].                          */
int orc_warp(const float *z, int rows, int V, double T, double top_p, double *p_out,
             int32_t *row_status) {
    int err = 0;
#pragma omp parallel
    {
        rowbuf rb;
        int ok = rowbuf_init(&rb, V);
        if (!ok) {
#pragma omp atomic write
            err = 1;
        }
#pragma omp for schedule(dynamic, 1)
        for (int r = 0; r < rows; ++r) {
            if (!ok) continue;
            rowinfo ri = warp_row(z + (size_t)r * V, V, T, top_p, &rb);
            row_status[r] = ri.status;
            for (int x = 0; x < V; ++x) p_out[(size_t)r * V + x] = ri.status ? 0.0 : rb.p[x];
        }
        rowbuf_free(&rb);
    }
    return err;
}

/* ---------------------------------------------------------------------- */
/* Public: edge-side resample from the sparse payload (Alg. 1             */
/* RESAMPLE(P^_target, Q); Sec. III-B: the cloud returns pi and the        */
/* partial target distribution of row pi, the edge draws the token).       */
/*                                                                         */
/* The edge knows p only on the payload ids I (probs p^_I) and the mass    */
/* tau = tail outside them.  Reading used here:                            */
/*   pi < K:  p^(x) = p^_x on I; outside I the mass tau is spread like the */
/*            draft, p^(x) = tau * q(x) / q_rest, q_rest = sum_{x not in I} */
/*            q(x) (0 when q_rest = 0).  r^ = max(0, p^ - q), i.e.          */
/*            max(0, p^_x - q(x)) on I and q(x) * max(0, tau/q_rest - 1)    */
/*            outside.  When tau = 0 the draft row is read on I only.       */
/*   pi = K:  the bonus draw uses the payload alone, r^ = p^_I.             */
/*   Token: smallest id j with sum_{x <= j} r^(x) > u[b, K] * sum r^ (the   */
/*   exact path's rule).  If sum r^ = 0 the draw uses p^_I.                 */
/* When the nucleus of row pi fits in the payload, tau = 0 and p^ = p:     */
/* the result is the exact residual draw.                                   */
/*                                                                         */
/* Inputs: accept_len [B]; the payload of every row, ids [B, K+1, k],       */
/* probs [B, K+1, k] (float32), tail [B, K+1]; row_status [B, K+1] of the   */
/* verification; q [B, K, V]; u [B, K+1].  Outputs: token [B] (-1 when row  */
/* pi is NONFINITE, the payload is empty, or q is NaN/negative where it is  */
/* read: status [B] gets ORC_ROW_NONFINITE / ORC_ROW_BAD_Q).                */
/* Diagnostics (may be NULL): res_target, res_cj, res_cjm1, res_sum [B] as  */
/* in orc_verify; dist [B, V] the normalised distribution drawn from.       */
int orc_resample_sparse(const int32_t *accept_len, const int32_t *ids, const float *probs,
                        const float *tail, const int32_t *row_status, const float *q,
                        const float *u, int B, int K, int V, int k, int32_t *token,
                        int32_t *status, double *res_target, double *res_cj, double *res_cjm1,
                        double *res_sum, double *dist) {
    int err = 0;
#pragma omp parallel
    {
        double *r = (double *)malloc(sizeof(double) * (size_t)V);
        char *in = (char *)malloc((size_t)V);
        if (!r || !in) {
#pragma omp atomic write
            err = 1;
        }
#pragma omp for schedule(dynamic, 1)
        for (int b = 0; b < B; ++b) {
            if (!r || !in) continue;
            const int R1 = K + 1;
            const int pi = accept_len[b];
            const size_t row = (size_t)b * R1 + (size_t)pi;
            int32_t tok = -1;
            int st = 0;
            double tgt = NAN, cj = NAN, cjm1 = NAN, sr = NAN;
            if (pi < 0 || pi > K || (row_status[row] & ORC_ROW_NONFINITE)) {
                st = ORC_ROW_NONFINITE;
            } else {
                const int32_t *I = ids + row * (size_t)k;
                const float *P = probs + row * (size_t)k;
                const double tau = (double)tail[row];
                for (int x = 0; x < V; ++x) { r[x] = 0.0; in[x] = 0; }
                int n_in = 0;
                for (int j = 0; j < k; ++j)
                    if (I[j] >= 0 && I[j] < V) { in[I[j]] = 1; ++n_in; }
                const float *qr = pi < K ? q + ((size_t)b * K + (size_t)pi) * (size_t)V : NULL;
                int bad = 0;
                if (qr) {
                    /* payload ids: max(0, p^ - q) */
                    for (int j = 0; j < k; ++j) {
                        int32_t x = I[j];
                        if (x < 0 || x >= V) continue;
                        double qx = (double)qr[x];
                        if (isnan(qx) || qx < 0.0) { bad = 1; break; }
                        double d = (double)P[j] - qx;
                        r[x] = d > 0.0 ? d : 0.0;
                    }
                    /* outside the payload: the tail spread like q */
                    if (!bad && tau > 0.0) {
                        nsum qs = {0, 0};
                        for (int x = 0; x < V && !bad; ++x) {
                            double qx = (double)qr[x];
                            if (isnan(qx) || qx < 0.0) { bad = 1; break; }
                            if (!in[x]) nadd(&qs, qx);
                        }
                        double q_rest = nval(&qs);
                        double g = q_rest > 0.0 ? tau / q_rest - 1.0 : 0.0;
                        if (!bad && g > 0.0)
                            for (int x = 0; x < V; ++x)
                                if (!in[x]) r[x] = (double)qr[x] * g;
                    }
                } else {
                    for (int j = 0; j < k; ++j)
                        if (I[j] >= 0 && I[j] < V) r[I[j]] = (double)P[j];
                }
                if (bad) {
                    st = ORC_ROW_BAD_Q;
                } else if (n_in > 0) {
                    nsum s = {0, 0};
                    for (int x = 0; x < V; ++x) nadd(&s, r[x]);
                    sr = nval(&s);
                    if (!(sr > 0.0)) { /* p^ <= q wherever it is known: draw from p^_I */
                        for (int x = 0; x < V; ++x) r[x] = 0.0;
                        for (int j = 0; j < k; ++j)
                            if (I[j] >= 0 && I[j] < V) r[I[j]] = (double)P[j];
                        nsum s2 = {0, 0};
                        for (int x = 0; x < V; ++x) nadd(&s2, r[x]);
                        sr = nval(&s2);
                    }
                    if (sr > 0.0) {
                        tgt = (double)u[(size_t)b * R1 + K] * sr;
                        nsum c = {0, 0};
                        int last_pos = -1;
                        for (int x = 0; x < V; ++x) {
                            double before = nval(&c);
                            nadd(&c, r[x]);
                            if (r[x] > 0.0) last_pos = x;
                            if (nval(&c) > tgt) { tok = x; cj = nval(&c); cjm1 = before; break; }
                        }
                        if (tok < 0) tok = last_pos;
                    }
                }
            }
            token[b] = tok;
            if (status) status[b] = st;
            if (res_target) res_target[b] = tgt;
            if (res_cj) res_cj[b] = cj;
            if (res_cjm1) res_cjm1[b] = cjm1;
            if (res_sum) res_sum[b] = sr;
            if (dist)
                for (int x = 0; x < V; ++x)
                    dist[(size_t)b * V + x] = (tok >= 0 && sr > 0.0) ? r[x] / sr : 0.0;
        }
        free(r);
        free(in);
    }
    return err;
}

/* ---------------------------------------------------------------------- */
/* Public: probability that the branch cache recovers the sequence (Sec.  */
/* III-C, Eq. for P_hit): given the drafted chain x~ and the branches      */
/* branch_tok [B, sum F], the only randomness left is the uniforms.  With  */
/* a_i = min(1, p_i(x~_i) / q_i(x~_i)) (0 when q_i(x~_i) <= 0) and R_i the */
/* mass of norm(max(0, p_i - q_i)) (of p_i when that is all zero) on the   */
/* branches of depth i:                                                    */
/*   hit_prob[b]   = sum_{i<K} (prod_{j<i} a_j)(1 - a_i) R_i + prod a_j    */
/*                   (first rejection at i and its token cached, or the   */
/*                   whole chain accepted: lookup slot >= 0 or -2);        */
/*   paper_prob[b] = prod_{i<K} (a_i + (1 - a_i) R_i), the product form of */
/*                   Sec. IV-C, evaluated with the same a_i and R_i.       */
int orc_hit_prob(const float *z, const float *q, const int32_t *xt, int B, int K, int V, double T,
                 double top_p, const int32_t *branch_tok, const int32_t *F, double *hit_prob,
                 double *paper_prob) {
    int err = 0;
    int total = 0;
    for (int d = 0; d < K; ++d) total += F[d];
#pragma omp parallel
    {
        rowbuf rb;
        int ok = rowbuf_init(&rb, V);
        if (!ok) {
#pragma omp atomic write
            err = 1;
        }
#pragma omp for schedule(dynamic, 1)
        for (int b = 0; b < B; ++b) {
            if (!ok) continue;
            double survive = 1.0, hit = 0.0, prod = 1.0;
            int off = 0;
            for (int i = 0; i < K; ++i) {
                const float *zr = z + ((size_t)b * (K + 1) + i) * (size_t)V;
                const float *qr = q + ((size_t)b * K + i) * (size_t)V;
                rowinfo ri = warp_row(zr, V, T, top_p, &rb);
                double a = 0.0, R = 0.0;
                if (!ri.status) {
                    int32_t x = xt[(size_t)b * K + i];
                    if (x >= 0 && x < V && (double)qr[x] > 0.0) {
                        double ratio = rb.p[x] / (double)qr[x];
                        a = ratio < 1.0 ? ratio : 1.0;
                    }
                    nsum rs = {0, 0};
                    for (int y = 0; y < V; ++y) {
                        double d = rb.p[y] - (double)qr[y];
                        nadd(&rs, d > 0.0 ? d : 0.0);
                    }
                    double Rt = nval(&rs);
                    nsum cs = {0, 0};
                    for (int j = 0; j < F[i]; ++j) {
                        int32_t y = branch_tok[(size_t)b * total + off + j];
                        if (y < 0 || y >= V) continue;
                        double d = rb.p[y] - (double)qr[y];
                        nadd(&cs, Rt > 0.0 ? (d > 0.0 ? d : 0.0) : rb.p[y]);
                    }
                    R = Rt > 0.0 ? nval(&cs) / Rt : nval(&cs);
                }
                hit += survive * (1.0 - a) * R;
                survive *= a;
                prod *= a + (1.0 - a) * R;
                off += F[i];
            }
            hit_prob[b] = hit + survive;
            if (paper_prob) paper_prob[b] = prod;
        }
        rowbuf_free(&rb);
    }
    return err;
}

int orc_num_threads(void) {
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* Threads of the parallel loops that follow (n >= 1); returns the previous
 * count.  The results do not depend on it (every loop is over independent
 * rows or sequences). */
int orc_set_threads(int n) {
#ifdef _OPENMP
    const int prev = omp_get_max_threads();
    if (n >= 1) omp_set_num_threads(n);
    return prev;
#else
    (void)n;
    return 1;
#endif
}
