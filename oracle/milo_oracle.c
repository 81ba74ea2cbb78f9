/*
 * milo_oracle.c -- plain, slow, fp64 CPU reference for MILO
 * ("Efficient Many-shot In-Context Learning with Block-wise Low-rank
 * Compression").
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the oracle that the CUDA path is
 * checked against.  Only the test suite, the smoke check and the benchmark's
 * CPU-baseline leg may load it.  It shares no code, header, table or helper
 * with the CUDA library, and the CUDA library never calls it.
 *
 * What it computes, each part written as the paper defines it:
 *   - mo_attention_dense:     Alg. 1 (Stage 2) reconstruction K^_b = C_b P_b
 *                             of every stored block (Eq. 3 with Sigma folded
 *                             into C), followed by exact softmax attention
 *                             (Eq. 1) over [blocks..., query's own tail].
 *   - mo_attention_dense_rope: the same, for factors of pre-RoPE keys (the
 *                             observation of Sec. 3: keys are compressed
 *                             before the rotary position embedding), so every
 *                             reconstructed prefix key is rotated to its
 *                             position before the scores.
 *   - mo_rope_rotate:         that rotation of a set of rows.
 *   - mo_attention_rankspace: the same attention written in rank space,
 *                             q.K^_b^T = (q P_b^T) C_b^T and
 *                             p V^_b   = (p C_b) P_b.  A second, independent
 *                             routine used only to cross-check the first.
 *   - mo_svd_jacobi:          SVD of one block (Eq. 3) by one-sided
 *                             (Hestenes) Jacobi rotations, the textbook method
 *                             of Demmel & Veselic (1992).
 *   - mo_spectral_information: H_i(r) of Eq. 5.
 *   - mo_allocate_ranks:      greedy marginal-gain rank allocation of Eq. 7
 *                             for the budget problem of Eq. 6.
 *   - mo_compression_ratio:   rho of Eq. 4 as an exact integer fraction.
 *   - mo_kv_cache_bytes:      M of Eq. 2 (fp16 dense KV footprint).
 *
 * Readings of points the paper leaves open (each also listed in the design
 * notes): Sigma is folded into the coefficient matrix C = A Sigma; K and V
 * are decomposed separately (Eq. 3, not the joint form printed in Alg. 1);
 * the allocation maximises Eq. 6 (Alg. 1 prints argmin); the softmax scale is
 * 1/sqrt(head_dim); query head h reads KV head h / (Hq / Hkv); a query attends
 * to every stored block in table order and then to all of its own tail
 * tokens, with no mask.  RoPE (where asked for): dimension i pairs with
 * i + d/2 (the half-split form of the Qwen2.5 models), pair i turns by the
 * angle pos * theta^(-2i/d) counter-clockwise, block b's token t sits at
 * position block_pos[b] + t (by default the block's start in the
 * concatenated prefix), and q and the dense tails arrive already rotated.
 *
 * Parity status: every function here is pinned by CPU tests (brute force,
 * closed forms, invariants, numpy.linalg.svd, exhaustive search).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

enum {
    MO_OK = 0,
    MO_ERR_ARG = 1,
    MO_ERR_NOMEM = 2,
    MO_ERR_INFEASIBLE = 3,
    MO_ERR_NOCONV = 4
};

enum { MO_F64 = 0, MO_BF16 = 1 };

/* bf16 is the top half of an IEEE binary32; widening to fp64 is exact. */
static double bf16_bits_to_f64(uint16_t h)
{
    uint32_t u = ((uint32_t)h) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

/* Copy `count` elements starting at element `off` of a bf16 or fp64 array
 * into fp64. */
static void fetch(int dtype, const void *base, int64_t off, int64_t count,
                  double *dst)
{
    if (dtype == MO_F64) {
        memcpy(dst, (const double *)base + off, (size_t)count * sizeof(double));
    } else {
        const uint16_t *p = (const uint16_t *)base + off;
        for (int64_t i = 0; i < count; ++i) dst[i] = bf16_bits_to_f64(p[i]);
    }
}

int mo_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void mo_set_threads(int n)
{
#ifdef _OPENMP
    if (n > 0) omp_set_num_threads(n);
#else
    (void)n;
#endif
}

/* ------------------------------------------------------------------------ */
/* Shared argument checks for both attention forms.                          */
/* ------------------------------------------------------------------------ */
typedef struct {
    int dtype, batch, hq, hkv, d, nblk;
    const int32_t *blen, *rk, *rv;
    const int64_t *ock, *opk, *ocv, *opv;
    const void *arena, *q, *tk, *tv;
    const int64_t *toff;
    double scale;
    double rope_theta;        /* > 0: prefix keys are pre-RoPE (rotate them) */
    const int64_t *block_pos; /* [nblk] first position of each block, or NULL */
} mo_problem;

static int check_problem(const mo_problem *p, int64_t *n_prefix, int64_t *t_max)
{
    if (p->dtype != MO_F64 && p->dtype != MO_BF16) return MO_ERR_ARG;
    if (p->batch < 0 || p->hq <= 0 || p->hkv <= 0 || p->d <= 0 || p->nblk < 0)
        return MO_ERR_ARG;
    if (p->hq % p->hkv != 0) return MO_ERR_ARG;
    int64_t np = 0;
    for (int b = 0; b < p->nblk; ++b) {
        if (p->blen[b] <= 0) return MO_ERR_ARG;
        np += p->blen[b];
        for (int g = 0; g < p->hkv; ++g) {
            int i = b * p->hkv + g;
            if (p->rk[i] < 0 || p->rv[i] < 0) return MO_ERR_ARG;
            if (p->rk[i] > p->d || p->rv[i] > p->d) return MO_ERR_ARG;
        }
    }
    int64_t tm = 0;
    for (int i = 0; i < p->batch; ++i) {
        int64_t t = p->toff ? p->toff[i + 1] - p->toff[i] : 0;
        if (p->toff && i == 0 && p->toff[0] != 0) return MO_ERR_ARG;
        if (t < 0) return MO_ERR_ARG;
        if (np + t == 0) return MO_ERR_ARG; /* softmax over nothing */
        if (t > tm) tm = t;
    }
    if (tm > 0 && (!p->tk || !p->tv)) return MO_ERR_ARG;
    if (p->rope_theta > 0.0) {
        if (p->d % 2 != 0) return MO_ERR_ARG;
        if (p->block_pos)
            for (int b = 0; b < p->nblk; ++b)
                if (p->block_pos[b] < 0) return MO_ERR_ARG;
    }
    *n_prefix = np;
    *t_max = tm;
    return MO_OK;
}

static int64_t tail_len(const mo_problem *p, int i)
{
    return p->toff ? p->toff[i + 1] - p->toff[i] : 0;
}

/* Dense reconstruction X^ = C P of one stored factor pair (Eq. 3 with Sigma
 * folded into C; Alg. 1 Stage 2 "full-rank reconstruction").
 * C is n x r, P is r x d, both row-major; out is n x d. */
static void reconstruct(const double *C, const double *P, int n, int r, int d,
                        double *out)
{
    for (int t = 0; t < n; ++t) {
        double *o = out + (int64_t)t * d;
        for (int c = 0; c < d; ++c) o[c] = 0.0;
        for (int j = 0; j < r; ++j) {
            double a = C[(int64_t)t * r + j];
            const double *pr = P + (int64_t)j * d;
            for (int c = 0; c < d; ++c) o[c] += a * pr[c];
        }
    }
}

/* Rotary position embedding of n rows of width d (row t at position
 * pos0 + t, or pos[t] when pos is given): pair (i, i + d/2) turns by the
 * angle position * theta^(-2i/d),
 *   x_i       <- x_i cos a - x_{i+d/2} sin a
 *   x_{i+d/2} <- x_{i+d/2} cos a + x_i sin a. */
static void rope_rows(double *X, int n, int d, int64_t pos0, const int64_t *pos,
                      double theta)
{
    const int h = d / 2;
    for (int t = 0; t < n; ++t) {
        const double where = (double)(pos ? pos[t] : pos0 + t);
        double *x = X + (int64_t)t * d;
        for (int i = 0; i < h; ++i) {
            const double a = where * pow(theta, -2.0 * i / d);
            const double c = cos(a), s = sin(a);
            const double x0 = x[i], x1 = x[i + h];
            x[i] = x0 * c - x1 * s;
            x[i + h] = x1 * c + x0 * s;
        }
    }
}

static double dot(const double *a, const double *b, int n)
{
    double s = 0.0;
    for (int i = 0; i < n; ++i) s += a[i] * b[i];
    return s;
}

/* ------------------------------------------------------------------------ */
/* Attention, dense-reconstruction form: Alg. 1 Stage 2 followed by Eq. 1.   */
/*                                                                           */
/* For every query i, query head h (KV head g = h / G):                      */
/*   keys   = [K^_1; ...; K^_N; Ktail_i[:, g, :]]                             */
/*   values = [V^_1; ...; V^_N; Vtail_i[:, g, :]]                             */
/*   s_t = scale * <q_h, key_t>;  M = max_t s_t;  w_t = exp(s_t - M)          */
/*   out = sum_t w_t value_t / sum_t w_t                                       */
/* Two passes (all scores first, then values): no online rescaling.          */
/* ------------------------------------------------------------------------ */
static int attention_dense(const mo_problem *p, double *out, double *weights,
                           int64_t wstride)
{
    int64_t np, tmax;
    int rc = check_problem(p, &np, &tmax);
    if (rc) return rc;
    const int G = p->hq / p->hkv, d = p->d;
    const int rows = p->batch * G;
    const int64_t ncol = np + tmax;
    if (p->batch == 0) return MO_OK;

    int64_t *pos = (int64_t *)malloc(sizeof(int64_t) * (size_t)(p->nblk + 1));
    double *S = (double *)malloc(sizeof(double) * (size_t)rows * (size_t)ncol);
    double *Z = (double *)malloc(sizeof(double) * (size_t)rows);
    double *qv = (double *)malloc(sizeof(double) * (size_t)rows * (size_t)d);
    double *ob = (double *)malloc(sizeof(double) * (size_t)(p->nblk + 1) *
                                  (size_t)rows * (size_t)d);
    if (!pos || !S || !Z || !qv || !ob) {
        free(pos); free(S); free(Z); free(qv); free(ob);
        return MO_ERR_NOMEM;
    }
    pos[0] = 0;
    for (int b = 0; b < p->nblk; ++b) pos[b + 1] = pos[b] + p->blen[b];

    for (int g = 0; g < p->hkv; ++g) {
        /* query vectors of the G heads of every query that read KV head g */
        for (int i = 0; i < p->batch; ++i)
            for (int hh = 0; hh < G; ++hh)
                fetch(p->dtype, p->q, ((int64_t)i * p->hq + g * G + hh) * d, d,
                      qv + (int64_t)(i * G + hh) * d);

        /* pass 1a: scores against every reconstructed prefix key */
        int fail = 0;
#pragma omp parallel for schedule(dynamic, 1)
        for (int b = 0; b < p->nblk; ++b) {
            const int e = b * p->hkv + g, n = p->blen[b], r = p->rk[e];
            double *C = (double *)malloc(sizeof(double) * ((size_t)n * r + 1));
            double *P = (double *)malloc(sizeof(double) * ((size_t)r * d + 1));
            double *K = (double *)malloc(sizeof(double) * (size_t)n * d);
            if (!C || !P || !K) {
#pragma omp atomic write
                fail = 1;
                free(C); free(P); free(K);
                continue;
            }
            fetch(p->dtype, p->arena, p->ock[e], (int64_t)n * r, C);
            fetch(p->dtype, p->arena, p->opk[e], (int64_t)r * d, P);
            reconstruct(C, P, n, r, d, K);
            if (p->rope_theta > 0.0)
                rope_rows(K, n, d, p->block_pos ? p->block_pos[b] : pos[b], NULL,
                          p->rope_theta);
            for (int row = 0; row < rows; ++row)
                for (int t = 0; t < n; ++t)
                    S[(int64_t)row * ncol + pos[b] + t] =
                        p->scale * dot(qv + (int64_t)row * d, K + (int64_t)t * d, d);
            free(C); free(P); free(K);
        }
        if (fail) { rc = MO_ERR_NOMEM; break; }

        /* pass 1b: scores against the query's own dense tail keys */
        double *kt = (double *)malloc(sizeof(double) * (size_t)d);
        if (!kt) { rc = MO_ERR_NOMEM; break; }
        for (int i = 0; i < p->batch; ++i) {
            const int64_t T = tail_len(p, i);
            for (int64_t t = 0; t < T; ++t) {
                fetch(p->dtype, p->tk, ((p->toff[i] + t) * p->hkv + g) * d, d, kt);
                for (int hh = 0; hh < G; ++hh) {
                    const int row = i * G + hh;
                    S[(int64_t)row * ncol + np + t] =
                        p->scale * dot(qv + (int64_t)row * d, kt, d);
                }
            }
        }

        /* softmax weights, row by row: w = exp(s - max s), Z = sum w */
        for (int row = 0; row < rows; ++row) {
            const int64_t valid = np + tail_len(p, row / G);
            double *s = S + (int64_t)row * ncol;
            double M = -INFINITY;
            for (int64_t t = 0; t < valid; ++t) if (s[t] > M) M = s[t];
            double z = 0.0;
            for (int64_t t = 0; t < valid; ++t) { s[t] = exp(s[t] - M); z += s[t]; }
            Z[row] = z;
        }

        /* pass 2a: per-block weighted sums of reconstructed values */
#pragma omp parallel for schedule(dynamic, 1)
        for (int b = 0; b < p->nblk; ++b) {
            const int e = b * p->hkv + g, n = p->blen[b], r = p->rv[e];
            double *C = (double *)malloc(sizeof(double) * ((size_t)n * r + 1));
            double *P = (double *)malloc(sizeof(double) * ((size_t)r * d + 1));
            double *V = (double *)malloc(sizeof(double) * (size_t)n * d);
            double *o = ob + (int64_t)b * rows * d;
            if (!C || !P || !V) {
#pragma omp atomic write
                fail = 1;
                free(C); free(P); free(V);
                continue;
            }
            fetch(p->dtype, p->arena, p->ocv[e], (int64_t)n * r, C);
            fetch(p->dtype, p->arena, p->opv[e], (int64_t)r * d, P);
            reconstruct(C, P, n, r, d, V);
            for (int row = 0; row < rows; ++row) {
                double *orow = o + (int64_t)row * d;
                const double *w = S + (int64_t)row * ncol + pos[b];
                for (int c = 0; c < d; ++c) orow[c] = 0.0;
                for (int t = 0; t < n; ++t) {
                    const double *v = V + (int64_t)t * d;
                    for (int c = 0; c < d; ++c) orow[c] += w[t] * v[c];
                }
            }
            free(C); free(P); free(V);
        }
        if (fail) { free(kt); rc = MO_ERR_NOMEM; break; }

        /* pass 2b: tail values; then sum blocks in table order, divide by Z */
        double *otail = ob + (int64_t)p->nblk * rows * d;
        for (int64_t x = 0; x < (int64_t)rows * d; ++x) otail[x] = 0.0;
        for (int i = 0; i < p->batch; ++i) {
            const int64_t T = tail_len(p, i);
            for (int64_t t = 0; t < T; ++t) {
                fetch(p->dtype, p->tv, ((p->toff[i] + t) * p->hkv + g) * d, d, kt);
                for (int hh = 0; hh < G; ++hh) {
                    const int row = i * G + hh;
                    const double w = S[(int64_t)row * ncol + np + t];
                    for (int c = 0; c < d; ++c) otail[(int64_t)row * d + c] += w * kt[c];
                }
            }
        }
        free(kt);
        for (int row = 0; row < rows; ++row) {
            const int i = row / G, h = g * G + row % G;
            double *o = out + ((int64_t)i * p->hq + h) * d;
            for (int c = 0; c < d; ++c) {
                double acc = 0.0;
                for (int b = 0; b <= p->nblk; ++b)
                    acc += ob[((int64_t)b * rows + row) * d + c];
                o[c] = acc / Z[row];
            }
            if (weights) {
                const int64_t valid = np + tail_len(p, i);
                double *wr = weights + ((int64_t)i * p->hq + h) * wstride;
                for (int64_t t = 0; t < valid; ++t)
                    wr[t] = S[(int64_t)row * ncol + t] / Z[row];
            }
        }
    }
    free(pos); free(S); free(Z); free(qv); free(ob);
    return rc;
}

/* ------------------------------------------------------------------------ */
/* Attention, rank-space form (cross-check only).  Per block:               */
/*   q~ = P^K q,  s_t = scale * <C^K[t,:], q~>,                              */
/*   v~ = sum_t w_t C^V[t,:],  contribution = v~ P^V.                         */
/* Same two-pass softmax, no reconstruction of K^ or V^.                     */
/* ------------------------------------------------------------------------ */
static int attention_rankspace(const mo_problem *p, double *out)
{
    int64_t np, tmax;
    int rc = check_problem(p, &np, &tmax);
    if (rc) return rc;
    const int G = p->hq / p->hkv, d = p->d;
    const int64_t ncol = np + tmax;
    if (p->batch == 0) return MO_OK;
    int fail = 0;

#pragma omp parallel for schedule(dynamic, 1) collapse(2)
    for (int i = 0; i < p->batch; ++i)
        for (int h = 0; h < p->hq; ++h) {
            const int g = h / G;
            const int64_t T = tail_len(p, i), valid = np + T;
            double *s = (double *)malloc(sizeof(double) * (size_t)(ncol + 1));
            double *qv = (double *)malloc(sizeof(double) * (size_t)d);
            double *x = (double *)malloc(sizeof(double) * (size_t)d);
            double *qt = (double *)malloc(sizeof(double) * (size_t)d);
            double *acc = (double *)malloc(sizeof(double) * (size_t)d);
            double *row = (double *)malloc(sizeof(double) * (size_t)d);
            if (!s || !qv || !x || !qt || !acc || !row) {
#pragma omp atomic write
                fail = 1;
                free(s); free(qv); free(x); free(qt); free(acc); free(row);
                continue;
            }
            fetch(p->dtype, p->q, ((int64_t)i * p->hq + h) * d, d, qv);
            int64_t base = 0;
            for (int b = 0; b < p->nblk; ++b) {
                const int e = b * p->hkv + g, n = p->blen[b], r = p->rk[e];
                for (int j = 0; j < r; ++j) {          /* q~ = P^K q */
                    fetch(p->dtype, p->arena, p->opk[e] + (int64_t)j * d, d, row);
                    qt[j] = dot(row, qv, d);
                }
                for (int t = 0; t < n; ++t) {           /* s = C^K q~ */
                    fetch(p->dtype, p->arena, p->ock[e] + (int64_t)t * r, r, row);
                    s[base + t] = p->scale * dot(row, qt, r);
                }
                base += n;
            }
            for (int64_t t = 0; t < T; ++t) {
                fetch(p->dtype, p->tk, ((p->toff[i] + t) * p->hkv + g) * d, d, x);
                s[np + t] = p->scale * dot(x, qv, d);
            }
            double M = -INFINITY, z = 0.0;
            for (int64_t t = 0; t < valid; ++t) if (s[t] > M) M = s[t];
            for (int64_t t = 0; t < valid; ++t) { s[t] = exp(s[t] - M); z += s[t]; }
            for (int c = 0; c < d; ++c) acc[c] = 0.0;
            base = 0;
            for (int b = 0; b < p->nblk; ++b) {
                const int e = b * p->hkv + g, n = p->blen[b], r = p->rv[e];
                for (int j = 0; j < r; ++j) qt[j] = 0.0; /* v~ = sum_t w_t C^V[t] */
                for (int t = 0; t < n; ++t) {
                    fetch(p->dtype, p->arena, p->ocv[e] + (int64_t)t * r, r, row);
                    for (int j = 0; j < r; ++j) qt[j] += s[base + t] * row[j];
                }
                for (int j = 0; j < r; ++j) {           /* + v~ P^V */
                    fetch(p->dtype, p->arena, p->opv[e] + (int64_t)j * d, d, row);
                    for (int c = 0; c < d; ++c) acc[c] += qt[j] * row[c];
                }
                base += n;
            }
            for (int64_t t = 0; t < T; ++t) {
                fetch(p->dtype, p->tv, ((p->toff[i] + t) * p->hkv + g) * d, d, x);
                for (int c = 0; c < d; ++c) acc[c] += s[np + t] * x[c];
            }
            double *o = out + ((int64_t)i * p->hq + h) * d;
            for (int c = 0; c < d; ++c) o[c] = acc[c] / z;
            free(s); free(qv); free(x); free(qt); free(acc); free(row);
        }
    return fail ? MO_ERR_NOMEM : MO_OK;
}

/*
 * Public attention entry points.  All arrays are host memory.
 *   dtype          MO_F64 (arrays of double) or MO_BF16 (arrays of uint16
 *                  bf16 bit patterns) for arena, q, tail_k, tail_v.
 *   block_len      [num_blocks] tokens per block (>= 1).
 *   rank_k/rank_v  [num_blocks * num_kv_heads], entry (b, g) at b*Hkv + g,
 *                  0 <= rank <= head_dim.
 *   off_*          same indexing; element offsets into `arena` of
 *                  C^K (n x r^k), P^K (r^k x d), C^V (n x r^v), P^V (r^v x d),
 *                  all row-major.
 *   q              [batch, Hq, d].
 *   tail_k/tail_v  [tail_offsets[batch], Hkv, d]; tail_offsets [batch+1]
 *                  cumulative, may be NULL for no tail.
 *   scale          softmax scale; <= 0 selects 1/sqrt(d).
 *   out            [batch, Hq, d] fp64.
 *   weights        optional [batch, Hq, wstride] fp64: normalised softmax
 *                  weights, prefix tokens in table order then tail tokens.
 */
int mo_attention_dense(int dtype, int batch, int num_q_heads, int num_kv_heads,
                       int head_dim, int num_blocks, const int32_t *block_len,
                       const int32_t *rank_k, const int32_t *rank_v,
                       const int64_t *off_ck, const int64_t *off_pk,
                       const int64_t *off_cv, const int64_t *off_pv,
                       const void *arena, const void *q, const void *tail_k,
                       const void *tail_v, const int64_t *tail_offsets,
                       double scale, double *out, double *weights,
                       int64_t wstride)
{
    mo_problem p = {dtype, batch, num_q_heads, num_kv_heads, head_dim,
                    num_blocks, block_len, rank_k, rank_v, off_ck, off_pk,
                    off_cv, off_pv, arena, q, tail_k, tail_v, tail_offsets,
                    scale > 0.0 ? scale : 1.0 / sqrt((double)head_dim)};
    return attention_dense(&p, out, weights, wstride);
}

/* Pre-RoPE factors: as mo_attention_dense, with every reconstructed prefix
 * key rotated (rope_theta > 0; head_dim even) to its position block_pos[b]
 * + t (block_pos NULL: the block's start in the concatenated prefix). */
int mo_attention_dense_rope(int dtype, int batch, int num_q_heads, int num_kv_heads,
                            int head_dim, int num_blocks, const int32_t *block_len,
                            const int32_t *rank_k, const int32_t *rank_v,
                            const int64_t *off_ck, const int64_t *off_pk,
                            const int64_t *off_cv, const int64_t *off_pv,
                            const void *arena, const void *q, const void *tail_k,
                            const void *tail_v, const int64_t *tail_offsets,
                            double scale, double rope_theta, const int64_t *block_pos,
                            double *out, double *weights, int64_t wstride)
{
    if (!(rope_theta > 0.0)) return MO_ERR_ARG;
    mo_problem p = {dtype, batch, num_q_heads, num_kv_heads, head_dim,
                    num_blocks, block_len, rank_k, rank_v, off_ck, off_pk,
                    off_cv, off_pv, arena, q, tail_k, tail_v, tail_offsets,
                    scale > 0.0 ? scale : 1.0 / sqrt((double)head_dim),
                    rope_theta, block_pos};
    return attention_dense(&p, out, weights, wstride);
}

/* The rotation alone, in place, on n fp64 rows of width d: row t at
 * position pos[t]. */
int mo_rope_rotate(int n, int d, double *X, const int64_t *pos, double theta)
{
    if (n < 0 || d <= 0 || d % 2 != 0 || !(theta > 0.0) || (n > 0 && (!X || !pos)))
        return MO_ERR_ARG;
    rope_rows(X, n, d, 0, pos, theta);
    return MO_OK;
}

int mo_attention_rankspace(int dtype, int batch, int num_q_heads,
                           int num_kv_heads, int head_dim, int num_blocks,
                           const int32_t *block_len, const int32_t *rank_k,
                           const int32_t *rank_v, const int64_t *off_ck,
                           const int64_t *off_pk, const int64_t *off_cv,
                           const int64_t *off_pv, const void *arena,
                           const void *q, const void *tail_k,
                           const void *tail_v, const int64_t *tail_offsets,
                           double scale, double *out)
{
    mo_problem p = {dtype, batch, num_q_heads, num_kv_heads, head_dim,
                    num_blocks, block_len, rank_k, rank_v, off_ck, off_pk,
                    off_cv, off_pv, arena, q, tail_k, tail_v, tail_offsets,
                    scale > 0.0 ? scale : 1.0 / sqrt((double)head_dim)};
    return attention_rankspace(&p, out);
}

/* ------------------------------------------------------------------------ */
/* SVD of one block, Eq. 3: X (n x d) = A Sigma B^T.                        */
/* One-sided Jacobi: rotate pairs of columns of W (= X, or X^T when n < d)  */
/* until every pair is orthogonal to working precision; the column norms    */
/* are then the singular values.  Outputs, with k = min(n, d) and singular  */
/* values in non-increasing order:                                           */
/*   sigma[k];  C = A Sigma (n x k, row-major);  P = B^T (k x d, row-major). */
/* A zero singular value leaves its row of P (n >= d: a column of the       */
/* rotation, still orthonormal; n < d: zero) -- its column of C is zero.    */
/* ------------------------------------------------------------------------ */
int mo_svd_jacobi(int n, int d, const double *X, double *sigma, double *C,
                  double *P, int *sweeps_out)
{
    if (n <= 0 || d <= 0 || !X || !sigma || !C || !P) return MO_ERR_ARG;
    const int tall = n >= d;
    const int rows = tall ? n : d, k = tall ? d : n; /* W is rows x k */
    double *W = (double *)malloc(sizeof(double) * (size_t)rows * k);
    double *R = (double *)malloc(sizeof(double) * (size_t)k * k); /* rotations */
    int *perm = (int *)malloc(sizeof(int) * (size_t)k);
    double *nrm = (double *)malloc(sizeof(double) * (size_t)k);
    if (!W || !R || !perm || !nrm) {
        free(W); free(R); free(perm); free(nrm);
        return MO_ERR_NOMEM;
    }
    /* W column-major: column c occupies W[c*rows ... c*rows + rows) */
    for (int c = 0; c < k; ++c)
        for (int x = 0; x < rows; ++x)
            W[(int64_t)c * rows + x] = tall ? X[(int64_t)x * d + c] : X[(int64_t)c * d + x];
    for (int a = 0; a < k; ++a)
        for (int b = 0; b < k; ++b) R[(int64_t)a * k + b] = (a == b) ? 1.0 : 0.0;

    /* a pair counts as orthogonal once |cos| <= sqrt(rows) * machine epsilon */
    const double tol = sqrt((double)rows) * 2.220446049250313e-16;
    int sweep, converged = 0;
    for (sweep = 0; sweep < 100 && !converged; ++sweep) {
        converged = 1;
        for (int pcol = 0; pcol < k - 1; ++pcol)
            for (int qcol = pcol + 1; qcol < k; ++qcol) {
                double *wp = W + (int64_t)pcol * rows, *wq = W + (int64_t)qcol * rows;
                double alpha = dot(wp, wp, rows), beta = dot(wq, wq, rows);
                double gamma = dot(wp, wq, rows);
                if (gamma == 0.0 || fabs(gamma) <= tol * sqrt(alpha * beta)) continue;
                converged = 0;
                double zeta = (beta - alpha) / (2.0 * gamma);
                double t = (zeta >= 0 ? 1.0 : -1.0) / (fabs(zeta) + sqrt(1.0 + zeta * zeta));
                double cs = 1.0 / sqrt(1.0 + t * t), sn = cs * t;
                for (int x = 0; x < rows; ++x) {
                    double u = wp[x], v = wq[x];
                    wp[x] = cs * u - sn * v;
                    wq[x] = sn * u + cs * v;
                }
                double *rp = R + (int64_t)pcol * k, *rq = R + (int64_t)qcol * k;
                for (int x = 0; x < k; ++x) {
                    double u = rp[x], v = rq[x];
                    rp[x] = cs * u - sn * v;
                    rq[x] = sn * u + cs * v;
                }
            }
    }
    if (sweeps_out) *sweeps_out = sweep;
    /* singular values = column norms; sort non-increasing (stable) */
    for (int c = 0; c < k; ++c) {
        nrm[c] = sqrt(dot(W + (int64_t)c * rows, W + (int64_t)c * rows, rows));
        perm[c] = c;
    }
    for (int a = 1; a < k; ++a) {
        int v = perm[a], b = a - 1;
        while (b >= 0 && nrm[perm[b]] < nrm[v]) { perm[b + 1] = perm[b]; --b; }
        perm[b + 1] = v;
    }
    for (int j = 0; j < k; ++j) {
        const int c = perm[j];
        const double s = nrm[c];
        const double *w = W + (int64_t)c * rows; /* = U[:,j] * s */
        const double *rcol = R + (int64_t)c * k; /* column c of the rotation */
        sigma[j] = s;
        if (tall) {
            /* X R = W  =>  X = W R^T : C[:,j] = W[:,c], P[j,:] = R[:,c]^T */
            for (int x = 0; x < n; ++x) C[(int64_t)x * k + j] = w[x];
            for (int x = 0; x < d; ++x) P[(int64_t)j * d + x] = rcol[x];
        } else {
            /* X^T R = W  =>  X = R W^T : C[:,j] = s * R[:,c], P[j,:] = W[:,c]^T / s */
            for (int x = 0; x < n; ++x) C[(int64_t)x * k + j] = s * rcol[x];
            for (int x = 0; x < d; ++x) P[(int64_t)j * d + x] = s > 0.0 ? w[x] / s : 0.0;
        }
    }
    free(W); free(R); free(perm); free(nrm);
    return converged ? MO_OK : MO_ERR_NOCONV;
}

/* Eq. 5: H(r) = sum_{j<=r} log(1 + sigma_j^2 / eps^2), sigma sorted. */
double mo_spectral_information(int r, const double *sigma, double eps)
{
    double h = 0.0;
    for (int j = 0; j < r; ++j) h += log1p(sigma[j] * sigma[j] / (eps * eps));
    return h;
}

/*
 * Eq. 6 / Eq. 7: greedy allocation of a total rank budget.
 *   sigma      [num_blocks][ld] singular values of each block, sorted
 *              non-increasing; block i has avail[i] = min(n_i, d) of them.
 *   Start:     r_i = min(r_min, avail_i).
 *   Repeat:    while sum r_i < R_tot, give one unit to the eligible block
 *              (r_i < min(r_max, avail_i)) with the largest marginal gain
 *              log(1 + sigma_{i, r_i+1}^2 / eps^2); ties go to the lowest
 *              block index.  With stop_at_zero_gain set, a block whose next
 *              singular value is zero is not eligible.
 * Returns MO_ERR_INFEASIBLE if the starting ranks already exceed R_tot.
 */
int mo_allocate_ranks(int num_blocks, const int32_t *avail, const double *sigma,
                      int ld, int r_min, int r_max, int64_t R_tot, double eps,
                      int stop_at_zero_gain, int32_t *ranks_out)
{
    if (num_blocks < 0 || r_min < 0 || r_max < r_min || eps <= 0.0) return MO_ERR_ARG;
    int64_t used = 0;
    for (int i = 0; i < num_blocks; ++i) {
        if (avail[i] < 0 || avail[i] > ld) return MO_ERR_ARG;
        ranks_out[i] = r_min < avail[i] ? r_min : avail[i];
        used += ranks_out[i];
    }
    if (used > R_tot) return MO_ERR_INFEASIBLE;
    while (used < R_tot) {
        int best = -1;
        double best_gain = -1.0;
        for (int i = 0; i < num_blocks; ++i) {
            const int cap = r_max < avail[i] ? r_max : avail[i];
            if (ranks_out[i] >= cap) continue;
            const double s = sigma[(int64_t)i * ld + ranks_out[i]];
            if (stop_at_zero_gain && s == 0.0) continue;
            const double gain = log1p(s * s / (eps * eps));
            if (gain > best_gain) { best_gain = gain; best = i; }
        }
        if (best < 0) break;
        ranks_out[best] += 1;
        used += 1;
    }
    return MO_OK;
}

/* Eq. 4, generalised to per-block token counts n_i:
 *   rho = sum_i (r^k_i + r^v_i)(n_i + d) / sum_i 2 n_i d,
 * returned as an exact integer fraction num / den. */
int mo_compression_ratio(int num_blocks, const int32_t *block_len,
                         const int32_t *rank_k, const int32_t *rank_v, int d,
                         int64_t *num, int64_t *den)
{
    if (num_blocks < 0 || d <= 0) return MO_ERR_ARG;
    int64_t a = 0, b = 0;
    for (int i = 0; i < num_blocks; ++i) {
        a += (int64_t)(rank_k[i] + rank_v[i]) * (block_len[i] + d);
        b += 2 * (int64_t)block_len[i] * d;
    }
    *num = a;
    *den = b;
    return MO_OK;
}

/* Eq. 2: fp16 bytes of a dense KV cache, 2 (K and V) * N * L * H * d * 2. */
int64_t mo_kv_cache_bytes(int64_t N, int64_t L, int64_t H, int64_t d)
{
    return 2 * N * L * H * d * 2;
}
