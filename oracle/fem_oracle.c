/*
 * Float64 CPU oracle for the Free Energy Mixer forward read with a softmax
 * prior (arXiv 2602.07160).
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the slow, obviously correct
 * statement of what the GPU path computes.  It is used by the tests, by
 * __graft_entry__.smoke() and by the CPU-baseline leg of bench.py, and by
 * nothing else.  It shares no code, header, table or constant with the CUDA
 * library, and the library never calls it.
 *
 * What it computes (Sec. 2.3, Eq. "fem-free-energy-main"; App. C,
 * Eq. "softmax-prior"; Sec. 1 for the masked scaled scores):
 *
 *   s_{t,i} = q_t . k_i / sqrt(d)          for i in M_t
 *   M_t     = {0..t} (causal)  or  {0..T-1} (full prior)
 *   p_t(i)  = softmax_i(s_{t,i})
 *   o_{t,j} = (1/beta_j) log sum_{i in M_t} p_t(i) exp(beta_j v_{i,j})
 *           = (1/beta_j) ( LSE_i(s_{t,i} + beta_j v_{i,j}) - LSE_i s_{t,i} )
 *   lse_t   = LSE_i s_{t,i}                   (natural log)
 *
 * beta_j = 0 is the continuous extension of the read, the prior mean
 * o_{t,j} = sum_i p_t(i) v_{i,j} (the small-beta expansion of Prop.
 * "app-baseline").  Negative beta is outside the method (beta > 0 in Sec. 2.3)
 * and is rejected.
 *
 * Each LSE is stabilised by its own maximum, the per-channel stabilisation
 * the paper states in App. E ("Numerical stability").  Everything is double
 * precision and there is no blocking, fusion or reordering beyond the two
 * LSEs of the definition.
 *
 * Layout: q, k, v are [B, H, T, d] row-major (d fastest), beta is [H, d],
 * out is [B, H, T, d], lse is [B, H, T] (may be NULL).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* One output row (b, h, t).  q_t is the query row, kbase/vbase point at row
 * 0 of the keys/values of this (b, h), n is |M_t| (the support is the first n
 * keys).  s must hold n doubles. */
static void fem_oracle_row(const double *q_t, const double *kbase,
                           const double *vbase, const double *beta_h,
                           int64_t n, int64_t d, double *s, double *out_t,
                           double *lse_t)
{
    const double scale = 1.0 / sqrt((double)d);

    /* masked scaled scores s_{t,i} = q_t . k_i / sqrt(d) */
    for (int64_t i = 0; i < n; ++i) {
        const double *k_i = kbase + i * d;
        double dot = 0.0;
        for (int64_t c = 0; c < d; ++c)
            dot += q_t[c] * k_i[c];
        s[i] = dot * scale;
    }

    /* lse_t = LSE_i s_{t,i}: the log-normaliser of the softmax prior */
    double m = -INFINITY;
    for (int64_t i = 0; i < n; ++i)
        if (s[i] > m) m = s[i];
    double z = 0.0;
    for (int64_t i = 0; i < n; ++i)
        z += exp(s[i] - m);
    const double lse = m + log(z);
    if (lse_t) *lse_t = lse;

    for (int64_t j = 0; j < d; ++j) {
        const double b = beta_h[j];
        if (b == 0.0) {
            /* beta -> 0 limit: the prior mean sum_i p_t(i) v_{i,j} */
            double mu = 0.0;
            for (int64_t i = 0; i < n; ++i)
                mu += exp(s[i] - lse) * vbase[i * d + j];
            out_t[j] = mu;
            continue;
        }
        /* G = LSE_i (s_{t,i} + beta_j v_{i,j}), stabilised by its own max */
        double a_max = -INFINITY;
        for (int64_t i = 0; i < n; ++i) {
            const double a = s[i] + b * vbase[i * d + j];
            if (a > a_max) a_max = a;
        }
        double g = 0.0;
        for (int64_t i = 0; i < n; ++i)
            g += exp(s[i] + b * vbase[i * d + j] - a_max);
        const double G = a_max + log(g);
        out_t[j] = (G - lse) / b;
    }
}

static int check_args(const double *q, const double *k, const double *v,
                      const double *beta, int64_t B, int64_t H, int64_t T,
                      int64_t d)
{
    if (!q || !k || !v || !beta) return 1;
    if (B <= 0 || H <= 0 || T <= 0 || d <= 0) return 1;
    for (int64_t x = 0; x < H * d; ++x)
        if (!(beta[x] >= 0.0) || isinf(beta[x])) return 1;
    return 0;
}

/* Selected rows of the read.  rows[r] is a flat row index (b*H + h)*T + t.
 * out_rows is [n_rows, d]; lse_rows is [n_rows] or NULL.  Returns 0 on
 * success, 1 on a bad argument, 2 on allocation failure. */
int fem_oracle_rows(const double *q, const double *k, const double *v,
                    const double *beta, int64_t B, int64_t H, int64_t T,
                    int64_t d, int causal, const int64_t *rows,
                    int64_t n_rows, double *out_rows, double *lse_rows,
                    int nthreads)
{
    if (check_args(q, k, v, beta, B, H, T, d) || !rows || !out_rows ||
        n_rows < 0)
        return 1;
    for (int64_t r = 0; r < n_rows; ++r)
        if (rows[r] < 0 || rows[r] >= B * H * T) return 1;
    int failed = 0;
#ifdef _OPENMP
    if (nthreads <= 0) nthreads = omp_get_max_threads();
#pragma omp parallel num_threads(nthreads) reduction(| : failed)
#endif
    {
        double *s = (double *)malloc(sizeof(double) * (size_t)T);
        if (!s) {
            failed = 1;
        } else {
#ifdef _OPENMP
#pragma omp for schedule(dynamic, 16)
#endif
            for (int64_t r = 0; r < n_rows; ++r) {
                const int64_t row = rows[r];
                const int64_t bh = row / T, t = row % T;
                const int64_t h = bh % H;
                const int64_t n = causal ? t + 1 : T;
                fem_oracle_row(q + row * d, k + bh * T * d, v + bh * T * d,
                               beta + h * d, n, d, s, out_rows + r * d,
                               lse_rows ? lse_rows + r : NULL);
            }
            free(s);
        }
    }
    (void)nthreads;
    return failed ? 2 : 0;
}

/* The whole read: out [B, H, T, d], lse [B, H, T] (or NULL). */
int fem_oracle_fwd(const double *q, const double *k, const double *v,
                   const double *beta, int64_t B, int64_t H, int64_t T,
                   int64_t d, int causal, double *out, double *lse,
                   int nthreads)
{
    if (check_args(q, k, v, beta, B, H, T, d) || !out) return 1;
    const int64_t n_rows = B * H * T;
    int64_t *rows = (int64_t *)malloc(sizeof(int64_t) * (size_t)n_rows);
    if (!rows) return 2;
    for (int64_t r = 0; r < n_rows; ++r) rows[r] = r;
    const int rc = fem_oracle_rows(q, k, v, beta, B, H, T, d, causal, rows,
                                   n_rows, out, lse, nthreads);
    free(rows);
    return rc;
}

/* Number of OpenMP threads the oracle would use by default (1 without
 * OpenMP). */
int fem_oracle_max_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}
