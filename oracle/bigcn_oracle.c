/*
 * bigcn_oracle.c -- plain CPU oracle of the Bi-GCN layer forward
 * (Wang et al., CVPR 2021, arXiv:2010.07565). See bigcn_oracle.h.
 *
 * TEST INFRASTRUCTURE: loaded only by the tests, the smoke check and the
 * benchmark's CPU-baseline leg. No code here is shared with the CUDA path.
 *
 * Each function follows one definition of the paper in its own order:
 *   centring ........ Sec. 6.2 (batch normalisation of the input features)
 *   signs ........... Eq. 3 (weights), Eq. 8 (node features), sign(0) = +1
 *   scales .......... Eq. 4 (weight column), Eq. 7 (node row), both read as the
 *                     mean absolute value over the d_in entries of the bucket
 *   binary product .. Eq. 11 / Eq. 12 (dot of +-1 vectors, then scaled)
 *   aggregation ..... Eq. 13 with the operator of Eq. 1, D^-1/2 (A+I) D^-1/2,
 *                     for a 0/1 adjacency and for a weighted one (Sec. 3's
 *                     A = [a_ij], D^_ii = sum_j a^_ij)
 *   back-propagation  Algorithm 1 (A~^T dH, H~^T G, G W~^T), Eq. bp-H (the
 *                     gradient of the layer input, clipped to |.| < 1) and
 *                     Eq. bp-W (the weight gradient through the column scale
 *                     and the straight-through estimator of sign)
 *
 * The pins that tie these routines to the paper and to mathematics (brute
 * force on tiny inputs, the scale's least-squares optimality, dense-matrix
 * special cases, operator invariants, the paper's printed cost figures) live
 * in the test suite, tests/test_oracle_pins.py.
 */
#include "bigcn_oracle.h"

#include <math.h>
#include <stddef.h>
#include <stdlib.h>

void oracle_centre(const float *X, int64_t N, int32_t K, int64_t ldx,
                   const float *s, const float *t, float *Y) {
    for (int64_t i = 0; i < N; ++i) {
        for (int32_t k = 0; k < K; ++k) {
            float x = X[i * ldx + k];
            /* One fp32 fused multiply-add: the sign decided later from Y must
             * be taken in the same precision on every implementation. */
            Y[i * (int64_t)K + k] = (s != NULL) ? fmaf(x, s[k], t[k]) : x;
        }
    }
}

void oracle_sign(const float *V, int64_t n, int8_t *S) {
    for (int64_t e = 0; e < n; ++e)
        S[e] = (V[e] >= 0.0f) ? (int8_t)1 : (int8_t)-1;
}

void oracle_row_scale(const float *Y, int64_t N, int32_t K, double *alpha) {
    for (int64_t i = 0; i < N; ++i) {
        double l1 = 0.0;
        for (int32_t k = 0; k < K; ++k)
            l1 += fabs((double)Y[i * (int64_t)K + k]);
        alpha[i] = l1 / (double)K;
    }
}

void oracle_weight_binarize(const float *Wt, int32_t K, int32_t F, int64_t ldw,
                            int8_t *SB, double *beta) {
    for (int32_t j = 0; j < F; ++j) {
        double l1 = 0.0;
        for (int32_t k = 0; k < K; ++k) {
            float w = Wt[(int64_t)k * ldw + j];
            SB[(int64_t)j * K + k] = (w >= 0.0f) ? (int8_t)1 : (int8_t)-1;
            l1 += fabs((double)w);
        }
        beta[j] = l1 / (double)K;
    }
}

void oracle_pack(const int8_t *S, int64_t n, int32_t K, int32_t words,
                 uint64_t *bits) {
    for (int64_t r = 0; r < n; ++r) {
        for (int32_t w = 0; w < words; ++w)
            bits[r * words + w] = 0;
        for (int32_t k = 0; k < K; ++k) {
            if (S[r * (int64_t)K + k] > 0)
                bits[r * words + k / 64] |= (uint64_t)1 << (k % 64);
        }
    }
}

void oracle_binary_dot(const int8_t *SF, int64_t N, const int8_t *SB, int32_t F,
                       int32_t K, int32_t *dot) {
    for (int64_t i = 0; i < N; ++i) {
        const int8_t *f = SF + i * (int64_t)K;
        for (int32_t j = 0; j < F; ++j) {
            const int8_t *b = SB + (int64_t)j * K;
            int32_t acc = 0;
            for (int32_t k = 0; k < K; ++k)
                acc += (int32_t)f[k] * (int32_t)b[k];
            dot[i * (int64_t)F + j] = acc;
        }
    }
}

void oracle_zeta(const int32_t *dot, const double *alpha, const double *beta,
                 int64_t N, int32_t F, double *zeta) {
    for (int64_t i = 0; i < N; ++i)
        for (int32_t j = 0; j < F; ++j)
            zeta[i * (int64_t)F + j] =
                alpha[i] * beta[j] * (double)dot[i * (int64_t)F + j];
}

void oracle_degree(const int64_t *rowptr, int64_t N, double *dhat) {
    for (int64_t i = 0; i < N; ++i)
        dhat[i] = 1.0 + (double)(rowptr[i + 1] - rowptr[i]);
}

/* h += zeta_j / sqrt(di * dj), and a += |zeta_j / sqrt(di * dj)|. */
static void add_neighbour(double *h, double *a, const double *zeta_j,
                          int32_t F, double di, double dj) {
    double norm = sqrt(di * dj);
    for (int32_t f = 0; f < F; ++f) {
        double term = zeta_j[f] / norm;
        h[f] += term;
        if (a != NULL)
            a[f] += fabs(term);
    }
}

int oracle_aggregate(const int64_t *rowptr, const int32_t *colidx, int64_t N,
                     const double *zeta, int32_t F, const int64_t *rows,
                     int64_t nrows, double *H, double *absterm) {
    if (rowptr[0] != 0)
        return -1;
    for (int64_t i = 0; i < N; ++i)
        if (rowptr[i + 1] < rowptr[i])
            return -1;
    for (int64_t e = 0; e < rowptr[N]; ++e)
        if (colidx[e] < 0 || (int64_t)colidx[e] >= N)
            return -1;

    int64_t count = (rows != NULL) ? nrows : N;
    for (int64_t r = 0; r < count; ++r) {
        int64_t i = (rows != NULL) ? rows[r] : r;
        if (i < 0 || i >= N)
            return -1;
        double di = 1.0 + (double)(rowptr[i + 1] - rowptr[i]);
        double *h = H + r * (int64_t)F;
        double *a = (absterm != NULL) ? absterm + r * (int64_t)F : NULL;
        for (int32_t f = 0; f < F; ++f) {
            h[f] = 0.0;
            if (a != NULL)
                a[f] = 0.0;
        }
        /* The self-loop that A + I adds ... */
        add_neighbour(h, a, zeta + i * (int64_t)F, F, di, di);
        /* ... then every neighbour listed in row i of A. */
        for (int64_t e = rowptr[i]; e < rowptr[i + 1]; ++e) {
            int64_t j = colidx[e];
            double dj = 1.0 + (double)(rowptr[j + 1] - rowptr[j]);
            add_neighbour(h, a, zeta + j * (int64_t)F, F, di, dj);
        }
    }
    return 0;
}

/* ---- Back-propagation (Algorithm 1, Eqs. bp-H, bp-W) ---- */

int oracle_aggregate_t(const int64_t *rowptr, const int32_t *colidx, int64_t N,
                       const double *dH, int32_t F, double *G) {
    double *dhat;
    int64_t i, e;
    int32_t f;
    if (rowptr[0] != 0) return -1;
    for (i = 0; i < N; ++i)
        if (rowptr[i + 1] < rowptr[i]) return -1;
    for (e = 0; e < rowptr[N]; ++e)
        if (colidx[e] < 0 || colidx[e] >= N) return -1;
    dhat = (double *)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    if (!dhat) return -1;
    oracle_degree(rowptr, N, dhat);
    for (i = 0; i < N * (int64_t)F; ++i) G[i] = 0.0;
    for (i = 0; i < N; ++i) {
        /* the self-loop of A + I, then the CSR entries of row i */
        for (e = rowptr[i] - 1; e < rowptr[i + 1]; ++e) {
            const int64_t jj = (e < rowptr[i]) ? i : (int64_t)colidx[e];
            const double c = 1.0 / sqrt(dhat[i] * dhat[jj]);
            for (f = 0; f < F; ++f) G[jj * F + f] += dH[i * F + f] * c;
        }
    }
    free(dhat);
    return 0;
}

void oracle_grad_wtilde(const int8_t *SF, const double *alpha, const double *G,
                        int64_t N, int32_t K, int32_t F, double *out, double *absterm) {
    int64_t i;
    int32_t k, j;
    for (k = 0; k < K; ++k)
        for (j = 0; j < F; ++j) {
            double acc = 0.0;
            for (i = 0; i < N; ++i) acc += alpha[i] * (double)SF[i * K + k] * G[i * F + j];
            out[(int64_t)k * F + j] = acc;
        }
    if (absterm)
        for (j = 0; j < F; ++j) {
            double a = 0.0;
            for (i = 0; i < N; ++i) a += fabs(alpha[i] * G[i * F + j]);
            absterm[j] = a;
        }
}

void oracle_grad_htilde(const double *G, const double *beta, const int8_t *SB,
                        int64_t N, int32_t K, int32_t F, double *out, double *absterm) {
    int64_t i;
    int32_t k, j;
    for (i = 0; i < N; ++i) {
        for (k = 0; k < K; ++k) {
            double acc = 0.0;
            for (j = 0; j < F; ++j) acc += G[i * F + j] * beta[j] * (double)SB[(int64_t)j * K + k];
            out[i * K + k] = acc;
        }
        if (absterm) {
            double a = 0.0;
            for (j = 0; j < F; ++j) a += fabs(G[i * F + j] * beta[j]);
            absterm[i] = a;
        }
    }
}

void oracle_grad_input(const double *Ht, int64_t n, double *out) {
    int64_t q;
    for (q = 0; q < n; ++q) out[q] = fabs(Ht[q]) < 1.0 ? Ht[q] : 0.0;
}

void oracle_grad_weight(const double *Wg, const int8_t *SB, const double *beta,
                        const float *Wt, int32_t K, int32_t F, int64_t ldw, double *out) {
    int32_t k, j, m;
    for (j = 0; j < F; ++j) {
        double c = 0.0;   /* sum_m dL/dW~[m,j] B[m,j] */
        for (m = 0; m < K; ++m) c += Wg[(int64_t)m * F + j] * (double)SB[(int64_t)j * K + m];
        for (k = 0; k < K; ++k) {
            const double w = (double)Wt[(int64_t)k * ldw + j];
            const double ste = fabs(w) < 1.0 ? 1.0 : 0.0;
            out[(int64_t)k * F + j] = (double)SB[(int64_t)j * K + k] * c / (double)K +
                                      beta[j] * Wg[(int64_t)k * F + j] * ste;
        }
    }
}

void oracle_real_binary_product(const float *Y, int64_t N, int32_t K, const int8_t *SB,
                                const double *beta, int32_t F, double *zeta, double *absterm) {
    int64_t i;
    int32_t j, k;
    for (i = 0; i < N; ++i) {
        const float *y = Y + i * (int64_t)K;
        for (j = 0; j < F; ++j) {
            const int8_t *b = SB + (int64_t)j * K;
            double acc = 0.0, mag = 0.0;
            for (k = 0; k < K; ++k) {
                const double w = beta[j] * (double)b[k];   /* W~[k,j] */
                acc += (double)y[k] * w;
                mag += fabs((double)y[k] * w);
            }
            zeta[i * (int64_t)F + j] = acc;
            if (absterm != NULL) absterm[i * (int64_t)F + j] = mag;
        }
    }
}

void oracle_binary_real_product(const int8_t *SF, const double *alpha, int64_t N, int32_t K,
                                const float *Wt, int32_t F, int64_t ldw, double *zeta,
                                double *absterm) {
    int64_t i;
    int32_t j, k;
    for (i = 0; i < N; ++i) {
        const int8_t *f = SF + i * (int64_t)K;
        for (j = 0; j < F; ++j) {
            double acc = 0.0, mag = 0.0;
            for (k = 0; k < K; ++k) {
                const double h = alpha[i] * (double)f[k];   /* H~[i,k] */
                const double w = (double)Wt[(int64_t)k * ldw + j];
                acc += h * w;
                mag += fabs(h * w);
            }
            zeta[i * (int64_t)F + j] = acc;
            if (absterm != NULL) absterm[i * (int64_t)F + j] = mag;
        }
    }
}

/* 0 if the CSR is well formed (rowptr monotone from 0, indices in [0, N)). */
static int csr_check(const int64_t *rowptr, const int32_t *colidx, int64_t N) {
    int64_t i, e;
    if (rowptr[0] != 0)
        return -1;
    for (i = 0; i < N; ++i)
        if (rowptr[i + 1] < rowptr[i])
            return -1;
    for (e = 0; e < rowptr[N]; ++e)
        if (colidx[e] < 0 || (int64_t)colidx[e] >= N)
            return -1;
    return 0;
}

/* h += w * z, a += |w * z| over F entries. */
static void add_weighted(double *h, double *a, const double *z, int32_t F, double w) {
    int32_t f;
    for (f = 0; f < F; ++f) {
        double term = w * z[f];
        h[f] += term;
        if (a != NULL)
            a[f] += fabs(term);
    }
}

int oracle_aggregate_mean(const int64_t *rowptr, const int32_t *colidx, int64_t N,
                          const double *zeta, int32_t F, const int64_t *rows,
                          int64_t nrows, double *H, double *absterm) {
    int64_t r, e, count = (rows != NULL) ? nrows : N;
    int32_t f;
    if (csr_check(rowptr, colidx, N) != 0)
        return -1;
    for (r = 0; r < count; ++r) {
        int64_t i = (rows != NULL) ? rows[r] : r;
        double *h = H + r * (int64_t)F;
        double *a = (absterm != NULL) ? absterm + r * (int64_t)F : NULL;
        double w;
        if (i < 0 || i >= N)
            return -1;
        w = 1.0 / (1.0 + (double)(rowptr[i + 1] - rowptr[i]));   /* 1 / dhat_i */
        for (f = 0; f < F; ++f) {
            h[f] = 0.0;
            if (a != NULL)
                a[f] = 0.0;
        }
        add_weighted(h, a, zeta + i * (int64_t)F, F, w);          /* the node itself */
        for (e = rowptr[i]; e < rowptr[i + 1]; ++e)               /* its neighbours */
            add_weighted(h, a, zeta + (int64_t)colidx[e] * F, F, w);
    }
    return 0;
}

int oracle_aggregate_sage(const int64_t *rowptr, const int32_t *colidx, int64_t N,
                          const double *zself, const double *zneigh, int32_t F,
                          const int64_t *rows, int64_t nrows, double *H, double *absterm) {
    int64_t r, e, count = (rows != NULL) ? nrows : N;
    int32_t f;
    if (csr_check(rowptr, colidx, N) != 0)
        return -1;
    for (r = 0; r < count; ++r) {
        int64_t i = (rows != NULL) ? rows[r] : r;
        double *h = H + r * (int64_t)F;
        double *a = (absterm != NULL) ? absterm + r * (int64_t)F : NULL;
        int64_t deg;
        if (i < 0 || i >= N)
            return -1;
        deg = rowptr[i + 1] - rowptr[i];
        for (f = 0; f < F; ++f) {
            h[f] = 0.0;
            if (a != NULL)
                a[f] = 0.0;
        }
        add_weighted(h, a, zself + i * (int64_t)F, F, 1.0);       /* W_self h_i */
        for (e = rowptr[i]; e < rowptr[i + 1]; ++e)               /* W_neigh mean_j h_j */
            add_weighted(h, a, zneigh + (int64_t)colidx[e] * F, F, 1.0 / (double)deg);
    }
    return 0;
}

/* ---- A weighted adjacency (Sec. 3 notations, Eq. 1) ---- */

void oracle_degree_weighted(const int64_t *rowptr, const double *values, int64_t N,
                            double *dhat) {
    int64_t i, e;
    for (i = 0; i < N; ++i) {
        double d = 1.0;                         /* the self-loop's a^_ii = 1 */
        for (e = rowptr[i]; e < rowptr[i + 1]; ++e)
            d += values[e];
        dhat[i] = d;
    }
}

int oracle_aggregate_weighted(const int64_t *rowptr, const int32_t *colidx,
                              const double *values, int64_t N, const double *zeta,
                              int32_t F, const int64_t *rows, int64_t nrows, double *H,
                              double *absterm) {
    int64_t r, e, count = (rows != NULL) ? nrows : N;
    int32_t f;
    double *dhat;
    if (csr_check(rowptr, colidx, N) != 0)
        return -1;
    for (e = 0; e < rowptr[N]; ++e)
        if (!(values[e] >= 0.0) || !isfinite(values[e]))
            return -1;
    dhat = (double *)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    if (!dhat)
        return -1;
    oracle_degree_weighted(rowptr, values, N, dhat);
    for (r = 0; r < count; ++r) {
        int64_t i = (rows != NULL) ? rows[r] : r;
        double *h = H + r * (int64_t)F;
        double *a = (absterm != NULL) ? absterm + r * (int64_t)F : NULL;
        if (i < 0 || i >= N) {
            free(dhat);
            return -1;
        }
        for (f = 0; f < F; ++f) {
            h[f] = 0.0;
            if (a != NULL)
                a[f] = 0.0;
        }
        /* the self-loop of A + I, weight 1 ... */
        add_weighted(h, a, zeta + i * (int64_t)F, F, 1.0 / sqrt(dhat[i] * dhat[i]));
        /* ... then each entry a_ij of row i of A */
        for (e = rowptr[i]; e < rowptr[i + 1]; ++e) {
            int64_t j = colidx[e];
            add_weighted(h, a, zeta + j * (int64_t)F, F, values[e] / sqrt(dhat[i] * dhat[j]));
        }
    }
    free(dhat);
    return 0;
}

/* Number of buckets of B entries that cover K entries. */
static int32_t bucket_count(int32_t K, int32_t B) { return (K + B - 1) / B; }

void oracle_row_scale_bucketed(const float *Y, int64_t N, int32_t K, int32_t B, double *alpha) {
    const int32_t nb = bucket_count(K, B);
    int64_t i;
    int32_t b, k;
    for (i = 0; i < N; ++i)
        for (b = 0; b < nb; ++b) {
            const int32_t k0 = b * B, k1 = (k0 + B < K) ? k0 + B : K;
            double sum = 0.0;
            for (k = k0; k < k1; ++k) sum += fabs((double)Y[i * (int64_t)K + k]);
            alpha[i * nb + b] = sum / (double)(k1 - k0);
        }
}

void oracle_weight_scale_bucketed(const float *Wt, int32_t K, int32_t F, int64_t ldw, int32_t B,
                                  double *beta) {
    const int32_t nb = bucket_count(K, B);
    int32_t j, b, k;
    for (j = 0; j < F; ++j)
        for (b = 0; b < nb; ++b) {
            const int32_t k0 = b * B, k1 = (k0 + B < K) ? k0 + B : K;
            double sum = 0.0;
            for (k = k0; k < k1; ++k) sum += fabs((double)Wt[(int64_t)k * ldw + j]);
            beta[(int64_t)j * nb + b] = sum / (double)(k1 - k0);
        }
}

void oracle_zeta_bucketed(const int8_t *SF, const double *alpha, int64_t N, const int8_t *SB,
                          const double *beta, int32_t F, int32_t K, int32_t B, double *zeta,
                          double *absterm) {
    const int32_t nb = bucket_count(K, B);
    int64_t i;
    int32_t j, b, k;
    for (i = 0; i < N; ++i)
        for (j = 0; j < F; ++j) {
            double acc = 0.0, mag = 0.0;
            for (b = 0; b < nb; ++b) {
                const int32_t k0 = b * B, k1 = (k0 + B < K) ? k0 + B : K;
                int32_t dot = 0;
                double term;
                for (k = k0; k < k1; ++k)
                    dot += (int32_t)SF[i * (int64_t)K + k] * (int32_t)SB[(int64_t)j * K + k];
                term = alpha[i * nb + b] * beta[(int64_t)j * nb + b] * (double)dot;
                acc += term;
                mag += fabs(term);
            }
            zeta[i * (int64_t)F + j] = acc;
            if (absterm != NULL) absterm[i * (int64_t)F + j] = mag;
        }
}
