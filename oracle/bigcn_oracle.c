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
 *   aggregation ..... Eq. 13 with the operator of Eq. 1, D^-1/2 (A+I) D^-1/2
 *
 * The pins that tie these routines to the paper and to mathematics (brute
 * force on tiny inputs, the scale's least-squares optimality, dense-matrix
 * special cases, operator invariants, the paper's printed cost figures) live
 * in the test suite, tests/test_oracle_pins.py.
 */
#include "bigcn_oracle.h"

#include <math.h>
#include <stddef.h>

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
