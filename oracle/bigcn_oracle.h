/*
 * bigcn_oracle.h -- plain CPU oracle of the Bi-GCN binarized graph-convolution
 * layer, forward and back-propagation (Wang et al., "Bi-GCN: Binary Graph
 * Convolutional Network", CVPR 2021, arXiv:2010.07565).
 *
 * TEST INFRASTRUCTURE. Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg load this library. It shares no source, header,
 * table or helper with the CUDA path, and the CUDA path never calls it.
 *
 * Every routine is a slow, element-by-element restatement of one definition of
 * the paper, in its order, with floating point carried in double except where
 * a decision (a sign bit) must be taken in the same fp32 precision as the
 * kernel. All arrays are host memory owned by the caller; row-major.
 *
 * Naming: this library follows the naming of the layer's C interface, which
 * swaps the paper's letters. Here alpha_i is the per-NODE scale (the paper's
 * beta_i, Eq. 7) and beta_j is the per-WEIGHT-COLUMN scale (the paper's
 * alpha_j, Eq. 4).
 */
#ifndef BIGCN_ORACLE_H
#define BIGCN_ORACLE_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Step 1 -- input batch normalisation in inference form (Sec. 6.2):
 * Y[i,k] = fmaf(X[i,k], s[k], t[k]) in fp32, one rounding. s == t == NULL
 * means the identity (layer 2 binarizes its input raw, Sec. 4.1.2). */
void oracle_centre(const float *X, int64_t N, int32_t K, int64_t ldx,
                   const float *s, const float *t, float *Y);

/* Eq. 8 (F_i = sign(H_i,:)) and Eq. 3 (B_j = sign(W_:,j)): +1 where v >= 0
 * (so sign(0) = sign(-0) = +1), else -1. */
void oracle_sign(const float *V, int64_t n, int8_t *S);

/* Eq. 7 read as mean |y_i| (the bucket is the whole row, Sec. 4.1):
 * alpha[i] = (sum_k |Y[i,k]|) / K, summed in double. */
void oracle_row_scale(const float *Y, int64_t N, int32_t K, double *alpha);

/* Eq. 3 and Eq. 4 for the weight matrix Wt (K x F, row stride ldw):
 * SB[j,k] = sign(Wt[k,j]) (F x K, i.e. transposed) and
 * beta[j] = (sum_k |Wt[k,j]|) / K in double. */
void oracle_weight_binarize(const float *Wt, int32_t K, int32_t F, int64_t ldw,
                            int8_t *SB, double *beta);

/* Storage of a sign matrix S (n x K, entries +-1) in the interface's packed
 * layout: element k of row r is bit (k % 64) of 64-bit word r*words + k/64,
 * set for +1; bits at k >= K are 0. */
void oracle_pack(const int8_t *S, int64_t n, int32_t K, int32_t words,
                 uint64_t *bits);

/* Eq. 11, the integer part: dot[i,j] = sum_k SF[i,k] * SB[j,k]. */
void oracle_binary_dot(const int8_t *SF, int64_t N, const int8_t *SB, int32_t F,
                       int32_t K, int32_t *dot);

/* Eq. 11/12, the scaled result: zeta[i,j] = alpha[i] * beta[j] * dot[i,j]. */
void oracle_zeta(const int32_t *dot, const double *alpha, const double *beta,
                 int64_t N, int32_t F, double *zeta);

/* Sec. 3.1: dhat[i] = sum_j ahat[i,j] with Ahat = A + I and a_ij = 1 on the
 * CSR's entries, i.e. 1 + (rowptr[i+1] - rowptr[i]). */
void oracle_degree(const int64_t *rowptr, int64_t N, double *dhat);

/* Eq. 13 with Eq. 1's operator: H[r,:] = sum over j in N(i) u {i} of
 * zeta[j,:] / sqrt(dhat_i * dhat_j), for each requested row i = rows[r]
 * (rows == NULL: all N rows, r = i). absterm[r,:] (nullable) receives the sum
 * of the absolute values of the same terms, the scale of the rounding error
 * of any evaluation order. Returns 0, or -1 if the CSR is malformed (rowptr
 * not monotone from 0 to its end, or a column index outside [0, N)). */
int oracle_aggregate(const int64_t *rowptr, const int32_t *colidx, int64_t N,
                     const double *zeta, int32_t F, const int64_t *rows,
                     int64_t nrows, double *H, double *absterm);

/* ---- Back-propagation of one layer (Algorithm 1, Eqs. bp-H and bp-W). ----
 * G = dL/dzeta, Ht = dL/dH~, Wt~ = dL/dW~ below are all double. The layer's
 * binarized operands are H~ = diag(alpha) SF (N x K) and W~[k,j] =
 * beta_j SB[j,k] (K x F). */

/* Algorithm 1, first line: G = A~^T dH with A~ = D^-1/2 (A + I) D^-1/2,
 * applied as written: row i's incoming gradient is scattered to every j in
 * N(i) u {i} as dH[i,:] / sqrt(dhat_i dhat_j). Returns 0, or -1 for a
 * malformed CSR. */
int oracle_aggregate_t(const int64_t *rowptr, const int32_t *colidx, int64_t N,
                       const double *dH, int32_t F, double *G);

/* Algorithm 1: dL/dW~ = H~^T G, i.e. out[k,j] = sum_i alpha_i SF[i,k] G[i,j]
 * (K x F). absterm[j] (nullable) = sum_i |alpha_i G[i,j]|, the scale of any
 * evaluation order's rounding error (the same for every k). */
void oracle_grad_wtilde(const int8_t *SF, const double *alpha, const double *G,
                        int64_t N, int32_t K, int32_t F, double *out, double *absterm);

/* Algorithm 1: dL/dH~ = G W~^T (the printed "G . W~" is read with the
 * transpose the shapes require): out[i,k] = sum_j G[i,j] beta_j SB[j,k]
 * (N x K). absterm[i] (nullable) = sum_j |G[i,j] beta_j|. */
void oracle_grad_htilde(const double *G, const double *beta, const int8_t *SB,
                        int64_t N, int32_t K, int32_t F, double *out, double *absterm);

/* Eq. bp-H: dL/dH[i,k] = dL/dH~[i,k] * 1(|dL/dH~[i,k]| < 1), over n values. */
void oracle_grad_input(const double *Ht, int64_t n, double *out);

/* Eq. bp-W with d_in = K: out[k,j] = (1/K) SB[j,k] sum_m Wg[m,j] SB[j,m]
 * + beta_j Wg[k,j] 1(|W[k,j]| < 1), Wg = dL/dW~ (K x F), W = Wt (K x F,
 * row stride ldw), the straight-through estimator of sign() being
 * 1(|r| < 1). */
void oracle_grad_weight(const double *Wg, const int8_t *SB, const double *beta,
                        const float *Wt, int32_t K, int32_t F, int64_t ldw, double *out);

/* ---- Ablation variants of the product (Sec. 6.3, the transductive table's
 * "binarize features only" and "binarize weights only" rows): one operand of
 * Eq. 11 keeps its real values, the other is binarized as in Bi-GCN. ---- */

/* Weights binarized, features real: zeta = Y W~ with W~[k,j] = beta_j SB[j,k]:
 * zeta[i,j] = sum_k Y[i,k] beta_j SB[j,k] (N x F, double). absterm[i,j]
 * (nullable) = sum_k |Y[i,k]| beta_j, the scale of any evaluation order's
 * rounding error. */
void oracle_real_binary_product(const float *Y, int64_t N, int32_t K, const int8_t *SB,
                                const double *beta, int32_t F, double *zeta, double *absterm);

/* Features binarized, weights real: zeta = H~ W with H~[i,k] = alpha_i SF[i,k]
 * and W = Wt (K x F, row stride ldw): zeta[i,j] = sum_k alpha_i SF[i,k] W[k,j]
 * (N x F, double). absterm[i,j] (nullable) = sum_k alpha_i |W[k,j]|. */
void oracle_binary_real_product(const int8_t *SF, const double *alpha, int64_t N, int32_t K,
                                const float *Wt, int32_t F, int64_t ldw, double *zeta,
                                double *absterm);

/* ---- Inductive aggregators (Sec. 6.3's inductive models, Table 3, which
 * take GraphSAGE's definitions: the binarized feature extraction of every
 * node's own features first, then the aggregation of the products). ---- */

/* The "GCN" (mean) aggregator of inductive GCN: H[r,:] = (1/dhat_i) sum over
 * j in N(i) u {i} of zeta[j,:], dhat_i = 1 + |N(i)|, for each requested row
 * i = rows[r] (rows == NULL: all rows). absterm as in oracle_aggregate.
 * Returns 0, or -1 for a malformed CSR or row index. */
int oracle_aggregate_mean(const int64_t *rowptr, const int32_t *colidx, int64_t N,
                          const double *zeta, int32_t F, const int64_t *rows,
                          int64_t nrows, double *H, double *absterm);

/* GraphSAGE's mean aggregator with concatenation, W [h_i || mean_j h_j] =
 * W_self h_i + W_neigh mean_j h_j, applied to the products:
 * H[r,:] = zself[i,:] + (1/|N(i)|) sum over j in N(i) of zneigh[j,:]
 * (the mean is 0 for a node without neighbours). Returns 0 or -1 as above. */
int oracle_aggregate_sage(const int64_t *rowptr, const int32_t *colidx, int64_t N,
                          const double *zself, const double *zneigh, int32_t F,
                          const int64_t *rows, int64_t nrows, double *H, double *absterm);

/* ---- A weighted adjacency (Sec. 3: A = [a_ij] with general entries, d_i =
 * sum_j a_ij, A^ = A + I and D^_ii = sum_j a^_ij; Eq. 1's operator on it). The
 * CSR's values[e] is a_ij for the entry e = (i, colidx[e]); the weights must be
 * finite and non-negative. ---- */

/* dhat[i] = 1 + sum of values[e] over the entries e of row i. */
void oracle_degree_weighted(const int64_t *rowptr, const double *values, int64_t N,
                            double *dhat);

/* Eq. 13 with the weighted operator of Eq. 1: for each requested row
 * i = rows[r] (rows == NULL: all rows),
 *   H[r,:] = zeta[i,:] / dhat_i + sum over the entries e of row i of
 *            values[e] zeta[j,:] / sqrt(dhat_i dhat_j),   j = colidx[e],
 * the first term being the self-loop that I adds. absterm as in
 * oracle_aggregate. Returns 0, or -1 for a malformed CSR or row index or a
 * negative or non-finite weight. */
int oracle_aggregate_weighted(const int64_t *rowptr, const int32_t *colidx,
                              const double *values, int64_t N, const double *zeta,
                              int32_t F, const int64_t *rows, int64_t nrows, double *H,
                              double *absterm);

/* ---- Sub-row bucketing (Sec. 4.1: buckets of B consecutive values, each
 * scaled separately). Bucket b of a row (column) holds its entries k in
 * [bB, min(K, (b + 1)B)); nb = ceil(K / B) buckets. ---- */

/* alpha[i * nb + b] = mean over bucket b of |Y[i,k]| (Eq. 7 per bucket). */
void oracle_row_scale_bucketed(const float *Y, int64_t N, int32_t K, int32_t B, double *alpha);

/* beta[j * nb + b] = mean over bucket b of |Wt[k,j]| (Eq. 4 per bucket). */
void oracle_weight_scale_bucketed(const float *Wt, int32_t K, int32_t F, int64_t ldw, int32_t B,
                                  double *beta);

/* zeta[i,j] = sum over buckets b of alpha[i,b] beta[j,b] sum_{k in b} SF[i,k] SB[j,k]
 * (Eq. 11-12 with one scale pair per bucket). absterm[i,j] (nullable) = the
 * sum over b of |alpha[i,b] beta[j,b] dot_b|. */
void oracle_zeta_bucketed(const int8_t *SF, const double *alpha, int64_t N, const int8_t *SB,
                          const double *beta, int32_t F, int32_t K, int32_t B, double *zeta,
                          double *absterm);

#ifdef __cplusplus
}
#endif

#endif /* BIGCN_ORACLE_H */
