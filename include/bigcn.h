/*
 * bigcn.h -- C interface of the GB300 (sm_103a) Bi-GCN layer forward.
 *
 * Bi-GCN (Wang et al., "Bi-GCN: Binary Graph Convolutional Network", CVPR
 * 2021, arXiv:2010.07565) replaces the feature-extraction product H W of a
 * graph-convolution layer (Eq. 1) by a product of sign matrices scaled per
 * row and per column (Eqs. 10-12), then aggregates with the normalised
 * adjacency (Eq. 13). One layer is five steps, each one call below:
 *
 *   1+2  bigcn_pack_rows     centre (Sec. 6.2), sign-pack rows, row scale (Eqs. 7-8)
 *   3    bigcn_pack_weights  sign-pack weight columns, column scale (Eqs. 3-4)
 *   4    bigcn_xnor_gemm     XNOR/popcount product, scaled (Eqs. 11-12)
 *   5    bigcn_spmm_norm     H = D^-1/2 (A + I) D^-1/2 Z (Eqs. 1, 13)
 *        bigcn_layer_forward all five, fused where the layout allows
 *
 * Naming. The interface follows the layer's own naming, which swaps the
 * paper's letters: alpha_i is the per-NODE scale (the paper's beta_i, Eq. 7)
 * and beta_j is the per-WEIGHT-COLUMN scale (the paper's alpha_j, Eq. 4).
 * Both scales are the mean absolute value over the d_in = K entries of the
 * row / column (the least-squares optimum of the sign approximation; Eq. 4
 * and Eq. 7 as printed divide by d_out and N, which is read as a misprint).
 *
 * Conventions for every call:
 *  - Array pointers are DEVICE pointers owned by the caller. The library
 *    allocates no memory and keeps no state besides a per-device cache of
 *    the device's properties.
 *  - Every call is asynchronous on `stream` (a cudaStream_t; NULL = the
 *    legacy default stream). Outputs are valid once the stream reaches the
 *    call; inputs must stay valid until then.
 *  - Matrices are row-major with a leading dimension (row stride) in
 *    elements. Pointers must be aligned to their element size; faster
 *    vectorised paths are chosen internally when alignment allows.
 *  - Argument errors are detected on the host before any launch; the
 *    outputs are then untouched and nothing is enqueued.
 *  - Packed sign layout: element k of a packed row is bit (k % 64) of the
 *    row's 64-bit word k / 64, set for +1 and clear for -1, with
 *    sign(v) = +1 for v >= 0 (so +0 and -0 give +1; NaN gives -1). Rows
 *    hold `words` >= ceil(K / 64) words; every bit at k >= K is written 0.
 *  - Floating point is IEEE fp32 with round-to-nearest; the centring is one
 *    fused multiply-add, so the sign bits are reproducible bit for bit.
 *  - NaN or infinite inputs are not supported (results are unspecified, but
 *    every access stays in bounds).
 */
#ifndef BIGCN_H
#define BIGCN_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum bigcn_status {
    BIGCN_OK = 0,
    BIGCN_ERR_INVALID_ARG = 1,  /* null pointer, bad size, aliasing, short workspace */
    BIGCN_ERR_MISALIGNED = 2,   /* a pointer not aligned as documented */
    BIGCN_ERR_CUDA = 3,         /* a CUDA runtime error (launch or device query) */
    BIGCN_ERR_UNSUPPORTED = 4,  /* the current device is not sm_103 */
    BIGCN_ERR_SCRATCH_LIMIT = 5 /* bigcn_layer_forward_static: workspace > its static scratch */
} bigcn_status;

/* Human-readable name of a status code (static storage; never NULL). */
const char *bigcn_status_string(int status);

/* ceil(K / 64): the minimum `words` of a packed row of K signs (0 if K <= 0). */
int32_t bigcn_words(int32_t K);

/*
 * Steps 1+2. Centring (Sec. 6.2: batch normalisation of the input features,
 * inference form, as one fp32 fma per element) fused with the sign
 * binarization of node features (Eq. 8) and the per-node scale (Eq. 7):
 *
 *   y[i,k]    = fmaf(X[i,k], scale[k], shift[k])   (y = X if both are NULL)
 *   bits[i]   = packed sign(y[i,:])
 *   alpha[i]  = (1/K) sum_k |y[i,k]|
 *
 * X      N x K fp32, row stride ldx >= K.
 * scale, shift  K fp32 each, or both NULL (identity: layer 2 and beyond
 *        binarize their input raw, Sec. 4.1.2). Exactly one NULL is an error.
 * bits   N x words uint64, row stride `words` >= ceil(K/64).
 * alpha  N fp32.
 * N >= 0 (N == 0 enqueues nothing), 1 <= K, N * ldx and N * words < 2^62.
 */
bigcn_status bigcn_pack_rows(const float *X, int64_t N, int32_t K, int64_t ldx,
                             const float *scale, const float *shift,
                             uint64_t *bits, int32_t words, float *alpha,
                             void *stream);

/*
 * Step 3. Sign binarization of the weight columns (Eq. 3) and the
 * per-column scale (Eq. 4):
 *
 *   bits[j]  = packed sign(Wt[:, j])   (column j becomes packed row j)
 *   beta[j]  = (1/K) sum_k |Wt[k, j]|
 *
 * Wt     K x F fp32 (the layer's W, d_in x d_out), row stride ldw >= F.
 * bits   F x words uint64, words >= ceil(K/64).   beta  F fp32.
 * 1 <= K, 1 <= F.
 */
bigcn_status bigcn_pack_weights(const float *Wt, int32_t K, int32_t F, int64_t ldw,
                                uint64_t *bits, int32_t words, float *beta,
                                void *stream);

/*
 * Step 4. The binary feature extraction of Eqs. 11-12: the +-1 inner
 * product of packed row i of A with packed row j of B, evaluated as
 *
 *   dot[i,j] = K - 2 popcount(a_i XOR b_j)       (= sum_k sign * sign)
 *   Z[i,j]   = (alpha[i] * beta[j]) * (float)dot[i,j]
 *
 * a_bits N x words, alpha N;  b_bits F x words, beta F (from the two pack
 * calls, same K and words; all bits at k >= K must be 0, as they write).
 * Z      N x F fp32, row stride ldz >= F.
 * dots   nullable; if given, N x F int32 (row stride F) receives dot.
 * 0 <= N, 1 <= F, 1 <= K <= 64 * words. Z must not overlap the inputs.
 */
bigcn_status bigcn_xnor_gemm(const uint64_t *a_bits, const float *alpha, int64_t N,
                             const uint64_t *b_bits, const float *beta, int32_t F,
                             int32_t K, int32_t words, float *Z, int64_t ldz,
                             int32_t *dots, void *stream);

/*
 * Step 5. Aggregation with the normalised adjacency of Eq. 1 (Eq. 13):
 *
 *   H[i,:] = sum over j in N(i) u {i} of Z[j,:] / sqrt(dhat_i * dhat_j),
 *   dhat_i = 1 + (rowptr[i+1] - rowptr[i])     (A + I, Sec. 3.1)
 *
 * rowptr N+1 int64, colidx nnz int32: the CSR of A, unweighted, without
 *        self-loops (the call adds I). Symmetry is the caller's contract;
 *        the formula is evaluated for any CSR. rowptr[0] = 0,
 *        rowptr[N] = nnz, non-decreasing, 0 <= colidx < N. The kernel
 *        clamps row ranges to [0, nnz] and skips out-of-range column
 *        indices, so a malformed CSR gives wrong numbers, never a fault.
 * Z      N x F fp32, row stride ldz >= F.   H  N x F fp32, stride ldh >= F.
 * 0 <= N < 2^31, 0 <= nnz, 1 <= F. H must not overlap Z.
 */
bigcn_status bigcn_spmm_norm(const int64_t *rowptr, const int32_t *colidx,
                             int64_t N, int64_t nnz, const float *Z, int64_t ldz,
                             int32_t F, float *H, int64_t ldh, void *stream);

/*
 * Steps 4 and 5 with the degree normalisation split between them, as
 * bigcn_layer_forward runs them: D^-1/2 (A + I) D^-1/2 Z = D^-1/2 (A + I) Z'
 * with Z' = D^-1/2 Z (Eq. 1). bigcn_xnor_gemm_degscaled writes
 *
 *   Z'[i,j] = (alpha[i] * (1 / sqrt(dhat_i))) * (beta[j] * (float)dot[i,j]),
 *   dhat_i  = 1 + rowptr[i+1] - rowptr[i],
 *
 * and bigcn_spmm_prescaled then computes
 *
 *   H[i,:] = (1 / sqrt(dhat_i)) * sum over j in N(i) u {i} of Z'[j,:],
 *
 * which saves the aggregation one random read of the row pointers per edge.
 * Arguments, layouts and errors are those of bigcn_xnor_gemm (plus `rowptr`,
 * N+1 int64, required) and of bigcn_spmm_norm.
 */
bigcn_status bigcn_xnor_gemm_degscaled(const uint64_t *a_bits, const float *alpha, int64_t N,
                                       const uint64_t *b_bits, const float *beta, int32_t F,
                                       int32_t K, int32_t words, const int64_t *rowptr,
                                       float *Z, int64_t ldz, void *stream);

bigcn_status bigcn_spmm_prescaled(const int64_t *rowptr, const int32_t *colidx,
                                  int64_t N, int64_t nnz, const float *Z, int64_t ldz,
                                  int32_t F, float *H, int64_t ldh, void *stream);

/*
 * The XNOR product of step 4 runs on the tensor cores (tcgen05, the signs
 * as FP8 +-1, exact fp32 integer sums) when K >= 128, F >= 32 and N is at
 * least 128 rows per SM, and on the CUDA cores (XOR + popcount) otherwise;
 * the dots are identical either way.
 * Its kernels, and those of the ablation products below, wait on
 * shared-memory barriers with a bounded number of tries.
 * bigcn_device_timeouts synchronizes the current device, returns how
 * many such waits ran out since its last call (0 in correct operation; a
 * CTA whose wait ran out writes no output) and resets the count; -1 on a
 * CUDA error.
 */
int32_t bigcn_device_timeouts(void);

/* Bytes of device workspace bigcn_layer_forward needs for (N, K, F); 0 on
 * invalid sizes. */
size_t bigcn_layer_workspace_bytes(int64_t N, int32_t K, int32_t F);

/*
 * One binarized graph-convolution layer, H = A~ zeta (Eq. 13), with zeta from
 * the centred (scale/shift, as in bigcn_pack_rows) and binarized X and the
 * binarized W (Eqs. 3-12). The result equals the composition of the four
 * calls above within fp32 rounding; it runs the kernels of bigcn_pack_rows,
 * bigcn_pack_weights, bigcn_xnor_gemm_degscaled and bigcn_spmm_prescaled on
 * `stream`, except that when K <= 32767 the product keeps Z' factored in the
 * workspace -- the integer dots (as uint16 with a bias of 32768) and each
 * row's alpha_i / sqrt(dhat_i) -- and the aggregation applies the row factor
 * per neighbour and beta_j per column, gathering half the bytes. No
 * activation follows (Sec. 4.1.2).
 *
 * X N x K (ldx), Wt K x F (ldw), CSR as in bigcn_spmm_norm, H N x F (ldh).
 * workspace  device memory of at least bigcn_layer_workspace_bytes(N, K, F)
 *            bytes, 256-byte aligned, not overlapping any argument; its
 *            contents on entry do not matter and on exit are unspecified.
 * H must not overlap the workspace; it may not be X either.
 * The tensor-core product (many rows) waits on shared-memory barriers a
 * bounded number of times: a tile whose wait runs out leaves its part of the
 * product, and so of H, unwritten while the call still returns BIGCN_OK
 * (the call is asynchronous). bigcn_device_timeouts() reports such waits;
 * callers that must know call it after the layer (it synchronizes).
 */
bigcn_status bigcn_layer_forward(const float *X, int64_t N, int32_t K, int64_t ldx,
                                 const float *scale, const float *shift,
                                 const float *Wt, int32_t F, int64_t ldw,
                                 const int64_t *rowptr, const int32_t *colidx,
                                 int64_t nnz, void *workspace, size_t ws_bytes,
                                 float *H, int64_t ldh, void *stream);

/*
 * bigcn_layer_forward with timing events: event q of the n_events given
 * (cudaEvent_t as void*, nullable array) is recorded on `stream` before the
 * layer's kernel q (pack rows, pack weights, XNOR product, aggregation) and
 * event 4 after the last (as external events while the stream is being
 * captured); entries beyond 5 are not touched. When the rows are few and
 * long (fewer than a wave of warps), the rows are packed inside the product's
 * kernel and the first interval is empty. Everything else is
 * bigcn_layer_forward's.
 */
bigcn_status bigcn_layer_forward_timed(const float *X, int64_t N, int32_t K, int64_t ldx,
                                       const float *scale, const float *shift,
                                       const float *Wt, int32_t F, int64_t ldw,
                                       const int64_t *rowptr, const int32_t *colidx,
                                       int64_t nnz, void *workspace, size_t ws_bytes,
                                       float *H, int64_t ldh, void *const *events,
                                       int32_t n_events, void *stream);

/*
 * The two-layer Bi-GCN of Sec. 6.2 in one call: a hidden layer of width Fh on
 * the centred features (scale/shift as in bigcn_pack_rows) and an output
 * layer of width Fo on the hidden layer's output taken raw (no activation,
 * Sec. 4.1.2), both H = A~ zeta (Eq. 13) over the same graph:
 *
 *   H1  = D^-1/2 (A + I) D^-1/2 zeta(X centred, W1)      N x Fh
 *   out = D^-1/2 (A + I) D^-1/2 zeta(H1, W2)             N x Fo (the logits)
 *
 * The result equals two bigcn_layer_forward calls within fp32 rounding.
 * Fusions, when the widths allow: layer 1's centring, packing and XNOR
 * product run as one kernel whose packed rows stay in shared memory
 * (Fh <= 128 and the packed tiles fit); and when Fh is a multiple of 4 and at
 * most 128 and Fo <= 64, layer 1's aggregation kernel also binarizes H1 and
 * computes layer 2's XNOR product while the row is in registers, so H1 never
 * goes through memory. When K <= 32767, layer 1's Z' stays factored in the
 * workspace (integer dots as biased uint16 and a row scale, as in
 * bigcn_layer_forward), so its aggregation gathers half-size rows. When
 * K <= 2048 (the dots exact in fp16), Fh <= 128 and Fo <= 64, both products
 * stay factored as fp16 dots and a row scale and both aggregations run on the
 * tensor cores (bigcn_forward_2layer_aggregation); layer 1's aggregation then
 * binarizes H1 and computes layer 2's dots for any Fh <= 128. The call
 * launches 4 to 7 kernels (bigcn_forward_2layer_launches).
 *
 * X N x K (ldx), W1 K x Fh (ldw1), W2 Fh x Fo (ldw2), CSR as in
 * bigcn_spmm_norm, out N x Fo (ldo).
 * H1         nullable; if given (N x Fh, ldh1) it also receives layer 1's output.
 * workspace  >= bigcn_forward_2layer_workspace_bytes(N, K, Fh, Fo) bytes of
 *            device memory, 256-byte aligned, overlapping nothing else.
 * events     nullable array of n_events cudaEvent_t (as void*): event q is
 *            recorded on `stream` before kernel q and the last one after the
 *            last kernel (recorded with cudaEventRecordExternal), for timing
 *            each kernel; entries beyond launches + 1 are not touched.
 * pred       nullable N int32: each node's predicted class, the argmax of its
 *            logits row (lowest index on ties; computed in the last
 *            aggregation's epilogue, or by one more kernel when Fo > 256).
 * out, H1, pred and the workspace must not overlap each other or any input.
 */
size_t bigcn_forward_2layer_workspace_bytes(int64_t N, int32_t K, int32_t Fh, int32_t Fo);

/* Kernel launches bigcn_forward_2layer makes for these sizes on the current
 * device (4 to 7), or -1 on invalid sizes or a device error. */
int32_t bigcn_forward_2layer_launches(int64_t N, int32_t K, int32_t Fh, int32_t Fo);

/* Which aggregation bigcn_forward_2layer runs for these widths: 1 = both on
 * the tensor cores over fp16 dots, 0 = on the CUDA cores, -1 = invalid sizes.
 * An interface query with no counterpart in the paper (it selects how the
 * sums of Eq. 13 are evaluated, not what they are); needs no device. */
int32_t bigcn_forward_2layer_aggregation(int32_t K, int32_t Fh, int32_t Fo);

bigcn_status bigcn_forward_2layer(const float *X, int64_t N, int32_t K, int64_t ldx,
                                  const float *scale, const float *shift,
                                  const float *W1, int32_t Fh, int64_t ldw1,
                                  const float *W2, int32_t Fo, int64_t ldw2,
                                  const int64_t *rowptr, const int32_t *colidx, int64_t nnz,
                                  void *workspace, size_t ws_bytes,
                                  float *H1, int64_t ldh1, float *out, int64_t ldo,
                                  int32_t *pred, void *const *events, int32_t n_events,
                                  void *stream);

/*
 * Ablation variants of the layer (Sec. 6.3, the transductive table's rows
 * "binarize weights only" and "binarize features only"): one operand of the
 * product of Eq. 11 keeps its real fp32 values, the other is binarized as in
 * Bi-GCN (sign and mean-|.| scale, Eqs. 3-4 / 7-8).
 *
 * Both products run on the tensor cores: the real operand is split into
 * three bf16 parts whose sum equals it to within 2^-24 of its magnitude
 * (each part the bf16 rounding of what the earlier parts leave), the signs
 * are exact in bf16, and the three products are accumulated in fp32. The
 * result is therefore that of an fp32 evaluation of the sum in some order.
 * Sums over K may be split between the CTAs of a cluster and added in a
 * fixed order, so results are deterministic.
 */
typedef enum bigcn_binarize {
    BIGCN_BINARIZE_BOTH = 0,      /* Bi-GCN: zeta = H~ W~ (Eqs. 11-12) */
    BIGCN_BINARIZE_WEIGHTS = 1,   /* features real:  zeta = Y W~ */
    BIGCN_BINARIZE_FEATURES = 2   /* weights real:   zeta = H~ W */
} bigcn_binarize;

/*
 * zeta = Y W~ with Y[i,k] = fmaf(X[i,k], scale[k], shift[k]) (the centring of
 * bigcn_pack_rows; scale == shift == NULL: Y = X) and W~[k,j] =
 * beta[j] * (bit k of column j ? +1 : -1):
 *
 *   Z[i,j] = beta[j] * sum_k Y[i,k] * sign_jk.
 *
 * X N x K (row stride ldx >= K), b_bits/beta from bigcn_pack_weights (F x
 * words, words = bigcn_words(K)), Z N x F (row stride ldz >= F). Z must not
 * overlap an input. Pointers 4-byte aligned (b_bits 8).
 */
bigcn_status bigcn_real_binary_gemm(const float *X, int64_t N, int32_t K, int64_t ldx,
                                    const float *scale, const float *shift,
                                    const uint64_t *b_bits, const float *beta, int32_t F,
                                    int32_t words, float *Z, int64_t ldz, void *stream);

/* Bytes of device workspace bigcn_binary_real_gemm needs (the bf16 parts of
 * W); 0 on invalid sizes. */
size_t bigcn_binary_real_gemm_workspace_bytes(int32_t K, int32_t F);

/*
 * zeta = H~ W with H~[i,k] = alpha[i] * (bit k of row i ? +1 : -1):
 *
 *   Z[i,j] = alpha[i] * sum_k sign_ik * W[k,j].
 *
 * a_bits/alpha from bigcn_pack_rows (N x words), Wt K x F (row stride
 * ldw >= F), Z N x F (row stride ldz >= F). workspace >=
 * bigcn_binary_real_gemm_workspace_bytes(K, F) bytes, 256-byte aligned;
 * neither it nor Z may overlap an input or each other.
 */
bigcn_status bigcn_binary_real_gemm(const uint64_t *a_bits, const float *alpha, int64_t N,
                                    int32_t K, int32_t words, const float *Wt, int32_t F,
                                    int64_t ldw, void *workspace, size_t ws_bytes, float *Z,
                                    int64_t ldz, void *stream);

/* Bytes of device workspace bigcn_layer_forward_ablation needs; 0 on invalid
 * sizes or an unknown `binarize`. */
size_t bigcn_layer_ablation_workspace_bytes(int32_t binarize, int64_t N, int32_t K, int32_t F);

/*
 * One graph-convolution layer H = A~ zeta (Eq. 13) with zeta binarized as
 * `binarize` (a bigcn_binarize) says. BIGCN_BINARIZE_BOTH is
 * bigcn_layer_forward. The others run bigcn_pack_weights (resp.
 * bigcn_pack_rows) and the product above with each row j multiplied by
 * 1/sqrt(dhat_j), then bigcn_spmm_prescaled. Arguments, layouts and errors
 * are bigcn_layer_forward's, with this call's workspace size.
 */
bigcn_status bigcn_layer_forward_ablation(int32_t binarize, const float *X, int64_t N,
                                          int32_t K, int64_t ldx, const float *scale,
                                          const float *shift, const float *Wt, int32_t F,
                                          int64_t ldw, const int64_t *rowptr,
                                          const int32_t *colidx, int64_t nnz, void *workspace,
                                          size_t ws_bytes, float *H, int64_t ldh, void *stream);

/*
 * Sub-row bucketing (Sec. 4.1: the matrix split into buckets of B consecutive
 * values, each scaled separately). Bucket b of a node row / weight column
 * holds entries k in [bB, min(K, (b + 1)B)); nb = ceil(K / B). B must be a
 * positive multiple of 64 (a bucket is whole packed words) with nb <= 65535;
 * B >= K is one bucket, i.e. Bi-GCN. The packed signs are bigcn_pack_rows' /
 * bigcn_pack_weights'; the scales gain a bucket index:
 *
 *   alpha[i * nb + b] = mean over bucket b of |y_ik|   (N x nb)
 *   beta[j * nb + b]  = mean over bucket b of |W_kj|   (F x nb)
 *   Z[i,j] = sum over b of alpha_ib beta_jb (signs in b - 2 popc over b's words)
 *
 * Z is accumulated in fp32 bucket by bucket (exact integer counts per bucket).
 */
bigcn_status bigcn_pack_rows_bucketed(const float *X, int64_t N, int32_t K, int64_t ldx,
                                      const float *scale, const float *shift, int32_t B,
                                      uint64_t *bits, int32_t words, float *alpha, void *stream);

bigcn_status bigcn_pack_weights_bucketed(const float *Wt, int32_t K, int32_t F, int64_t ldw,
                                         int32_t B, uint64_t *bits, int32_t words, float *beta,
                                         void *stream);

/* words must equal bigcn_words(K). */
bigcn_status bigcn_xnor_gemm_bucketed(const uint64_t *a_bits, const float *alpha, int64_t N,
                                      const uint64_t *b_bits, const float *beta, int32_t F,
                                      int32_t K, int32_t words, int32_t B, float *Z, int64_t ldz,
                                      void *stream);

/* Bytes of device workspace bigcn_layer_forward_bucketed needs; 0 on invalid sizes. */
size_t bigcn_layer_bucketed_workspace_bytes(int64_t N, int32_t K, int32_t F, int32_t B);

/*
 * One layer H = A~ zeta (Eq. 13) with bucketed binarization: the three calls
 * above (the product's rows multiplied by 1/sqrt(dhat_i)), then
 * bigcn_spmm_prescaled. Arguments, layouts and errors are bigcn_layer_forward's
 * plus B, with this call's workspace size.
 */
bigcn_status bigcn_layer_forward_bucketed(int32_t B, const float *X, int64_t N, int32_t K,
                                          int64_t ldx, const float *scale, const float *shift,
                                          const float *Wt, int32_t F, int64_t ldw,
                                          const int64_t *rowptr, const int32_t *colidx,
                                          int64_t nnz, void *workspace, size_t ws_bytes,
                                          float *H, int64_t ldh, void *stream);

/*
 * Binarized layers of inductive GNNs (Sec. 6.3, Table 3: Bi-inductiveGCN and
 * Bi-GraphSAGE, which binarize every feature-extraction step of GraphSAGE's
 * models). The product of Eqs. 10-12 is taken on every node's own features,
 * then one of these aggregators combines the products:
 */
typedef enum bigcn_aggregator {
    BIGCN_AGG_GCN = 0,    /* Eq. 1: D^-1/2 (A + I) D^-1/2 zeta (bigcn_layer_forward) */
    BIGCN_AGG_MEAN = 1,   /* inductive GCN: H_i = mean of zeta_j over j in N(i) u {i} */
    BIGCN_AGG_SAGE = 2    /* GraphSAGE-mean: H_i = zeta_i + mean over j in N(i) of
                             zeta'_j, zeta' the product with a second weight matrix
                             W_neigh (0 for a node without neighbours) */
} bigcn_aggregator;

/* Bytes of device workspace bigcn_inductive_layer_forward needs; 0 on invalid
 * sizes or an unknown aggregator. */
size_t bigcn_inductive_layer_workspace_bytes(int32_t aggregator, int64_t N, int32_t K,
                                             int32_t F);

/*
 * One inductive layer. X, scale/shift, Wt (K x F, ldw), the CSR, workspace,
 * H and the errors are those of bigcn_layer_forward. W_neigh (K x F, row
 * stride ldwn >= F) is required for BIGCN_AGG_SAGE and ignored otherwise; its
 * columns are binarized like Wt's (their own signs and mean-|.| scales).
 * BIGCN_AGG_SAGE computes both products with one XNOR product over the
 * concatenated columns [Wt | W_neigh] (each half padded to a multiple of 8
 * columns) and keeps them factored like bigcn_layer_forward's when
 * K <= 32767. The mean over N(i) uses the CSR's row lengths, so a malformed
 * CSR (skipped indices) still divides by the listed degree.
 */
bigcn_status bigcn_inductive_layer_forward(int32_t aggregator, const float *X, int64_t N,
                                           int32_t K, int64_t ldx, const float *scale,
                                           const float *shift, const float *Wt, int32_t F,
                                           int64_t ldw, const float *W_neigh, int64_t ldwn,
                                           const int64_t *rowptr, const int32_t *colidx,
                                           int64_t nnz, void *workspace, size_t ws_bytes,
                                           float *H, int64_t ldh, void *stream);

/*
 * A weighted adjacency. Sec. 3 writes A = [a_ij] with general entries, the
 * degree d_i = sum_j a_ij, A^ = A + I and D^_ii = sum_j a^_ij, and Eq. 1's
 * operator D^-1/2 A^ D^-1/2 on that; the entry points above are the case
 * a_ij = 1. Here `values` holds a_ij for each CSR entry (nnz fp32, in the
 * order of colidx). Weights must be finite and >= 0: a negative degree has
 * no square root and gives NaN or Inf outputs (never a fault); the calls do
 * not check it. Symmetry of the weights is the caller's contract, as the
 * CSR's; the formulas below are evaluated for any weights.
 *
 * bigcn_weighted_dinv: dinv[i] = 1 / sqrt(1 + sum over the entries e of
 * row i of values[e]) for i < N (rows summed with compensated fp32 adds).
 * rowptr (N+1 int64) and values (nnz) as above, dinv N fp32 written, not
 * overlapping them. 0 <= N < 2^31, 0 <= nnz; values may be NULL when
 * nnz == 0.
 */
bigcn_status bigcn_weighted_dinv(const int64_t *rowptr, const float *values, int64_t N,
                                 int64_t nnz, float *dinv, void *stream);

/*
 * Step 5 over a weighted A (Eq. 13 with Eq. 1's operator):
 *
 *   H[i,:] = dinv_i * (dinv_i Z[i,:] + sum over the entries e of row i of
 *            values[e] * dinv_j * Z[j,:]),   j = colidx[e],
 *
 * with dinv from bigcn_weighted_dinv on the same rowptr and values. The CSR,
 * Z, H and the errors are those of bigcn_spmm_norm; values (nnz) and dinv
 * (N) are read only and must not overlap H.
 */
bigcn_status bigcn_spmm_norm_weighted(const int64_t *rowptr, const int32_t *colidx,
                                      const float *values, const float *dinv, int64_t N,
                                      int64_t nnz, const float *Z, int64_t ldz, int32_t F,
                                      float *H, int64_t ldh, void *stream);

/* Bytes of device workspace bigcn_weighted_layer_forward needs; 0 on invalid
 * sizes. */
size_t bigcn_weighted_layer_workspace_bytes(int64_t N, int32_t K, int32_t F);

/*
 * One binarized layer over a weighted A: H = D^-1/2 (A + I) D^-1/2 zeta with
 * zeta as in bigcn_layer_forward. Runs the kernels of bigcn_pack_rows,
 * bigcn_pack_weights, bigcn_weighted_dinv (which also forms each row's scale
 * s_j = alpha_j dinv_j), bigcn_xnor_gemm with s as its row scale (kept
 * factored, uint16 dots and s_j, when K <= 32767) and the weighted
 * aggregation. Arguments and errors are those of bigcn_layer_forward plus
 * `values` (nnz fp32, not overlapping the workspace or H); the workspace is
 * bigcn_weighted_layer_workspace_bytes(N, K, F) bytes, 256-byte aligned. The
 * tensor-core product's bounded waits behave as in bigcn_layer_forward.
 */
bigcn_status bigcn_weighted_layer_forward(const float *X, int64_t N, int32_t K, int64_t ldx,
                                          const float *scale, const float *shift,
                                          const float *Wt, int32_t F, int64_t ldw,
                                          const int64_t *rowptr, const int32_t *colidx,
                                          const float *values, int64_t nnz, void *workspace,
                                          size_t ws_bytes, float *H, int64_t ldh,
                                          void *stream);

/*
 * Back-propagation of one layer (Algorithm 1 with Eqs. bp-H and bp-W), from
 * the gradient dH = dL/dH^(l+1) of the layer's output (N x F, row stride ldg)
 * to
 *   dX = dL/dH^(l) (nullable; N x K, row stride lddx): Algorithm 1's
 *        dL/dH~ = G W~^T clipped by Eq. bp-H (entries with |.| >= 1 are 0),
 *        the gradient of the layer's binarized input (for layer 1, the
 *        centred features);
 *   dW = dL/dW (K x F, row stride lddw): Eq. bp-W with d_in = K and the
 *        straight-through estimator 1(|W| < 1) of sign(),
 * where G = A~^T dH, dL/dW~ = H~^T G, H~ = diag(alpha) sign(Y) and W~ =
 * sign(W) diag(beta) are those of the forward with the same X, scale/shift
 * and Wt (the signs and scales are recomputed from them). A~^T is applied as
 * A~: the CSR must be symmetric, as everywhere in this interface.
 * workspace  >= bigcn_layer_backward_workspace_bytes(N, K, F) bytes of device
 *            memory, 256-byte aligned, overlapping no argument.
 * dX and dW must not overlap each other or any input. The sums over the N
 * rows (dW) are evaluated in a fixed order (chunks of rows added in order).
 */
size_t bigcn_layer_backward_workspace_bytes(int64_t N, int32_t K, int32_t F);

bigcn_status bigcn_layer_backward(const float *X, int64_t N, int32_t K, int64_t ldx,
                                  const float *scale, const float *shift,
                                  const float *Wt, int32_t F, int64_t ldw,
                                  const int64_t *rowptr, const int32_t *colidx, int64_t nnz,
                                  const float *dH, int64_t ldg, float *dX, int64_t lddx,
                                  float *dW, int64_t lddw, void *workspace, size_t ws_bytes,
                                  void *stream);

/*
 * The aggregation of Eq. 13 for a block of output rows whose neighbours'
 * pre-scaled rows come from a separate table: a shard of the graph in a
 * multi-GPU layer (rows partitioned across GPUs, every GPU holding its own rows
 * of Z' followed by the rows of the neighbours other GPUs own -- its halo).
 *
 *   H_i = (1/sqrt(dhat_i)) * sum over q in N(i) u {i} of Z'[q]      i < n_rows
 *
 * rowptr (n_rows + 1) and colidx (nnz) describe the block's rows in the
 * table's numbering: entries of a row are indices into Z' (0 <= q < n_cols),
 * the self-loop of row i is Z'[i] (a block's own rows come first), and dhat_i
 * = 1 + the row's length (its full degree in the whole graph). Z' rows must
 * already carry their own 1/sqrt(dhat_q) (bigcn_xnor_gemm_degscaled on the
 * owning GPU). n_cols >= n_rows; other arguments, layouts and errors as in
 * bigcn_spmm_prescaled, which it equals when n_cols == n_rows.
 */
bigcn_status bigcn_spmm_prescaled_rows(const int64_t *rowptr, const int32_t *colidx,
                                       int64_t n_rows, int64_t n_cols, int64_t nnz,
                                       const float *Z, int64_t ldz, int32_t F, float *H,
                                       int64_t ldh, void *stream);

/* Bytes of the device scratch array behind bigcn_layer_forward_static. */
#define BIGCN_STATIC_SCRATCH_BYTES ((size_t)32 << 20)

/*
 * bigcn_layer_forward without a caller-supplied workspace, for callers that
 * cannot allocate device memory: serving loops that forbid cudaMalloc and
 * cudaFree in steady state because both can stall the whole device,
 * plug-ins whose host application owns every byte of the device memory
 * budget, and deployments that must fix their memory footprint when they
 * load. (The paper has no counterpart: this is an interface convenience.)
 *
 * The workspace is a file-scope __device__ array of BIGCN_STATIC_SCRATCH_BYTES
 * (32 MiB) inside this library. Every GPU on which the library's device code
 * is loaded holds that array until the process exits. The call allocates
 * nothing: no cudaMalloc, no cudaFree, no allocating library routine.
 *
 * Arguments, results and errors are those of bigcn_layer_forward minus
 * `workspace` and `ws_bytes`, plus: when bigcn_layer_workspace_bytes(N, K, F)
 * exceeds BIGCN_STATIC_SCRATCH_BYTES the call returns
 * BIGCN_ERR_SCRATCH_LIMIT and enqueues nothing. The exact test is
 * bigcn_layer_workspace_bytes(N, K, F) <= BIGCN_STATIC_SCRATCH_BYTES. Per
 * node that is 8*ceil(K/64) + 2*round_up(F, 8) + 8 bytes when K <= 32767
 * (the dots kept as 16-bit integers) and 8*ceil(K/64) + 4*F + 4 bytes above,
 * plus the packed weights: about 155,000 nodes fit with K = 602 and F = 64.
 * As in bigcn_layer_forward, a bounded device wait that runs out leaves
 * part of H unwritten while the call returns BIGCN_OK; bigcn_device_timeouts()
 * (which synchronizes) reports it.
 *
 * The first call on a device, with that device current, looks up the array's
 * device address (cudaGetSymbolAddress) and caches it for the device; make
 * that first call before any stream capture begins. Every call on a device
 * shares the one array and overwrites it; the layer writes every scratch
 * byte it reads, so nothing has to start at zero, but two calls whose
 * kernels overlap on the GPU (e.g. on two streams, or on one device from two
 * threads without ordering) race on the array and give wrong results.
 */
bigcn_status bigcn_layer_forward_static(const float *X, int64_t N, int32_t K, int64_t ldx,
                                        const float *scale, const float *shift,
                                        const float *Wt, int32_t F, int64_t ldw,
                                        const int64_t *rowptr, const int32_t *colidx,
                                        int64_t nnz, float *H, int64_t ldh, void *stream);

#ifdef __cplusplus
}
#endif

#endif /* BIGCN_H */
