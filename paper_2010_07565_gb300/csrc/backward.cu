// Back-propagation of one Bi-GCN layer (Wang et al., CVPR 2021, Algorithm 1,
// Eqs. bp-H and bp-W), from dL/dH^(l+1) (dH, N x F) to the gradient of the
// layer's binarized input and of its weights:
//
//   G      = A~^T dH                 = A~ dH (the CSR is symmetric)
//   dW~    = H~^T G,  H~ = diag(alpha) sign(Y)          (K x F)
//   dH~    = G W~^T,  W~[k,j] = beta_j sign(W_kj)       (N x K)
//   dL/dH  = dH~ * 1(|dH~| < 1)                          Eq. bp-H
//   dL/dW  = (1/K) B_kj sum_m dW~_mj B_mj
//            + beta_j dW~_kj 1(|W_kj| < 1)               Eq. bp-W
//
// (alpha: per-node scale, the paper's beta; beta: per-column scale, the
// paper's alpha; B = sign(W).) The signs come packed from the forward's own
// kernels (the rows re-packed from X with the same centring, the columns
// from W). Both products multiply a +-1 matrix by an fp32 one. dH~ runs on
// the tensor cores through the real x binary product of ablation.cu: the
// real operand G (times beta_j, applied as its centring scale and rounded
// once) split into three bf16 parts, the signs of W's rows (W packed row by
// row over its F columns) exact in bf16, fp32 accumulators, and the clip of
// Eq. bp-H in the epilogue. dW~ runs on the tensor cores too
// (sign_t_real_tc_kernel in ablation.cu): the node signs gathered
// feature-major from the packed rows, alpha_i G_ij as three bf16 parts.
//
// dW~ sums over all N rows: the rows are split into S chunks (grid z) whose
// partial sums are added, chunk by chunk in order, by a second kernel, so
// the result does not depend on scheduling.
#include "launch.cuh"

namespace bigcn {
namespace {

constexpr int kBwThreads = 256;
constexpr int kTile = 64;        // output tile edge

// +1.0f where bit b of w is set, else -1.0f.
__device__ __forceinline__ float pm1(uint64_t w, int b) {
    return ((w >> b) & 1ull) ? 1.0f : -1.0f;
}

// dW~ = the S partial sums added in chunk order.
__global__ void __launch_bounds__(kBwThreads)
sum_partials_kernel(const float *__restrict__ partial, int S, int64_t n, float *__restrict__ out) {
    for (int64_t q = int64_t(blockIdx.x) * kBwThreads + threadIdx.x; q < n;
         q += int64_t(gridDim.x) * kBwThreads) {
        float t = 0.0f;
        for (int s = 0; s < S; ++s) t += __ldg(partial + int64_t(s) * n + q);
        out[q] = t;
    }
}

constexpr int kColGroups = 32;   // row groups of the column-sum block (1024 threads)

// Eq. bp-W, first term's sum: c_j = sum_k dW~_kj B_kj. One block per 32
// columns: thread (c, g) sums rows g, g + 32, ... of column c (coalesced
// across the 32 columns), and the 32 group sums are added in group order.
__global__ void __launch_bounds__(32 * kColGroups)
weight_colsum_kernel(const float *__restrict__ Wg, const uint64_t *__restrict__ wbits, int words,
                     int K, int F, float *__restrict__ csum) {
    __shared__ float part[kColGroups][32];
    const int cl = threadIdx.x & 31, g = threadIdx.x >> 5;
    const int j = blockIdx.x * 32 + cl;
    float acc = 0.0f;
    if (j < F) {
        const uint64_t *wb = wbits + int64_t(j) * words;
        for (int k = g; k < K; k += kColGroups)
            acc = fmaf(__ldg(Wg + int64_t(k) * F + j), pm1(__ldg(wb + k / 64), k % 64), acc);
    }
    part[g][cl] = acc;
    __syncthreads();
    if (g == 0 && j < F) {
        float t = 0.0f;
        for (int q = 0; q < kColGroups; ++q) t += part[q][cl];
        csum[j] = t;
    }
}

// Eq. bp-W, every entry: dW_kj = B_kj c_j / K + beta_j dW~_kj 1(|W_kj| < 1).
__global__ void __launch_bounds__(kBwThreads)
grad_weight_kernel(const float *__restrict__ Wg, const uint64_t *__restrict__ wbits, int words,
                   const float *__restrict__ beta, const float *__restrict__ csum,
                   const float *__restrict__ Wt, int64_t ldw, int K, int F,
                   float *__restrict__ dW, int64_t lddw) {
    const int64_t n = int64_t(K) * F;
    for (int64_t q = int64_t(blockIdx.x) * kBwThreads + threadIdx.x; q < n;
         q += int64_t(gridDim.x) * kBwThreads) {
        const int k = int(q / F), j = int(q % F);
        const float w = __ldg(Wt + int64_t(k) * ldw + j);
        const float ste = fabsf(w) < 1.0f ? 1.0f : 0.0f;
        const float b = pm1(__ldg(wbits + int64_t(j) * words + k / 64), k % 64);
        dW[int64_t(k) * lddw + j] = b * (__ldg(csum + j) / float(K)) +
                                    __ldg(beta + j) * __ldg(Wg + q) * ste;
    }
}

constexpr size_t kAlign = 256;
size_t round_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Most row chunks the dW~ reduction may use for a K x F output: enough for
// about two blocks per SM on up to 256 SMs, at most 64.
int64_t max_chunks(int K, int F) {
    const int64_t tiles = int64_t((K + kTile - 1) / kTile) * ((F + kTile - 1) / kTile);
    const int64_t s = (512 + tiles - 1) / tiles;
    return s < 64 ? s : 64;
}

struct BackwardWorkspace {
    size_t bits, alpha, wbits, beta, g, wg, partial, wrows, wrow_scale, csum, total;
};

bool backward_workspace(int64_t N, int32_t K, int32_t F, BackwardWorkspace *w) {
    if (N < 0 || K < 1 || F < 1) return false;
    const int64_t words = bigcn_words(K);
    if (N > kMaxElems / (words > F ? words : F)) return false;
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t at = off; off = round_up(off + bytes); return at; };
    w->bits = take(size_t(N) * words * 8);
    w->alpha = take(size_t(N) * 4);
    w->wbits = take(size_t(F) * words * 8);
    w->beta = take(size_t(F) * 4);
    w->g = take(size_t(N) * F * 4);
    w->wg = take(size_t(K) * F * 4);
    w->partial = take(size_t(max_chunks(K, F)) * K * F * 4);
    w->wrows = take(size_t(K) * size_t(bigcn_words(F)) * 8);   // W's rows packed over F
    w->wrow_scale = take(size_t(K) * 4);                         // (their row scales, unused)
    w->csum = take(size_t(F) * 4);
    w->total = off;
    return true;
}

}  // namespace
}  // namespace bigcn

using namespace bigcn;

extern "C" size_t bigcn_layer_backward_workspace_bytes(int64_t N, int32_t K, int32_t F) {
    BackwardWorkspace w;
    return backward_workspace(N, K, F, &w) ? w.total : 0;
}

extern "C" bigcn_status bigcn_layer_backward(
    const float *X, int64_t N, int32_t K, int64_t ldx, const float *scale, const float *shift,
    const float *Wt, int32_t F, int64_t ldw, const int64_t *rowptr, const int32_t *colidx,
    int64_t nnz, const float *dH, int64_t ldg, float *dX, int64_t lddx, float *dW, int64_t lddw,
    void *workspace, size_t ws_bytes, void *stream) {
    BackwardWorkspace w;
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || ldx < K || ldw < F || ldg < F ||
        (dX && lddx < K) || lddw < F || nnz < 0)
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (!backward_workspace(N, K, F, &w)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / ldg || (dX && N > kMaxElems / lddx)))
        return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw || int64_t(K) > kMaxElems / lddw) return BIGCN_ERR_INVALID_ARG;
    if (!Wt || !dW) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (!X || !rowptr || !dH || !workspace || (nnz > 0 && !colidx)))
        return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && ws_bytes < w.total) return BIGCN_ERR_INVALID_ARG;
    if ((X && !aligned_to(X, 4)) || !aligned_to(Wt, 4) || (rowptr && !aligned_to(rowptr, 8)) ||
        (colidx && !aligned_to(colidx, 4)) || (dH && !aligned_to(dH, 4)) ||
        (dX && !aligned_to(dX, 4)) || !aligned_to(dW, 4) ||
        (workspace && !aligned_to(workspace, kAlign)) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t dwb = span_bytes(K, F, lddw, 4), dxb = dX ? span_bytes(N, K, lddx, 4) : 0;
    const void *in[] = {X, Wt, rowptr, colidx, dH, scale, shift};
    const size_t in_bytes[] = {span_bytes(N, K, ldx, 4), span_bytes(K, F, ldw, 4),
                               size_t(N + 1) * 8, size_t(nnz) * 4, span_bytes(N, F, ldg, 4),
                               size_t(K) * 4, size_t(K) * 4};
    const void *outs[] = {dW, dX, N > 0 ? workspace : nullptr};
    const size_t out_bytes[] = {dwb, dxb, N > 0 ? w.total : 0};
    for (int o = 0; o < 3; ++o) {
        for (int q = 0; q < 7; ++q)
            if (overlaps(outs[o], out_bytes[o], in[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
        for (int p = o + 1; p < 3; ++p)
            if (overlaps(outs[o], out_bytes[o], outs[p], out_bytes[p])) return BIGCN_ERR_INVALID_ARG;
    }
    DeviceInfo dev;
    bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    cudaStream_t s = as_stream(stream);
    if (N == 0) {       // no rows: dW~ = 0, so dW = 0
        if (cudaMemset2DAsync(dW, size_t(lddw) * 4, 0, size_t(F) * 4, size_t(K), s) != cudaSuccess) {
            cudaGetLastError();
            return BIGCN_ERR_CUDA;
        }
        return BIGCN_OK;
    }

    char *ws = static_cast<char *>(workspace);
    uint64_t *bits = reinterpret_cast<uint64_t *>(ws + w.bits);
    float *alpha = reinterpret_cast<float *>(ws + w.alpha);
    uint64_t *wbits = reinterpret_cast<uint64_t *>(ws + w.wbits);
    float *beta = reinterpret_cast<float *>(ws + w.beta);
    float *G = reinterpret_cast<float *>(ws + w.g);
    float *Wg = reinterpret_cast<float *>(ws + w.wg);
    float *partial = reinterpret_cast<float *>(ws + w.partial);
    const int words = bigcn_words(K);

    launch_pack_rows(X, N, K, ldx, scale, shift, bits, words, alpha, dev, s);
    launch_pack_weights(Wt, K, F, ldw, wbits, words, beta, s);
    SpmmArgs a{rowptr, colidx, N, nnz, dH, ldg, F, G, F, false, false};
    launch_spmm_norm(a, dev, s);                                   // G = A~ dH
    // dL/dW~ = H~^T G on the tensor cores, in node chunks added in order.
    SignTRealArgs gw{bits, words, alpha, G, F, N, K, F, partial};
    const int S = launch_sign_t_real_gemm(gw, int(max_chunks(K, F)), dev, s);
    const int64_t kf = int64_t(K) * F;
    sum_partials_kernel<<<unsigned((kf + kBwThreads - 1) / kBwThreads < 4096
                                       ? (kf + kBwThreads - 1) / kBwThreads : 4096),
                          kBwThreads, 0, s>>>(partial, S, kf, Wg);
    if (dX) {
        // dH~ = (G diag(beta)) sign(W)^T with the clip of Eq. bp-H: contraction
        // over F, one output column per feature k.
        uint64_t *wrows = reinterpret_cast<uint64_t *>(ws + w.wrows);
        float *wrow_scale = reinterpret_cast<float *>(ws + w.wrow_scale);
        const int fwords = bigcn_words(F);
        launch_pack_rows(Wt, K, F, ldw, nullptr, nullptr, wrows, fwords, wrow_scale, dev, s);
        RealBinaryArgs gi{G, F, beta, nullptr, wrows, nullptr, N, F, K, fwords, dX, lddx,
                          nullptr};
        gi.clip = true;
        launch_real_binary_gemm(gi, dev, s);
    }
    float *csum = reinterpret_cast<float *>(ws + w.csum);
    weight_colsum_kernel<<<unsigned((F + 31) / 32), 32 * kColGroups, 0, s>>>(Wg, wbits, words, K,
                                                                            F, csum);
    const int64_t kfs = (int64_t(K) * F + kBwThreads - 1) / kBwThreads;
    grad_weight_kernel<<<unsigned(kfs < 4096 ? kfs : 4096), kBwThreads, 0, s>>>(
        Wg, wbits, words, beta, csum, Wt, ldw, K, F, dW, lddw);
    return launch_status();
}
