// The Bi-GCN layer over a weighted adjacency. The paper's notation (Sec. 3)
// takes A = [a_ij] with general entries, d_i = sum_j a_ij, A^ = A + I and
// D^_ii = sum_j a^_ij, and Eq. 1's operator D^-1/2 A^ D^-1/2 on it; the 0/1
// graphs of the other entry points are the case a_ij = 1. Here the CSR
// carries one fp32 weight per entry (finite and non-negative).
//
//   bigcn_weighted_dinv        dinv_i = 1/sqrt(1 + sum of row i's weights)
//   bigcn_spmm_norm_weighted   H_i = dinv_i (dinv_i Z_i + sum_e a_ij dinv_j Z_j)
//   bigcn_weighted_layer_forward
//       pack_rows -> pack_weights -> the degree pass (which also forms the
//       row scale s_j = alpha_j dinv_j) -> the XNOR product with s as its row
//       scale (dots kept factored when K <= 32767) -> the aggregation, which
//       weights neighbour j by a_ij s_j and multiplies the sum by dinv_i.
//
// The degrees need a pass of their own: unlike 1 + row length, a weighted
// degree is a sum over the row, and every row's is read by its neighbours.
#include "launch.cuh"

using namespace bigcn;

namespace {

constexpr int kDegThreads = 256;
constexpr int kDegWarps = kDegThreads / 32;
// Rows longer than this are summed by the whole block instead of one warp.
constexpr int64_t kDegHeavy = 2048;

// Kahan's compensated sum (a running sum and the low-order part its last
// addition lost): a row of tens of thousands of weights is summed with an
// error of a few ulps instead of one growing with its length.
struct Compensated {
    float sum = 0.0f, lost = 0.0f;
    __device__ __forceinline__ void add(float v) {
        const float y = v - lost;
        const float t = sum + y;
        lost = (t - sum) - y;
        sum = t;
    }
    __device__ __forceinline__ float value() const { return sum - lost; }
};

// Sum of values[q] for q = q0, q0 + stride, ... below q1, four loads in flight.
__device__ __forceinline__ float strided_sum(const float *__restrict__ values, int64_t q0,
                                             int64_t q1, int stride) {
    Compensated c;
    for (int64_t q = q0; q < q1; q += 4 * int64_t(stride)) {
        float v[4];
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const int64_t qk = q + int64_t(k) * stride;
            v[k] = qk < q1 ? __ldg(values + qk) : 0.0f;
        }
#pragma unroll
        for (int k = 0; k < 4; ++k) c.add(v[k]);
    }
    return c.value();
}

// Block b owns rows 8b .. 8b + 7. Every warp reads the same eight row
// lengths, so the choice between the two paths is uniform over the block:
// rows of at most kDegHeavy entries are summed by their own warp, longer
// ones by all eight warps in turn (partials added in warp order).
__global__ void __launch_bounds__(kDegThreads)
weighted_dinv_kernel(const int64_t *__restrict__ rowptr, const float *__restrict__ values,
                     int64_t N, int64_t nnz, const float *__restrict__ alpha,
                     float *__restrict__ dinv, float *__restrict__ s) {
    __shared__ float part[kDegWarps];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t i0 = int64_t(blockIdx.x) * kDegWarps;
    // Row bounds of the block's rows, clamped to [0, nnz] (a malformed CSR
    // gives wrong degrees, never an out-of-range read).
    int64_t bound = 0;
    if (lane <= kDegWarps) bound = __ldg(rowptr + min(i0 + lane, N));
    bound = min(max(bound, int64_t(0)), nnz);
    float total = 0.0f;     // this warp's row (lane 0)
    for (int r = 0; r < kDegWarps; ++r) {
        const int64_t b = __shfl_sync(kFullMask, bound, r);
        const int64_t e = max(__shfl_sync(kFullMask, bound, r + 1), b);
        if (i0 + r >= N) break;
        if (e - b <= kDegHeavy) {
            if (r == warp) total = warp_sum(strided_sum(values, b + lane, e, 32));
        } else {
            const float v = warp_sum(strided_sum(values, b + threadIdx.x, e, kDegThreads));
            if (lane == 0) part[warp] = v;
            __syncthreads();
            if (r == warp) {
                float t = 0.0f;
                for (int w = 0; w < kDegWarps; ++w) t += part[w];
                total = t;
            }
            __syncthreads();    // part[] is rewritten by the next heavy row
        }
    }
    grid_dependency_wait();     // alpha is the row packing's output
    const int64_t i = i0 + warp;
    if (lane == 0 && i < N) {
        const float r = 1.0f / sqrtf(1.0f + total);
        dinv[i] = r;
        if (s != nullptr) s[i] = __ldg(alpha + i) * r;
    }
}

constexpr size_t kWAlign = 256;
size_t wround(size_t x) { return (x + kWAlign - 1) / kWAlign * kWAlign; }
constexpr int32_t kMaxDots16K = 32767;

// Workspace: A bits, alpha, B bits, beta, Z (factored or fp32), row scale,
// the tensor-core product's FP8 weight tiles, dinv, s.
struct WeightedWorkspace {
    size_t a_bits, alpha, b_bits, beta, z, rowscale, bexp, bexp_bytes, dinv, s, total;
    bool compressed;
    int64_t ldz;
};

bool weighted_workspace(int64_t N, int32_t K, int32_t F, WeightedWorkspace *w) {
    if (N < 0 || K < 1 || F < 1) return false;
    const int64_t words = bigcn_words(K);
    w->compressed = K <= kMaxDots16K;
    w->ldz = w->compressed ? (int64_t(F) + 7) / 8 * 8 : F;
    if (N > kMaxElems / (words > w->ldz ? words : w->ldz)) return false;
    size_t off = 0;
    w->a_bits = off;   off = wround(off + size_t(N) * size_t(words) * 8);
    w->alpha = off;    off = wround(off + size_t(N) * 4);
    w->b_bits = off;   off = wround(off + size_t(F) * size_t(words) * 8);
    w->beta = off;     off = wround(off + size_t(F) * 4);
    w->z = off;        off = wround(off + size_t(N) * size_t(w->ldz) * (w->compressed ? 2 : 4));
    w->rowscale = off; if (w->compressed) off = wround(off + size_t(N) * 4);
    w->bexp = off;
    w->bexp_bytes = xnor_gemm_tc_bexp_bytes(K, F);
    off = wround(off + w->bexp_bytes);
    w->dinv = off;     off = wround(off + size_t(N) * 4);
    w->s = off;        off = wround(off + size_t(N) * 4);
    w->total = off;
    return true;
}

}  // namespace

namespace bigcn {
void launch_weighted_dinv(const int64_t *rowptr, const float *values, int64_t N, int64_t nnz,
                          const float *alpha, float *dinv, float *s, cudaStream_t stream) {
    if (N == 0) return;
    const dim3 grid(unsigned((N + kDegWarps - 1) / kDegWarps));
    launch_kernel(weighted_dinv_kernel, grid, dim3(kDegThreads), 0, stream, false, dim3(1, 1, 1),
                  rowptr, values, N, nnz, alpha, dinv, s);
}
}  // namespace bigcn

extern "C" bigcn_status bigcn_weighted_dinv(const int64_t *rowptr, const float *values,
                                            int64_t N, int64_t nnz, float *dinv, void *stream) {
    if (N < 0 || N > int64_t(INT32_MAX) || nnz < 0) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!rowptr || !dinv || (nnz > 0 && !values)) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(rowptr, 8) || (values && !aligned_to(values, 4)) || !aligned_to(dinv, 4))
        return BIGCN_ERR_MISALIGNED;
    if (overlaps(dinv, size_t(N) * 4, rowptr, size_t(N + 1) * 8) ||
        overlaps(dinv, size_t(N) * 4, values, size_t(nnz) * 4))
        return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    launch_weighted_dinv(rowptr, values, N, nnz, nullptr, dinv, nullptr, as_stream(stream));
    return launch_status();
}

extern "C" bigcn_status bigcn_spmm_norm_weighted(const int64_t *rowptr, const int32_t *colidx,
                                                 const float *values, const float *dinv,
                                                 int64_t N, int64_t nnz, const float *Z,
                                                 int64_t ldz, int32_t F, float *H, int64_t ldh,
                                                 void *stream) {
    if (N < 0 || N > int64_t(INT32_MAX) || nnz < 0 || F < 1 || ldz < F || ldh < F)
        return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldz || N > kMaxElems / ldh)) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!rowptr || !dinv || !Z || !H || (nnz > 0 && (!colidx || !values)))
        return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(rowptr, 8) || (colidx && !aligned_to(colidx, 4)) ||
        (values && !aligned_to(values, 4)) || !aligned_to(dinv, 4) || !aligned_to(Z, 4) ||
        !aligned_to(H, 4))
        return BIGCN_ERR_MISALIGNED;
    const size_t hb = span_bytes(N, F, ldh, 4);
    if (overlaps(H, hb, Z, span_bytes(N, F, ldz, 4)) ||
        overlaps(H, hb, rowptr, size_t(N + 1) * 8) || overlaps(H, hb, colidx, size_t(nnz) * 4) ||
        overlaps(H, hb, values, size_t(nnz) * 4) || overlaps(H, hb, dinv, size_t(N) * 4))
        return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    SpmmArgs a{rowptr, colidx, N, nnz, Z, ldz, F, H, ldh, false, false};
    a.agg = kAggWeighted;
    a.values = values;
    a.dinv = dinv;
    launch_spmm_norm(a, dev, as_stream(stream));
    return launch_status();
}

extern "C" size_t bigcn_weighted_layer_workspace_bytes(int64_t N, int32_t K, int32_t F) {
    WeightedWorkspace w;
    return weighted_workspace(N, K, F, &w) ? w.total : 0;
}

extern "C" bigcn_status bigcn_weighted_layer_forward(
    const float *X, int64_t N, int32_t K, int64_t ldx, const float *scale, const float *shift,
    const float *Wt, int32_t F, int64_t ldw, const int64_t *rowptr, const int32_t *colidx,
    const float *values, int64_t nnz, void *workspace, size_t ws_bytes, float *H, int64_t ldh,
    void *stream) {
    WeightedWorkspace w;
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || ldx < K || ldw < F || ldh < F ||
        nnz < 0)
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (!weighted_workspace(N, K, F, &w)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / ldh)) return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!X || !Wt || !rowptr || !H || !workspace || (nnz > 0 && (!colidx || !values)))
        return BIGCN_ERR_INVALID_ARG;
    if (ws_bytes < w.total) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(Wt, 4) || !aligned_to(rowptr, 8) ||
        (colidx && !aligned_to(colidx, 4)) || (values && !aligned_to(values, 4)) ||
        !aligned_to(H, 4) || !aligned_to(workspace, kWAlign) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t hb = span_bytes(N, F, ldh, 4);
    const void *inputs[] = {X, Wt, rowptr, colidx, values, scale, shift};
    const size_t in_bytes[] = {span_bytes(N, K, ldx, 4), span_bytes(K, F, ldw, 4),
                               size_t(N + 1) * 8, size_t(nnz) * 4, size_t(nnz) * 4,
                               size_t(K) * 4, size_t(K) * 4};
    for (int q = 0; q < 7; ++q) {
        if (overlaps(workspace, w.total, inputs[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
        if (overlaps(H, hb, inputs[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
    }
    if (overlaps(H, hb, workspace, w.total)) return BIGCN_ERR_INVALID_ARG;

    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    char *ws = static_cast<char *>(workspace);
    uint64_t *a_bits = reinterpret_cast<uint64_t *>(ws + w.a_bits);
    float *alpha = reinterpret_cast<float *>(ws + w.alpha);
    uint64_t *b_bits = reinterpret_cast<uint64_t *>(ws + w.b_bits);
    float *beta = reinterpret_cast<float *>(ws + w.beta);
    float *dinv = reinterpret_cast<float *>(ws + w.dinv);
    float *srow = reinterpret_cast<float *>(ws + w.s);
    const int words = bigcn_words(K);
    cudaStream_t s = as_stream(stream);

    launch_pack_rows(X, N, K, ldx, scale, shift, a_bits, words, alpha, dev, s);
    launch_pack_weights(Wt, K, F, ldw, b_bits, words, beta, s);
    // Factored rows carry dinv_j in their row scale (s_j = alpha_j dinv_j);
    // fp32 rows are the plain product and the aggregation reads dinv_j.
    launch_weighted_dinv(rowptr, values, N, nnz, alpha, dinv, w.compressed ? srow : nullptr, s);
    GemmArgs g{a_bits, w.compressed ? srow : alpha, N, b_bits, beta, F, K, words, nullptr,
               w.ldz, nullptr, nullptr};
    if (w.bexp_bytes > 0) g.b_e4m3 = reinterpret_cast<uint8_t *>(ws + w.bexp);
    SpmmArgs a{rowptr, colidx, N, nnz, nullptr, w.ldz, F, H, ldh, false, false};
    a.agg = kAggWeighted;
    a.values = values;
    a.dinv = dinv;
    if (w.compressed) {
        uint16_t *D16 = reinterpret_cast<uint16_t *>(ws + w.z);
        float *rowscale = reinterpret_cast<float *>(ws + w.rowscale);
        g.dots16 = D16;
        g.ldd16 = w.ldz;
        g.rowscale = rowscale;
        a.D16 = D16;
        a.rowscale = rowscale;
        a.colscale = beta;
    } else {
        float *Z = reinterpret_cast<float *>(ws + w.z);
        g.Z = Z;
        a.Z = Z;
    }
    launch_xnor_gemm(g, dev, s);
    launch_spmm_norm(a, dev, s);
    return launch_status();
}
