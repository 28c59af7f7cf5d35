// Steps 1-3 of the Bi-GCN layer forward (Wang et al., CVPR 2021):
//   bigcn_pack_rows    -- centring (Sec. 6.2) + sign binarization of node
//                         features (Eq. 8) + per-node scale (Eq. 7)
//   bigcn_pack_weights -- sign binarization of weight columns (Eq. 3) +
//                         per-column scale (Eq. 4)
//
// pack_rows is HBM-bound: it reads 4K bytes per node and writes K/8 + 4.
// One warp walks one row at a time (persistent grid, a multiple of the SM
// count): lane l of chunk c owns feature 32c + l, so one __ballot_sync gives
// the 32-bit half-word of the packed row directly, and each lane keeps a
// running sum of |y| that one warp reduction turns into the scale. Eight
// chunks' loads are issued before any is consumed to keep 1 KB per warp in
// flight.
#include "launch.cuh"

namespace bigcn {
namespace {

constexpr int kPackThreads = 256;
constexpr int kPackUnroll = 8;

template <bool kAffine>
__global__ void __launch_bounds__(kPackThreads, 6)
pack_rows_kernel(const float *__restrict__ X, int64_t N, int K, int64_t ldx,
                 const float *__restrict__ scale, const float *__restrict__ shift,
                 uint32_t *__restrict__ bits32, int64_t ld32, float *__restrict__ alpha) {
    const int lane = threadIdx.x & 31;
    const int64_t warp0 = (int64_t(blockIdx.x) * kPackThreads + threadIdx.x) >> 5;
    const int64_t nwarps = (int64_t(gridDim.x) * kPackThreads) >> 5;
    const int nchunks = (K + 31) >> 5;          // 32-bit words that carry signs
    const float kf = float(K);

    for (int64_t row = warp0; row < N; row += nwarps) {
        const float *x = X + row * ldx;
        uint32_t *out = bits32 + row * ld32;
        float l1 = 0.0f;
        for (int c0 = 0; c0 < nchunks; c0 += kPackUnroll) {
            float v[kPackUnroll];
#pragma unroll
            for (int u = 0; u < kPackUnroll; ++u) {
                const int k = (c0 + u) * 32 + lane;
                v[u] = (k < K) ? __ldcs(x + k) : 0.0f;
            }
#pragma unroll
            for (int u = 0; u < kPackUnroll; ++u) {
                const int k = (c0 + u) * 32 + lane;
                const bool in = k < K;
                float y = v[u];
                if (kAffine && in) y = __fmaf_rn(y, __ldg(scale + k), __ldg(shift + k));
                const unsigned m = __ballot_sync(kFullMask, in && y >= 0.0f);
                if (c0 + u < nchunks && lane == 0) out[c0 + u] = m;
                l1 += in ? fabsf(y) : 0.0f;
            }
        }
        // Pad half-words past the last one that carries signs are zero.
        for (int64_t q = nchunks + lane; q < ld32; q += 32) out[q] = 0u;
        l1 = warp_sum(l1);
        if (lane == 0) alpha[row] = l1 / kf;
    }
}

// Weight columns: thread (x, y) of a 32 x 8 block owns column j = 32*bx + x
// and the packed words w = y, y + 8, ...; reads of one k are coalesced across
// the 32 columns. The per-column |W| sums are reduced over y in shared memory.
constexpr int kWCols = 32;
constexpr int kWRows = 8;

__global__ void __launch_bounds__(kWCols *kWRows)
pack_weights_kernel(const float *__restrict__ Wt, int K, int F, int64_t ldw,
                    uint64_t *__restrict__ bits, int words, float *__restrict__ beta) {
    __shared__ float partial[kWRows][kWCols];
    const int tx = threadIdx.x, ty = threadIdx.y;
    const int j = blockIdx.x * kWCols + tx;
    float l1 = 0.0f;
    if (j < F) {
        for (int w = ty; w < words; w += kWRows) {
            uint64_t word = 0;
            const int kb = w * 64;
#pragma unroll 16
            for (int b = 0; b < 64; ++b) {
                const int k = kb + b;
                if (k < K) {
                    const float v = __ldg(Wt + int64_t(k) * ldw + j);
                    word |= uint64_t(v >= 0.0f) << b;
                    l1 += fabsf(v);
                }
            }
            bits[int64_t(j) * words + w] = word;
        }
    }
    partial[ty][tx] = l1;
    __syncthreads();
    if (ty == 0 && j < F) {
        float s = 0.0f;
#pragma unroll
        for (int r = 0; r < kWRows; ++r) s += partial[r][tx];
        beta[j] = s / float(K);
    }
}

}  // namespace

void launch_pack_rows(const float *X, int64_t N, int K, int64_t ldx, const float *scale,
                      const float *shift, uint64_t *bits, int words, float *alpha,
                      const DeviceInfo &dev, cudaStream_t stream) {
    if (N == 0) return;
    const int64_t blocks_needed = (N * 32 + kPackThreads - 1) / kPackThreads;
    const int64_t resident = int64_t(dev.sm_count) * (2048 / kPackThreads);
    const int grid = int(blocks_needed < resident ? blocks_needed : resident);
    uint32_t *b32 = reinterpret_cast<uint32_t *>(bits);
    if (scale)
        pack_rows_kernel<true><<<grid, kPackThreads, 0, stream>>>(
            X, N, K, ldx, scale, shift, b32, int64_t(words) * 2, alpha);
    else
        pack_rows_kernel<false><<<grid, kPackThreads, 0, stream>>>(
            X, N, K, ldx, nullptr, nullptr, b32, int64_t(words) * 2, alpha);
}

void launch_pack_weights(const float *Wt, int K, int F, int64_t ldw, uint64_t *bits,
                         int words, float *beta, cudaStream_t stream) {
    dim3 block(kWCols, kWRows);
    dim3 grid((F + kWCols - 1) / kWCols);
    pack_weights_kernel<<<grid, block, 0, stream>>>(Wt, K, F, ldw, bits, words, beta);
}

}  // namespace bigcn

using namespace bigcn;

extern "C" bigcn_status bigcn_pack_rows(const float *X, int64_t N, int32_t K, int64_t ldx,
                                        const float *scale, const float *shift,
                                        uint64_t *bits, int32_t words, float *alpha,
                                        void *stream) {
    if (N < 0 || K < 1 || ldx < K || words < bigcn_words(K)) return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / words)) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (X == nullptr || bits == nullptr || alpha == nullptr) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(bits, 8) || !aligned_to(alpha, 4) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t xb = span_bytes(N, K, ldx, 4), bb = size_t(N) * words * 8;
    if (overlaps(bits, bb, X, xb) || overlaps(alpha, size_t(N) * 4, X, xb) ||
        overlaps(alpha, size_t(N) * 4, bits, bb))
        return BIGCN_ERR_INVALID_ARG;

    DeviceInfo dev;
    bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    launch_pack_rows(X, N, K, ldx, scale, shift, bits, words, alpha, dev, as_stream(stream));
    return launch_status();
}

extern "C" bigcn_status bigcn_pack_weights(const float *Wt, int32_t K, int32_t F, int64_t ldw,
                                           uint64_t *bits, int32_t words, float *beta,
                                           void *stream) {
    if (K < 1 || F < 1 || ldw < F || words < bigcn_words(K)) return BIGCN_ERR_INVALID_ARG;
    if (Wt == nullptr || bits == nullptr || beta == nullptr) return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(Wt, 4) || !aligned_to(bits, 8) || !aligned_to(beta, 4))
        return BIGCN_ERR_MISALIGNED;
    const size_t wb = span_bytes(K, F, ldw, 4), bb = size_t(F) * words * 8;
    if (overlaps(bits, bb, Wt, wb) || overlaps(beta, size_t(F) * 4, Wt, wb) ||
        overlaps(beta, size_t(F) * 4, bits, bb))
        return BIGCN_ERR_INVALID_ARG;

    DeviceInfo dev;
    bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    launch_pack_weights(Wt, K, F, ldw, bits, words, beta, as_stream(stream));
    return launch_status();
}
