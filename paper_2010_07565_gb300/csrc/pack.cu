// Steps 1-3 of the Bi-GCN layer forward (Wang et al., CVPR 2021):
//   bigcn_pack_rows    -- centring (Sec. 6.2) + sign binarization of node
//                         features (Eq. 8) + per-node scale (Eq. 7)
//   bigcn_pack_weights -- sign binarization of weight columns (Eq. 3) +
//                         per-column scale (Eq. 4)
//
// pack_rows is HBM-bound: it reads 4K bytes per node and writes K/8 + 4.
// Lane l of a 32-feature chunk c owns feature 32c + l, so one __ballot_sync
// yields the chunk's 32-bit half-word of the packed row directly, and every
// lane keeps a running sum of |y|. G warps (1, 2, 4 or 8, so that the grid
// fills the GPU even when N is small) share a row, warp g taking chunks
// g, g + G, ...; each warp issues eight chunks' loads (1 KB) before it
// consumes any, and the grids are persistent (eight blocks per SM). The
// whole-row kernel has no block barrier and stays at full occupancy, which
// -- not a deeper unroll -- is what overlaps one warp's ballots with the
// other warps' loads. The G partial |y| sums are added in a fixed order through
// shared memory, so alpha does not depend on scheduling.
//
// pack_weights reads W (K x F) column-wise: thread (x, y) of a 32 x 8 block
// owns one column and builds whole 64-bit words from 64 coalesced row reads,
// all 64 in flight at once (the kernel is latency-bound: few blocks, so it
// is given registers rather than occupancy); one launch can pack two
// matrices (both layers' weights). The words of a column are spread over a cluster of S <= 8 blocks
// (grid y); each block reduces its |W| partial sums in shared memory, and
// block 0 of the cluster adds the S partials through distributed shared
// memory in rank order (deterministic).
#include <cooperative_groups.h>

#include "launch.cuh"
#include "pack_row.cuh"

namespace bigcn {
namespace {

namespace cg = cooperative_groups;

constexpr int kPackThreads = 256;
constexpr int kPackWarps = kPackThreads / 32;
constexpr int kPackBlocksPerSM = 8;   // resident blocks the persistent grids assume
constexpr int kPackUnroll = 8;

// Whole rows per warp: every warp walks rows on its own (persistent grid,
// no block barrier), which keeps the kernel small enough for full occupancy.
template <bool kAffine, bool kUpstream>
__global__ void __launch_bounds__(kPackThreads, kPackBlocksPerSM)
pack_rows_kernel(const float *__restrict__ X, int64_t N, int K, int64_t ldx,
                 const float *__restrict__ scale, const float *__restrict__ shift,
                 uint32_t *__restrict__ bits32, int64_t ld32, float *__restrict__ alpha) {
    if (kUpstream) grid_dependency_wait();      // X is the previous kernel's output
    constexpr Affine kA = kAffine ? Affine::kGlobalLate : Affine::kNone;
    const int lane = threadIdx.x & 31;
    const int64_t nwarps = int64_t(gridDim.x) * kPackWarps;
    for (int64_t row = int64_t(blockIdx.x) * kPackWarps + (threadIdx.x >> 5); row < N;
         row += nwarps) {
        const float l1 = pack_share<1, kPackUnroll, kA>(X + row * ldx, K, scale, shift, nullptr,
                                                        bits32 + row * ld32, ld32, 0);
        if (lane == 0) alpha[row] = l1 / float(K);
    }
    // Otherwise wait only now: finishing after the predecessor keeps the
    // chain's completion order for the kernels that follow.
    if (!kUpstream) grid_dependency_wait();
}

// Rows shared by G > 1 warps (few, long rows): block b takes row groups
// b, b + gridDim.x, ...; the G partial sums meet in shared memory.
template <int G, bool kAffine>
__global__ void __launch_bounds__(kPackThreads, 5)
pack_rows_split_kernel(const float *__restrict__ X, int64_t N, int K, int64_t ldx,
                       const float *__restrict__ scale, const float *__restrict__ shift,
                       uint32_t *__restrict__ bits32, int64_t ld32, float *__restrict__ alpha,
                       bool x_upstream) {
    __shared__ float part[kPackWarps];
    if (x_upstream) grid_dependency_wait();
    constexpr Affine kA = kAffine ? Affine::kGlobal : Affine::kNone;
    constexpr int kRows = kPackWarps / G;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int sub = warp % G;
    for (int64_t group = blockIdx.x; group * kRows < N; group += gridDim.x) {
        const int64_t row = group * kRows + warp / G;
        const float l1 = (row < N) ? pack_share<G, kPackUnroll, kA>(X + row * ldx, K, scale, shift,
                                                                    nullptr, bits32 + row * ld32,
                                                                    ld32, sub)
                                   : 0.0f;
        if (lane == 0) part[warp] = l1;
        __syncthreads();
        if (row < N && sub == 0 && lane == 0) {
            float s = 0.0f;
            for (int g = 0; g < G; ++g) s += part[warp + g];
            alpha[row] = s / float(K);
        }
        __syncthreads();   // part[] is rewritten by the next group
    }
    if (!x_upstream) grid_dependency_wait();
}

constexpr int kWCols = 32;
constexpr int kWRows = 8;
constexpr int kMaxCluster = 8;

// Blocks with blockIdx.x < a.tiles pack matrix a, the rest matrix b (one
// launch can pack both layers' weights); each block owns 32 columns.
__global__ void __launch_bounds__(kWCols *kWRows, 2)
pack_weights_kernel(WeightPack a, WeightPack b) {
    __shared__ float partial[kWRows][kWCols];
    __shared__ float colsum[kWCols];
    allow_dependent_launch();   // what follows may start on the call's own inputs
    grid_dependency_wait();
    cg::cluster_group cluster = cg::this_cluster();
    const int S = int(cluster.num_blocks());
    const int rank = int(cluster.block_rank());
    const bool first = int(blockIdx.x) < a.tiles;
    const WeightPack &m = first ? a : b;
    const int tile = first ? int(blockIdx.x) : int(blockIdx.x) - a.tiles;
    const int tx = threadIdx.x, ty = threadIdx.y;
    const int j = tile * kWCols + tx;
    const int K = m.K;

    float l1 = 0.0f;
    if (j < m.F) {
        for (int w = rank * kWRows + ty; w < m.words; w += S * kWRows) {
            const int kb = w * 64;
            float v[64];
#pragma unroll
            for (int q = 0; q < 64; ++q)
                v[q] = (kb + q < K) ? __ldg(m.W + int64_t(kb + q) * m.ldw + j) : 0.0f;
            uint64_t word = 0;
#pragma unroll
            for (int q = 0; q < 64; ++q) {
                const bool in = kb + q < K;
                word |= uint64_t(in && v[q] >= 0.0f) << q;
                l1 += fabsf(v[q]);
            }
            m.bits[int64_t(j) * m.words + w] = word;
        }
    }
    partial[ty][tx] = l1;
    __syncthreads();
    if (ty == 0) {
        float s = 0.0f;
#pragma unroll
        for (int r = 0; r < kWRows; ++r) s += partial[r][tx];
        colsum[tx] = s;
    }
    cluster.sync();
    if (rank == 0 && ty == 0 && j < m.F) {
        float s = 0.0f;
        for (int r = 0; r < S; ++r) s += cluster.map_shared_rank(colsum, r)[tx];
        m.beta[j] = s / float(K);
    }
    cluster.sync();   // peers keep their shared memory until block 0 has read it
}

}  // namespace

void launch_pack_rows(const float *X, int64_t N, int K, int64_t ldx, const float *scale,
                      const float *shift, uint64_t *bits, int words, float *alpha,
                      const DeviceInfo &dev, cudaStream_t stream, bool pdl, bool x_upstream) {
    if (N == 0) return;
    // Split rows over up to 8 warps while the grid is short of one full wave
    // of warps, as long as every warp keeps at least one 8-chunk batch.
    const int nchunks = (K + 31) / 32;
    const int64_t full_wave = int64_t(dev.sm_count) * 64;
    int G = 1;
    while (G < kPackWarps && N * G < full_wave && nchunks >= 2 * G * 8) G *= 2;
    const int rows_per_block = kPackWarps / G;
    const int64_t groups = (N + rows_per_block - 1) / rows_per_block;
    const int64_t resident = int64_t(dev.sm_count) * kPackBlocksPerSM;
    const dim3 grid(unsigned(groups < resident ? groups : resident)), block(kPackThreads), one(1, 1, 1);
    uint32_t *b32 = reinterpret_cast<uint32_t *>(bits);
    const int64_t ld32 = int64_t(words) * 2;
    const float *no = nullptr;
    if (G == 1) {
        auto run = [&](auto kernel, const float *sc, const float *sh) {
            launch_kernel(kernel, grid, block, 0, stream, pdl, one, X, N, K, ldx, sc, sh, b32, ld32,
                          alpha);
        };
        if (scale && x_upstream) run(pack_rows_kernel<true, true>, scale, shift);
        else if (scale) run(pack_rows_kernel<true, false>, scale, shift);
        else if (x_upstream) run(pack_rows_kernel<false, true>, no, no);
        else run(pack_rows_kernel<false, false>, no, no);
    } else {
        auto run = [&](auto kernel, const float *sc, const float *sh) {
            launch_kernel(kernel, grid, block, 0, stream, pdl, one, X, N, K, ldx, sc, sh, b32, ld32,
                          alpha, x_upstream);
        };
        if (G == 2) {
            if (scale) run(pack_rows_split_kernel<2, true>, scale, shift);
            else run(pack_rows_split_kernel<2, false>, no, no);
        } else if (G == 4) {
            if (scale) run(pack_rows_split_kernel<4, true>, scale, shift);
            else run(pack_rows_split_kernel<4, false>, no, no);
        } else {
            if (scale) run(pack_rows_split_kernel<8, true>, scale, shift);
            else run(pack_rows_split_kernel<8, false>, no, no);
        }
    }
}

void launch_pack_weights2(const WeightPack &a, const WeightPack &b, cudaStream_t stream) {
    // One block row per 8 words of the longer matrix, at most a cluster of 8.
    auto rows = [](const WeightPack &m) { return (m.words + kWRows - 1) / kWRows; };
    WeightPack A = a, B = b;
    A.tiles = (a.F + kWCols - 1) / kWCols;
    B.tiles = (b.W != nullptr) ? (b.F + kWCols - 1) / kWCols : 0;
    int S = rows(A);
    if (B.tiles > 0 && rows(B) > S) S = rows(B);
    if (S > kMaxCluster) S = kMaxCluster;
    launch_kernel(pack_weights_kernel, dim3(A.tiles + B.tiles, S, 1), dim3(kWCols, kWRows, 1), 0,
                  stream, false, dim3(1, S, 1), A, B);
}

void launch_pack_weights(const float *Wt, int K, int F, int64_t ldw, uint64_t *bits,
                         int words, float *beta, cudaStream_t stream) {
    WeightPack a{Wt, K, F, ldw, bits, words, beta, 0};
    WeightPack none{nullptr, 1, 0, 0, nullptr, 0, nullptr, 0};
    launch_pack_weights2(a, none, stream);
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
