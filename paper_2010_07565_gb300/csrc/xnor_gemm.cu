// Step 4 of the Bi-GCN layer forward (Wang et al., CVPR 2021, Eqs. 11-12):
// the +-1 inner products of packed node rows with packed weight columns,
//   dot[i,j] = K - 2 popcount(a_i XOR b_j),  Z[i,j] = alpha_i beta_j dot[i,j].
//
// Products with K >= 128, F >= 32 and at least one 128-row tile per SM run on
// the tensor cores (xnor_gemm_tc.cu); the CUDA-core path below takes the rest.
//
// CUDA-core path: a 128 x (16*TN) output tile per 256-thread block, the two
// packed operand tiles staged in shared memory 8 words (512 signs) at a time
// with register double buffering; each thread accumulates TM x TN mismatch
// counts with XOR + POPC. Thread (tx, ty) owns rows ty + 16 i and columns
// tx + 16 j, which keeps the shared-memory reads free of bank conflicts (odd
// row pitch) and the Z stores coalesced along the columns.
//
// When the output has fewer tiles than the GPU has SMs, the k-steps of each
// tile are split over a thread-block cluster of S <= 8 blocks (grid z): each
// block counts mismatches over every S-th k-step, stores its counts in shared
// memory, and after a cluster barrier each block finishes 1/S of the tile's
// rows by adding the S partial counts through distributed shared memory. The
// counts are integers, so the split changes no bit of the result.
//
// The epilogue optionally multiplies row i by dinv_i = 1/sqrt(1 + deg_i), the
// source-side factor of D^-1/2 (A + I) D^-1/2, so that the aggregation that
// follows in the fused layer reads pre-scaled rows.
#include <cooperative_groups.h>

#include "launch.cuh"

namespace bigcn {
namespace {

constexpr int kBM = 128;     // rows per block tile
constexpr int kBKW = 8;      // 64-bit words per k-step
constexpr int kPitch = kBKW + 1;
constexpr int kTM = 8;       // rows per thread
constexpr int kThreads = 256;

namespace cg = cooperative_groups;

template <int TN, bool kDegreeScale, bool kSplit>
__global__ void __launch_bounds__(kThreads)
xnor_gemm_popc_kernel(const uint64_t *__restrict__ A, const float *__restrict__ alpha, int64_t N,
                      const uint64_t *__restrict__ B, const float *__restrict__ beta, int F,
                      int K, int words, float *__restrict__ Z, int64_t ldz,
                      int32_t *__restrict__ dots, const int64_t *__restrict__ rowptr,
                      uint16_t *__restrict__ dots16, int64_t ldd16, float *__restrict__ rowscale,
                      bool f16) {
    constexpr int BN = 16 * TN;
    constexpr int kALoads = kBM * kBKW / kThreads;                         // 4
    constexpr int kBLoads = (BN * kBKW + kThreads - 1) / kThreads;          // 1..2
    __shared__ uint64_t As[kBM][kPitch];
    __shared__ uint64_t Bs[BN][kPitch];

    grid_dependency_wait();     // the packed operands come from earlier kernels
    const int tid = threadIdx.x;
    const int tx = tid & 15, ty = tid >> 4;
    const int64_t m0 = int64_t(blockIdx.x) * kBM;
    const int n0 = blockIdx.y * BN;
    const int S = kSplit ? int(gridDim.z) : 1;
    const int rank = kSplit ? int(blockIdx.z) : 0;

    uint64_t ra[kALoads], rb[kBLoads];
    auto load_tile = [&](int k0) {
#pragma unroll
        for (int q = 0; q < kALoads; ++q) {
            const int e = tid + q * kThreads;
            const int r = e / kBKW, kw = e % kBKW;
            const int64_t row = m0 + r;
            ra[q] = (row < N && k0 + kw < words) ? __ldg(A + row * words + k0 + kw) : 0ull;
        }
#pragma unroll
        for (int q = 0; q < kBLoads; ++q) {
            const int e = tid + q * kThreads;
            const int c = e / kBKW, kw = e % kBKW;
            rb[q] = (e < BN * kBKW && n0 + c < F && k0 + kw < words)
                        ? __ldg(B + int64_t(n0 + c) * words + k0 + kw) : 0ull;
        }
    };
    auto store_tile = [&]() {
#pragma unroll
        for (int q = 0; q < kALoads; ++q) {
            const int e = tid + q * kThreads;
            As[e / kBKW][e % kBKW] = ra[q];
        }
#pragma unroll
        for (int q = 0; q < kBLoads; ++q) {
            const int e = tid + q * kThreads;
            if (e < BN * kBKW) Bs[e / kBKW][e % kBKW] = rb[q];
        }
    };

    int mism[kTM][TN];
#pragma unroll
    for (int i = 0; i < kTM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) mism[i][j] = 0;

    load_tile(rank * kBKW);
    for (int k0 = rank * kBKW; k0 < words; k0 += S * kBKW) {
        __syncthreads();
        store_tile();
        __syncthreads();
        if (k0 + S * kBKW < words) load_tile(k0 + S * kBKW);
#pragma unroll
        for (int kw = 0; kw < kBKW; ++kw) {
            uint64_t a[kTM], b[TN];
#pragma unroll
            for (int i = 0; i < kTM; ++i) a[i] = As[ty + 16 * i][kw];
#pragma unroll
            for (int j = 0; j < TN; ++j) b[j] = Bs[tx + 16 * j][kw];
#pragma unroll
            for (int i = 0; i < kTM; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) mism[i][j] += __popcll(a[i] ^ b[j]);
        }
    }

    if constexpr (kSplit) {
        __shared__ int red[kBM * BN];
        cg::cluster_group cluster = cg::this_cluster();
#pragma unroll
        for (int i = 0; i < kTM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) red[(ty + 16 * i) * BN + tx + 16 * j] = mism[i][j];
        cluster.sync();
#pragma unroll
        for (int i = 0; i < kTM; ++i) {
            if (i % S != rank) continue;
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                int total = 0;
                for (int r = 0; r < S; ++r)
                    total += cluster.map_shared_rank(red, r)[(ty + 16 * i) * BN + tx + 16 * j];
                mism[i][j] = total;
            }
        }
        cluster.sync();   // peers keep their counts until every block has read them
    }

#pragma unroll
    for (int i = 0; i < kTM; ++i) {
        if (kSplit && i % S != rank) continue;
        const int64_t row = m0 + ty + 16 * i;
        if (row >= N) continue;
        float ai = __ldg(alpha + row);
        if (kDegreeScale) ai *= inv_sqrt_degree(__ldg(rowptr + row + 1) - __ldg(rowptr + row));
        if (dots16 != nullptr) {            // compressed output: biased dots + row scale
            if (n0 == 0 && tx == 0) rowscale[row] = ai;
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                const int col = n0 + tx + 16 * j;
                if (col < ldd16) dots16[row * ldd16 + col] = encode_dot(K - 2 * mism[i][j], col < F, f16);
            }
            continue;
        }
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int col = n0 + tx + 16 * j;
            if (col >= F) continue;
            const int d = K - 2 * mism[i][j];
            if (kDegreeScale)
                Z[row * ldz + col] = ai * (__ldg(beta + col) * float(d));
            else
                Z[row * ldz + col] = (ai * __ldg(beta + col)) * float(d);
            if (dots != nullptr) dots[row * F + col] = d;
        }
    }
}

template <int TN, bool kDeg>
void launch_tn(const GemmArgs &g, const DeviceInfo &dev, cudaStream_t s, bool pdl) {
    constexpr int BN = 16 * TN;
    const unsigned gx = unsigned((g.N + kBM - 1) / kBM), gy = unsigned((g.F + BN - 1) / BN);
    const int ksteps = (g.words + kBKW - 1) / kBKW;
    const int64_t tiles = int64_t(gx) * gy;
    int S = 1;
    if (tiles < dev.sm_count && ksteps > 1) {
        const int64_t want = (2 * int64_t(dev.sm_count) + tiles - 1) / tiles;
        S = int(want < 8 ? want : 8);
        if (S > ksteps) S = ksteps;
    }
    if (S == 1) {
        launch_kernel(xnor_gemm_popc_kernel<TN, kDeg, false>, dim3(gx, gy), dim3(kThreads), 0, s,
                      pdl, dim3(1, 1, 1), g.A, g.alpha, g.N, g.B, g.beta, g.F, g.K, g.words, g.Z,
                      g.ldz, g.dots, g.rowptr, g.dots16, g.ldd16, g.rowscale, g.dots_f16);
        return;
    }
    launch_kernel(xnor_gemm_popc_kernel<TN, kDeg, true>, dim3(gx, gy, S), dim3(kThreads), 0, s,
                  pdl, dim3(1, 1, S), g.A, g.alpha, g.N, g.B, g.beta, g.F, g.K, g.words, g.Z,
                  g.ldz, g.dots, g.rowptr, g.dots16, g.ldd16, g.rowscale, g.dots_f16);
}

template <bool kDeg>
void launch_deg(const GemmArgs &g, const DeviceInfo &dev, cudaStream_t s, bool pdl) {
    if (g.F > 32) launch_tn<4, kDeg>(g, dev, s, pdl);
    else if (g.F > 16) launch_tn<2, kDeg>(g, dev, s, pdl);
    else launch_tn<1, kDeg>(g, dev, s, pdl);
}

}  // namespace

void launch_xnor_gemm(const GemmArgs &g, const DeviceInfo &dev, cudaStream_t stream, bool pdl) {
    if (g.N == 0) return;
    if (xnor_gemm_tc_supported(g.N, g.K, g.F, dev)) {
        launch_xnor_gemm_tc(g, dev, stream, pdl);
        return;
    }
    if (g.rowptr != nullptr) launch_deg<true>(g, dev, stream, pdl);
    else launch_deg<false>(g, dev, stream, pdl);
}

}  // namespace bigcn

using namespace bigcn;

namespace {
bigcn_status check_gemm(const uint64_t *a_bits, const float *alpha, int64_t N,
                        const uint64_t *b_bits, const float *beta, int32_t F, int32_t K,
                        int32_t words, const float *Z, int64_t ldz, const int32_t *dots,
                        const int64_t *rowptr, bool need_rowptr) {
    if (N < 0 || F < 1 || K < 1 || words < bigcn_words(K) || ldz < F) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldz || N > kMaxElems / words)) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!a_bits || !alpha || !b_bits || !beta || !Z || (need_rowptr && !rowptr))
        return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(a_bits, 8) || !aligned_to(b_bits, 8) || !aligned_to(alpha, 4) ||
        !aligned_to(beta, 4) || !aligned_to(Z, 4) || (dots && !aligned_to(dots, 4)) ||
        (rowptr && !aligned_to(rowptr, 8)))
        return BIGCN_ERR_MISALIGNED;
    const size_t zb = span_bytes(N, F, ldz, 4);
    const size_t ab = size_t(N) * words * 8, bb = size_t(F) * words * 8;
    if (overlaps(Z, zb, a_bits, ab) || overlaps(Z, zb, b_bits, bb) ||
        overlaps(Z, zb, alpha, size_t(N) * 4) || overlaps(Z, zb, beta, size_t(F) * 4) ||
        overlaps(Z, zb, rowptr, size_t(N + 1) * 8))
        return BIGCN_ERR_INVALID_ARG;
    if (dots) {
        const size_t db = size_t(N) * F * 4;
        if (overlaps(dots, db, Z, zb) || overlaps(dots, db, a_bits, ab) ||
            overlaps(dots, db, b_bits, bb) || overlaps(dots, db, alpha, size_t(N) * 4) ||
            overlaps(dots, db, beta, size_t(F) * 4))
            return BIGCN_ERR_INVALID_ARG;
    }
    return BIGCN_OK;
}
}  // namespace

extern "C" bigcn_status bigcn_xnor_gemm(const uint64_t *a_bits, const float *alpha, int64_t N,
                                        const uint64_t *b_bits, const float *beta, int32_t F,
                                        int32_t K, int32_t words, float *Z, int64_t ldz,
                                        int32_t *dots, void *stream) {
    bigcn_status st = check_gemm(a_bits, alpha, N, b_bits, beta, F, K, words, Z, ldz, dots,
                                 nullptr, false);
    if (st != BIGCN_OK || N == 0) return st;
    DeviceInfo dev;
    if ((st = current_device(&dev)) != BIGCN_OK) return st;
    GemmArgs g{a_bits, alpha, N, b_bits, beta, F, K, words, Z, ldz, dots, nullptr};
    launch_xnor_gemm(g, dev, as_stream(stream));
    return launch_status();
}

extern "C" bigcn_status bigcn_xnor_gemm_degscaled(const uint64_t *a_bits, const float *alpha,
                                                  int64_t N, const uint64_t *b_bits,
                                                  const float *beta, int32_t F, int32_t K,
                                                  int32_t words, const int64_t *rowptr,
                                                  float *Z, int64_t ldz, void *stream) {
    bigcn_status st = check_gemm(a_bits, alpha, N, b_bits, beta, F, K, words, Z, ldz, nullptr,
                                 rowptr, true);
    if (st != BIGCN_OK || N == 0) return st;
    DeviceInfo dev;
    if ((st = current_device(&dev)) != BIGCN_OK) return st;
    GemmArgs g{a_bits, alpha, N, b_bits, beta, F, K, words, Z, ldz, nullptr, rowptr};
    launch_xnor_gemm(g, dev, as_stream(stream));
    return launch_status();
}
