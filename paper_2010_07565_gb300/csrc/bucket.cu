// Sub-row bucketing of the Bi-GCN product (Sec. 4.1: the rows of H and the
// columns of W split into buckets of B consecutive values, each bucket with
// its own scale):
//
//   alpha_ib = mean over bucket b of |y_ik|,  beta_jb = mean over b of |W_kj|,
//   Z_ij     = sum over b of alpha_ib beta_jb dot_b(i, j),
//   dot_b    = (signs in bucket b) - 2 popcount(a_i XOR b_j over b's words).
//
// B is a multiple of 64, so a bucket is a whole number of packed words and
// the packed signs are exactly those of Bi-GCN's layout; only the scales
// gain a bucket index (alpha: N x nb, beta: F x nb, nb = ceil(K / B)).
//
// Kernels:
// * pack_rows_bucketed_kernel: one warp per (row, bucket), lane l of chunk c
//   owns feature 32c + l; eight chunks of loads in flight; one ballot per
//   chunk gives half a word; the bucket's |y| summed per lane, then across
//   the warp.
// * pack_weights_bucketed_kernel: one block per (32 columns, bucket), the
//   bucket's words spread over eight row groups, each word's 64 entries read
//   down the column (coalesced across columns), beta added in group order.
// * xnor_gemm_bucket_kernel: the CUDA-core product of xnor_gemm.cu's shape
//   (128 x 16 TN tiles, 8-word k-steps staged in shared memory) whose integer
//   mismatch counts are folded into fp32 accumulators with the bucket's
//   alpha_ib beta_jb at each bucket end (and at each k-step end, so that a
//   k-step split over a cluster folds only what it counted); split partials
//   are fp32 and added in rank order through distributed shared memory.
#include <cooperative_groups.h>

#include "launch.cuh"

namespace bigcn {
namespace {

namespace cg = cooperative_groups;

constexpr int kPackWarps = 8;
constexpr int kUnroll = 8;       // chunks of 32 features in flight per warp

// One warp per (row, bucket) -- grid y is the bucket, grid x strides over
// rows: the bucket's 2 bw chunks of 32 features, eight
// chunks (with their centring) loaded before any is used; one ballot per
// chunk gives half a packed word; the bucket's |y| are summed per lane and
// reduced across the warp at the end.
__global__ void __launch_bounds__(32 * kPackWarps)
pack_rows_bucketed_kernel(const float *__restrict__ X, int64_t N, int K, int64_t ldx,
                          const float *__restrict__ scale, const float *__restrict__ shift,
                          int bw, uint64_t *__restrict__ bits, int words,
                          float *__restrict__ alpha, int nb) {
    grid_dependency_wait();
    const int lane = threadIdx.x & 31;
    const int64_t nwarps = int64_t(gridDim.x) * kPackWarps;
    const int nchunks = (K + 31) / 32;
    const int bchunks = 2 * bw;                      // chunks per bucket
    const int b = blockIdx.y;                        // this block's bucket
    for (int64_t row = int64_t(blockIdx.x) * kPackWarps + (threadIdx.x >> 5); row < N;
         row += nwarps) {
        const float *x = X + row * ldx;
        const int cb = b * bchunks, ce = min(nchunks, cb + bchunks);
        float part = 0.0f;           // this lane's |y| in the bucket
        uint32_t lo = 0;             // ballot of the word's even chunk
        for (int c0 = cb; c0 < ce; c0 += kUnroll) {
            float v[kUnroll], sc[kUnroll], sh[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int k = 32 * (c0 + u) + lane;
                const bool in = c0 + u < ce && k < K;
                v[u] = in ? __ldg(x + k) : 0.0f;
                sc[u] = (in && scale != nullptr) ? __ldg(scale + k) : 1.0f;
                sh[u] = (in && scale != nullptr) ? __ldg(shift + k) : 0.0f;
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int c = c0 + u;
                if (c >= ce) break;
                const bool in = 32 * c + lane < K;
                const float y = scale != nullptr ? __fmaf_rn(v[u], sc[u], sh[u]) : v[u];
                const uint32_t m = __ballot_sync(kFullMask, in && y >= 0.0f);
                if (in) part += fabsf(y);
                if ((c & 1) == 0) {
                    lo = m;
                    if (c == ce - 1 && lane == 0) bits[row * words + c / 2] = uint64_t(lo);
                } else if (lane == 0) {
                    bits[row * words + c / 2] = uint64_t(lo) | (uint64_t(m) << 32);
                }
            }
        }
        const int len = min(K, (b + 1) * 64 * bw) - b * 64 * bw;
        const float sum = warp_sum(part);
        if (lane == 0) {
            alpha[row * nb + b] = sum / float(len);
            if (b == nb - 1)                         // words past the row's chunks
                for (int w = (nchunks + 1) / 2; w < words; ++w) bits[row * words + w] = 0ull;
        }
    }
}

constexpr int kWGroups = 8;      // row groups of the weight-packing block

// One block per (32 columns, bucket): thread (c, g) packs words w0 + g,
// w0 + g + 8, ... of the bucket for column c (each word's 64 entries read
// down the column, coalesced across the 32 columns) and sums their |W|; the
// eight group sums of a column are added in group order.
__global__ void __launch_bounds__(32 * kWGroups)
pack_weights_bucketed_kernel(const float *__restrict__ Wt, int K, int F, int64_t ldw, int bw,
                             uint64_t *__restrict__ bits, int words, float *__restrict__ beta,
                             int nb) {
    __shared__ float part[kWGroups][32];
    const int c = threadIdx.x & 31, grp = threadIdx.x >> 5;
    const int j = blockIdx.x * 32 + c;
    const int b = blockIdx.y;
    const int w0 = b * bw, w1 = min((K + 63) / 64, (b + 1) * bw);
    float sum = 0.0f;
    if (j < F) {
        for (int w = w0 + grp; w < w1; w += kWGroups) {
            float v[64];
#pragma unroll
            for (int e = 0; e < 64; ++e) {
                const int k = 64 * w + e;
                v[e] = k < K ? __ldg(Wt + int64_t(k) * ldw + j) : 0.0f;
            }
            uint64_t word = 0ull;
#pragma unroll
            for (int e = 0; e < 64; ++e) {
                if (64 * w + e < K) {
                    if (v[e] >= 0.0f) word |= uint64_t(1) << e;
                    sum += fabsf(v[e]);
                }
            }
            bits[int64_t(j) * words + w] = word;
        }
    }
    part[grp][c] = sum;
    __syncthreads();
    if (grp == 0 && j < F) {
        float t = 0.0f;
        for (int g = 0; g < kWGroups; ++g) t += part[g][c];
        const int len = min(K, (b + 1) * 64 * bw) - b * 64 * bw;
        beta[int64_t(j) * nb + b] = t / float(len);
        if (b == nb - 1)                             // words past the last bucket
            for (int w = w1; w < words; ++w) bits[int64_t(j) * words + w] = 0ull;
    }
}

constexpr int kBM = 128;     // rows per block tile
constexpr int kBKW = 8;      // 64-bit words per k-step
constexpr int kPitch = kBKW + 1;
constexpr int kTM = 8;       // rows per thread
constexpr int kThreads = 256;

template <int TN, bool kDeg, bool kSplit>
__global__ void __launch_bounds__(kThreads)
xnor_gemm_bucket_kernel(const uint64_t *__restrict__ A, const float *__restrict__ alpha, int64_t N,
                        const uint64_t *__restrict__ Bb, const float *__restrict__ beta, int F,
                        int K, int words, int bw, int nb, float *__restrict__ Z, int64_t ldz,
                        const int64_t *__restrict__ rowptr) {
    constexpr int BN = 16 * TN;
    constexpr int kALoads = kBM * kBKW / kThreads;
    constexpr int kBLoads = (BN * kBKW + kThreads - 1) / kThreads;
    __shared__ uint64_t As[kBM][kPitch];
    __shared__ uint64_t Bs[BN][kPitch];

    grid_dependency_wait();
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
                        ? __ldg(Bb + int64_t(n0 + c) * words + k0 + kw) : 0ull;
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

    // Row / column indices of this thread's outputs, clamped for the scale loads.
    int64_t rows[kTM];
    int cols[TN];
#pragma unroll
    for (int i = 0; i < kTM; ++i) rows[i] = min(m0 + ty + 16 * i, N - 1);
#pragma unroll
    for (int j = 0; j < TN; ++j) cols[j] = min(n0 + tx + 16 * j, F - 1);

    int mism[kTM][TN];
    float acc[kTM][TN];
#pragma unroll
    for (int i = 0; i < kTM; ++i)
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            mism[i][j] = 0;
            acc[i][j] = 0.0f;
        }
    int pending = 0;             // signs counted since the last fold
    // acc += alpha_ib beta_jb (pending - 2 mism) for the bucket b of the
    // words just counted; the counts restart.
    auto fold = [&](int b) {
        float a[kTM], c[TN];
#pragma unroll
        for (int i = 0; i < kTM; ++i) a[i] = __ldg(alpha + rows[i] * nb + b);
#pragma unroll
        for (int j = 0; j < TN; ++j) c[j] = __ldg(beta + int64_t(cols[j]) * nb + b);
#pragma unroll
        for (int i = 0; i < kTM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                acc[i][j] = fmaf(a[i] * c[j], float(pending - 2 * mism[i][j]), acc[i][j]);
                mism[i][j] = 0;
            }
        pending = 0;
    };

    load_tile(rank * kBKW);
    for (int k0 = rank * kBKW; k0 < words; k0 += S * kBKW) {
        __syncthreads();
        store_tile();
        __syncthreads();
        if (k0 + S * kBKW < words) load_tile(k0 + S * kBKW);
#pragma unroll
        for (int kw = 0; kw < kBKW; ++kw) {
            const int w = k0 + kw;
            if (w >= words) break;
            uint64_t a[kTM], b[TN];
#pragma unroll
            for (int i = 0; i < kTM; ++i) a[i] = As[ty + 16 * i][kw];
#pragma unroll
            for (int j = 0; j < TN; ++j) b[j] = Bs[tx + 16 * j][kw];
#pragma unroll
            for (int i = 0; i < kTM; ++i)
#pragma unroll
                for (int j = 0; j < TN; ++j) mism[i][j] += __popcll(a[i] ^ b[j]);
            pending += max(0, min(64, K - 64 * w));
            if ((w + 1) % bw == 0 || kw == kBKW - 1 || w + 1 == words) fold(w / bw);
        }
    }

    if constexpr (kSplit) {
        __shared__ float red[kBM * BN];
        cg::cluster_group cluster = cg::this_cluster();
#pragma unroll
        for (int i = 0; i < kTM; ++i)
#pragma unroll
            for (int j = 0; j < TN; ++j) red[(ty + 16 * i) * BN + tx + 16 * j] = acc[i][j];
        cluster.sync();
#pragma unroll
        for (int i = 0; i < kTM; ++i) {
            if (i % S != rank) continue;
#pragma unroll
            for (int j = 0; j < TN; ++j) {
                float total = 0.0f;
                for (int r = 0; r < S; ++r)
                    total += cluster.map_shared_rank(red, r)[(ty + 16 * i) * BN + tx + 16 * j];
                acc[i][j] = total;
            }
        }
        cluster.sync();   // peers keep their partials until every block has read them
    }

#pragma unroll
    for (int i = 0; i < kTM; ++i) {
        if (kSplit && i % S != rank) continue;
        const int64_t row = m0 + ty + 16 * i;
        if (row >= N) continue;
        const float d = kDeg ? inv_sqrt_degree(__ldg(rowptr + row + 1) - __ldg(rowptr + row)) : 1.0f;
#pragma unroll
        for (int j = 0; j < TN; ++j) {
            const int col = n0 + tx + 16 * j;
            if (col < F) Z[row * ldz + col] = kDeg ? d * acc[i][j] : acc[i][j];
        }
    }
}

template <int TN, bool kDeg>
void launch_bucket_tn(const BucketGemmArgs &g, const DeviceInfo &dev, cudaStream_t s) {
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
    const int nb = (g.K + 64 * g.bw - 1) / (64 * g.bw);
    if (S == 1) {
        launch_kernel(xnor_gemm_bucket_kernel<TN, kDeg, false>, dim3(gx, gy), dim3(kThreads), 0,
                      s, false, dim3(1, 1, 1), g.A, g.alpha, g.N, g.B, g.beta, g.F, g.K, g.words,
                      g.bw, nb, g.Z, g.ldz, g.rowptr);
        return;
    }
    launch_kernel(xnor_gemm_bucket_kernel<TN, kDeg, true>, dim3(gx, gy, S), dim3(kThreads), 0, s,
                  false, dim3(1, 1, S), g.A, g.alpha, g.N, g.B, g.beta, g.F, g.K, g.words, g.bw,
                  nb, g.Z, g.ldz, g.rowptr);
}

template <bool kDeg>
void launch_bucket_deg(const BucketGemmArgs &g, const DeviceInfo &dev, cudaStream_t s) {
    if (g.F > 32) launch_bucket_tn<4, kDeg>(g, dev, s);
    else if (g.F > 16) launch_bucket_tn<2, kDeg>(g, dev, s);
    else launch_bucket_tn<1, kDeg>(g, dev, s);
}

}  // namespace

void launch_pack_rows_bucketed(const float *X, int64_t N, int K, int64_t ldx, const float *scale,
                               const float *shift, int bw, uint64_t *bits, int words,
                               float *alpha, const DeviceInfo &dev, cudaStream_t stream) {
    if (N == 0) return;
    const int nb = (K + 64 * bw - 1) / (64 * bw);
    // Grid y = the bucket; grid x strides over rows, about 16 blocks per SM in all.
    const int64_t want = (N + kPackWarps - 1) / kPackWarps;
    int64_t cap = int64_t(dev.sm_count) * 16 / nb;
    if (cap < 1) cap = 1;
    pack_rows_bucketed_kernel<<<dim3(unsigned(want < cap ? want : cap), unsigned(nb)),
                                32 * kPackWarps, 0, stream>>>(X, N, K, ldx, scale, shift, bw,
                                                             bits, words, alpha, nb);
}

void launch_pack_weights_bucketed(const float *Wt, int K, int F, int64_t ldw, int bw,
                                  uint64_t *bits, int words, float *beta, cudaStream_t stream) {
    const int nb = (K + 64 * bw - 1) / (64 * bw);
    pack_weights_bucketed_kernel<<<dim3(unsigned((F + 31) / 32), unsigned(nb)), 32 * kWGroups, 0,
                                   stream>>>(Wt, K, F, ldw, bw, bits, words, beta, nb);
}

void launch_xnor_gemm_bucketed(const BucketGemmArgs &g, const DeviceInfo &dev,
                               cudaStream_t stream) {
    if (g.N == 0) return;
    if (g.rowptr != nullptr) launch_bucket_deg<true>(g, dev, stream);
    else launch_bucket_deg<false>(g, dev, stream);
}

}  // namespace bigcn

using namespace bigcn;

namespace {

constexpr size_t kBAlign = 256;
size_t bround(size_t x) { return (x + kBAlign - 1) / kBAlign * kBAlign; }

int bucket_words(int32_t B) { return (B > 0 && B % 64 == 0) ? B / 64 : 0; }
int64_t bucket_count(int32_t K, int32_t B) { return (int64_t(K) + B - 1) / B; }
// The packing kernels put the bucket on the grid's y dimension.
constexpr int64_t kMaxBuckets = 65535;

// Workspace of bigcn_layer_forward_bucketed: A bits, alpha (N x nb), B bits,
// beta (F x nb), Z' (N x F fp32).
struct BucketWorkspace {
    size_t a_bits, alpha, b_bits, beta, z, total;
};

bool bucket_workspace(int64_t N, int32_t K, int32_t F, int32_t B, BucketWorkspace *w) {
    if (N < 0 || K < 1 || F < 1 || bucket_words(B) == 0) return false;
    const int64_t words = bigcn_words(K), nb = bucket_count(K, B);
    if (nb > kMaxBuckets) return false;
    const int64_t widest = words > F ? (words > nb ? words : nb) : (F > nb ? F : nb);
    if (N > kMaxElems / widest) return false;
    size_t off = 0;
    w->a_bits = off; off = bround(off + size_t(N) * size_t(words) * 8);
    w->alpha = off;  off = bround(off + size_t(N) * size_t(nb) * 4);
    w->b_bits = off; off = bround(off + size_t(F) * size_t(words) * 8);
    w->beta = off;   off = bround(off + size_t(F) * size_t(nb) * 4);
    w->z = off;      off = bround(off + size_t(N) * size_t(F) * 4);
    w->total = off;
    return true;
}

}  // namespace

extern "C" bigcn_status bigcn_pack_rows_bucketed(const float *X, int64_t N, int32_t K,
                                                 int64_t ldx, const float *scale,
                                                 const float *shift, int32_t B, uint64_t *bits,
                                                 int32_t words, float *alpha, void *stream) {
    const int bw = bucket_words(B);
    if (N < 0 || K < 1 || ldx < K || bw == 0 || words < bigcn_words(K))
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    const int64_t nb = bucket_count(K, B);
    if (nb > kMaxBuckets) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / words || N > kMaxElems / nb))
        return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!X || !bits || !alpha) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(bits, 8) || !aligned_to(alpha, 4) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t xb = span_bytes(N, K, ldx, 4), bb = size_t(N) * words * 8,
                 ab = size_t(N) * size_t(nb) * 4;
    if (overlaps(bits, bb, X, xb) || overlaps(alpha, ab, X, xb) || overlaps(alpha, ab, bits, bb))
        return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    launch_pack_rows_bucketed(X, N, K, ldx, scale, shift, bw, bits, words, alpha, dev,
                              as_stream(stream));
    return launch_status();
}

extern "C" bigcn_status bigcn_pack_weights_bucketed(const float *Wt, int32_t K, int32_t F,
                                                    int64_t ldw, int32_t B, uint64_t *bits,
                                                    int32_t words, float *beta, void *stream) {
    const int bw = bucket_words(B);
    if (K < 1 || F < 1 || ldw < F || bw == 0 || words < bigcn_words(K))
        return BIGCN_ERR_INVALID_ARG;
    if (!Wt || !bits || !beta) return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(Wt, 4) || !aligned_to(bits, 8) || !aligned_to(beta, 4))
        return BIGCN_ERR_MISALIGNED;
    const int64_t nb = bucket_count(K, B);
    if (nb > kMaxBuckets) return BIGCN_ERR_INVALID_ARG;
    const size_t wb = span_bytes(K, F, ldw, 4), bb = size_t(F) * words * 8,
                 eb = size_t(F) * size_t(nb) * 4;
    if (overlaps(bits, bb, Wt, wb) || overlaps(beta, eb, Wt, wb) || overlaps(beta, eb, bits, bb))
        return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    launch_pack_weights_bucketed(Wt, K, F, ldw, bw, bits, words, beta, as_stream(stream));
    return launch_status();
}

extern "C" bigcn_status bigcn_xnor_gemm_bucketed(const uint64_t *a_bits, const float *alpha,
                                                 int64_t N, const uint64_t *b_bits,
                                                 const float *beta, int32_t F, int32_t K,
                                                 int32_t words, int32_t B, float *Z, int64_t ldz,
                                                 void *stream) {
    const int bw = bucket_words(B);
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || bw == 0 ||
        words != bigcn_words(K) || ldz < F)
        return BIGCN_ERR_INVALID_ARG;
    const int64_t nb = bucket_count(K, B);
    if (N > 0 && (N > kMaxElems / ldz || N > kMaxElems / words || N > kMaxElems / nb))
        return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!a_bits || !alpha || !b_bits || !beta || !Z) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(a_bits, 8) || !aligned_to(alpha, 4) || !aligned_to(b_bits, 8) ||
        !aligned_to(beta, 4) || !aligned_to(Z, 4))
        return BIGCN_ERR_MISALIGNED;
    const size_t zb = span_bytes(N, F, ldz, 4);
    const void *in[] = {a_bits, alpha, b_bits, beta};
    const size_t inb[] = {size_t(N) * words * 8, size_t(N) * size_t(nb) * 4,
                          size_t(F) * words * 8, size_t(F) * size_t(nb) * 4};
    for (int q = 0; q < 4; ++q)
        if (overlaps(Z, zb, in[q], inb[q])) return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    BucketGemmArgs g{a_bits, alpha, N, b_bits, beta, F, K, words, bw, Z, ldz, nullptr};
    launch_xnor_gemm_bucketed(g, dev, as_stream(stream));
    return launch_status();
}

extern "C" size_t bigcn_layer_bucketed_workspace_bytes(int64_t N, int32_t K, int32_t F,
                                                       int32_t B) {
    BucketWorkspace w;
    return bucket_workspace(N, K, F, B, &w) ? w.total : 0;
}

extern "C" bigcn_status bigcn_layer_forward_bucketed(int32_t B, const float *X, int64_t N,
                                                     int32_t K, int64_t ldx, const float *scale,
                                                     const float *shift, const float *Wt,
                                                     int32_t F, int64_t ldw,
                                                     const int64_t *rowptr, const int32_t *colidx,
                                                     int64_t nnz, void *workspace,
                                                     size_t ws_bytes, float *H, int64_t ldh,
                                                     void *stream) {
    BucketWorkspace w;
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || ldx < K || ldw < F || ldh < F ||
        nnz < 0)
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (!bucket_workspace(N, K, F, B, &w)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / ldh)) return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!X || !Wt || !rowptr || !H || !workspace || (nnz > 0 && !colidx))
        return BIGCN_ERR_INVALID_ARG;
    if (ws_bytes < w.total) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(Wt, 4) || !aligned_to(rowptr, 8) ||
        (colidx && !aligned_to(colidx, 4)) || !aligned_to(H, 4) ||
        !aligned_to(workspace, kBAlign) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t hb = span_bytes(N, F, ldh, 4);
    const void *inputs[] = {X, Wt, rowptr, colidx, scale, shift};
    const size_t in_bytes[] = {span_bytes(N, K, ldx, 4), span_bytes(K, F, ldw, 4),
                               size_t(N + 1) * 8, size_t(nnz) * 4, size_t(K) * 4, size_t(K) * 4};
    for (int q = 0; q < 6; ++q) {
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
    float *Zs = reinterpret_cast<float *>(ws + w.z);
    const int words = bigcn_words(K), bw = bucket_words(B);
    cudaStream_t s = as_stream(stream);
    launch_pack_rows_bucketed(X, N, K, ldx, scale, shift, bw, a_bits, words, alpha, dev, s);
    launch_pack_weights_bucketed(Wt, K, F, ldw, bw, b_bits, words, beta, s);
    BucketGemmArgs g{a_bits, alpha, N, b_bits, beta, F, K, words, bw, Zs, F, rowptr};
    launch_xnor_gemm_bucketed(g, dev, s);
    SpmmArgs a{rowptr, colidx, N, nnz, Zs, F, F, H, ldh, true, false};
    launch_spmm_norm(a, dev, s);
    return launch_status();
}
