// Layer-1 front of the fused forward (Wang et al., CVPR 2021): steps 1, 2
// and 4 of one layer in one kernel -- centring (Sec. 6.2), sign
// binarization with the per-node scale (Eqs. 7-8) and the XNOR-popcount
// product with its scaled, degree-normalised epilogue (Eqs. 11-12):
//
//   Z'[i,j] = (alpha_i / sqrt(dhat_i)) * (beta_j * (K - 2 popc(a_i ^ b_j)))
//
// Each block owns BM = 16 * RI rows. Phase A: its 8 warps stream the rows of
// X (one warp per row at a time, 8 chunks of 32 features in flight), and
// every chunk's ballot lands directly in shared memory as a 32-bit half-word
// of the packed row; the packed rows never go to global memory. Phase B:
// thread (cg, rg) counts mismatches for rows rg + 16 i and columns cg + 16 j
// against the packed weight columns, which the block loads once into shared
// memory (odd row pitch: conflict-free). Several blocks per SM overlap one
// block's HBM-bound phase A with another's POPC-bound phase B.
//
// Either kernel can leave Z' factored instead (D16 non-null, K <= 32767):
// the integer dots as uint16 with a bias of 32768 (rows padded to a multiple
// of 4 with zero dots) and the row scale alpha_i / sqrt(dhat_i), for an
// aggregation that gathers half-size rows and applies beta per column.
//
// The packed weight columns and beta come from the weight-packing kernel
// that runs first. This whole-row kernel is used when there are enough rows
// to give every warp its own, both packed tiles fit in shared memory and rows
// are at most 2048 features; with fewer rows the split front below shares
// each row between several warps, as the row-packing kernel does, so that
// more of the GPU's warps keep loads in flight (front_supported picks).
#include "launch.cuh"
#include "pack_row.cuh"

namespace bigcn {
namespace {

constexpr int kFrontThreads = 256;
constexpr int kFrontWarps = kFrontThreads / 32;
constexpr int kFrontUnroll = 8;
constexpr int kFrontMaxK = 2048;
constexpr size_t kFrontMaxSmem = 160 * 1024;

size_t front_smem(int BM, int F, int words) {
    const size_t pitch = size_t(words) + 1;   // odd pitch in 64-bit words
    return (size_t(BM) + size_t(F)) * pitch * 8 + size_t(BM) * 4;
}

template <int RI, int CJ>
__global__ void __launch_bounds__(kFrontThreads)
front_kernel(const float *__restrict__ X, int64_t N, int K, int64_t ldx,
             const float *__restrict__ scale, const float *__restrict__ shift,
             const uint64_t *__restrict__ wbits, const float *__restrict__ beta, int F, int words,
             const int64_t *__restrict__ rowptr, float *__restrict__ Z, int64_t ldz,
             uint16_t *__restrict__ D16, int64_t ldd16, float *__restrict__ rowscale, bool f16) {
    constexpr int BM = 16 * RI;
    extern __shared__ __align__(16) unsigned char smem[];
    const int pitch = words + 1;
    uint64_t *As = reinterpret_cast<uint64_t *>(smem);             // BM x pitch
    uint64_t *Bs = As + size_t(BM) * pitch;                          // F x pitch
    float *sAlpha = reinterpret_cast<float *>(Bs + size_t(F) * pitch);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t m0 = int64_t(blockIdx.x) * BM;

    // Phase A: centre + sign + pack + |y| sums, rows warp, warp + 8, ...
    const int nhalf = 2 * words;
    for (int r = warp; r < BM; r += kFrontWarps) {
        const int64_t row = m0 + r;
        uint32_t *a32 = reinterpret_cast<uint32_t *>(As + size_t(r) * pitch);
        if (row >= N) {
            for (int q = lane; q < nhalf; q += 32) a32[q] = 0u;
            if (lane == 0) sAlpha[r] = 0.0f;
            continue;
        }
        const float *x = X + row * ldx;
        const float l1 =
            scale != nullptr
                ? pack_share<1, kFrontUnroll, Affine::kGlobal>(x, K, scale, shift, nullptr, a32, nhalf, 0)
                : pack_share<1, kFrontUnroll, Affine::kNone>(x, K, nullptr, nullptr, nullptr, a32, nhalf, 0);
        if (lane == 0) sAlpha[r] = l1 / float(K);
    }

    // The packed weight columns are the previous kernel's output: wait for it
    // (phase A above only read the call's inputs), then stage them (coalesced,
    // once per block).
    grid_dependency_wait();
    for (int q = tid; q < F * words; q += kFrontThreads)
        Bs[(q / words) * pitch + (q % words)] = __ldg(wbits + q);
    __syncthreads();

    // Phase B: XNOR-popcount against every column.
    const int cg = tid & 15, rg = tid >> 4;
    int mism[RI][CJ];
#pragma unroll
    for (int i = 0; i < RI; ++i)
#pragma unroll
        for (int j = 0; j < CJ; ++j) mism[i][j] = 0;
    for (int w = 0; w < words; ++w) {
        uint64_t a[RI], b[CJ];
#pragma unroll
        for (int i = 0; i < RI; ++i) a[i] = As[size_t(rg + 16 * i) * pitch + w];
#pragma unroll
        for (int j = 0; j < CJ; ++j) {
            const int c = cg + 16 * j;
            b[j] = c < F ? Bs[size_t(c) * pitch + w] : 0ull;
        }
#pragma unroll
        for (int i = 0; i < RI; ++i)
#pragma unroll
            for (int j = 0; j < CJ; ++j) mism[i][j] += __popcll(a[i] ^ b[j]);
    }

#pragma unroll
    for (int i = 0; i < RI; ++i) {
        const int64_t row = m0 + rg + 16 * i;
        if (row >= N) continue;
        const float ai = rowptr == nullptr
                             ? sAlpha[rg + 16 * i]
                             : sAlpha[rg + 16 * i] *
                                   inv_sqrt_degree(__ldg(rowptr + row + 1) - __ldg(rowptr + row));
        if (D16 != nullptr) {               // compressed output: biased dots + row scale
            if (cg == 0) rowscale[row] = ai;
#pragma unroll
            for (int j = 0; j < CJ; ++j) {
                const int col = cg + 16 * j;
                if (col < ldd16) D16[row * ldd16 + col] = encode_dot(K - 2 * mism[i][j], col < F, f16);
            }
            continue;
        }
#pragma unroll
        for (int j = 0; j < CJ; ++j) {
            const int col = cg + 16 * j;
            if (col < F) Z[row * ldz + col] = ai * (__ldg(beta + col) * float(K - 2 * mism[i][j]));
        }
    }
}

template <int RI, int CJ>
void launch_ri_cj(const FrontArgs &a, int BM, size_t smem, cudaStream_t s, bool pdl) {
    const unsigned grid = unsigned((a.N + BM - 1) / BM);
    cudaFuncSetAttribute(front_kernel<RI, CJ>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         int(smem));
    launch_kernel(front_kernel<RI, CJ>, dim3(grid), dim3(kFrontThreads), smem, s, pdl,
                  dim3(1, 1, 1), a.X, a.N, a.K, a.ldx, a.scale, a.shift, a.wbits, a.beta, a.F,
                  a.words, a.rowptr, a.Z, a.ldz, a.D16, a.ldd16, a.rowscale, a.dots_f16);
}

template <int RI>
void launch_ri(const FrontArgs &a, int BM, size_t smem, cudaStream_t s, bool pdl) {
    if (a.F <= 16) launch_ri_cj<RI, 1>(a, BM, smem, s, pdl);
    else if (a.F <= 32) launch_ri_cj<RI, 2>(a, BM, smem, s, pdl);
    else if (a.F <= 64) launch_ri_cj<RI, 4>(a, BM, smem, s, pdl);
    else launch_ri_cj<RI, 8>(a, BM, smem, s, pdl);
}

// Rows per block: the largest of 64, 32, 16 that still gives every SM four
// blocks, so that phases of different blocks overlap.
int front_rows(int64_t N, const DeviceInfo &dev) {
    for (int BM = 64; BM > 16; BM /= 2)
        if ((N + BM - 1) / BM >= 4 * int64_t(dev.sm_count)) return BM;
    return 16;
}

// ---------------------------------------------------------------------------
// Split front, for layers with few rows (fewer than one warp per row would
// leave most of the GPU idle, e.g. a few thousand long rows): each 16-warp
// block takes R = 16 / G rows at a time, G warps per row (the row-packing
// kernel's split, the same chunk order and the same alpha summation), and
// writes the packed rows to shared memory. The block then computes their
// products: the 32 G threads of a row take P lanes per output column (P a
// power of two, words w = t mod P, t mod P + P, ... for lane t of the
// column), add their mismatch counts with shuffles and write Z' as above.
// The centring affine is staged in shared memory as (scale, shift) pairs
// when the block starts (it is the call's input); the packed weight columns
// are staged once per block after the dependency wait, which comes only
// after the block's first rows have been streamed.

// Shared memory: F x pitch packed columns, 16 x pitch packed rows, and the
// centring affine as K (scale, shift) pairs; at most kSplitMaxSmem, so that
// two blocks (with the 1 KB each that the SM reserves) share an SM's 228 KB.
constexpr int kSplitThreads = 512;
constexpr int kSplitWarps = kSplitThreads / 32;
constexpr size_t kSplitMaxSmem = 112 * 1024;

// Row pitch in 64-bit words. With one lane per output column (P = 1) a lane
// reads its column two words at a time (16-byte loads): the rows are padded
// to an even count of words with a zero word, and the pitch is = 2 mod 4
// words, so that the eight columns of a quarter-warp fall on the eight
// distinct 16-byte slots of a 128-byte line (conflict-free). Otherwise an
// odd pitch keeps the 8-byte loads of neighbouring columns conflict-free.
int split_pitch(int words, int P) {
    if (P != 1) return words | 1;
    const int even = (words + 1) & ~1;
    return even % 4 == 2 ? even : even + 2;
}

size_t split_smem(int F, int K, int pitch, bool affine) {
    return (size_t(F) + size_t(kSplitWarps)) * size_t(pitch) * 8 +
           (affine ? size_t(K) * 8 : 0);
}

// Warps per row: the row-packing kernel's policy (split while the grid is
// short of one wave of warps and every warp keeps an 8-chunk batch).
int split_warps(int64_t N, int K, const DeviceInfo &dev) {
    const int nchunks = (K + 31) / 32;
    const int64_t full_wave = int64_t(dev.sm_count) * 64;
    int G = 1;
    while (G < kFrontWarps && N * G < full_wave && nchunks >= 2 * G * 8) G *= 2;
    // Each warp that shares a row adds a product pass: stop splitting once
    // half a wave of warps is busy (measured: two warps per row beat four on
    // a few thousand rows of 3703 features).
    while (G > 2 && N * (G / 2) >= full_wave / 2) G /= 2;
    return G;
}

template <int G, bool kAffine>
__global__ void __launch_bounds__(kSplitThreads, 3)
front_split_kernel(const float *__restrict__ X, int64_t N, int K, int64_t ldx,
                   const float *__restrict__ scale, const float *__restrict__ shift,
                   const uint64_t *__restrict__ wbits, const float *__restrict__ beta, int F,
                   int words, const int64_t *__restrict__ rowptr, float *__restrict__ Z,
                   int64_t ldz, uint16_t *__restrict__ D16, int64_t ldd16,
                   float *__restrict__ rowscale, int P, int pitch, bool f16) {
    extern __shared__ __align__(16) unsigned char smem[];
    __shared__ float part[kSplitWarps];
    constexpr int R = kSplitWarps / G;       // rows per group
    constexpr int T = 32 * G;                // threads per row in the product
    constexpr Affine kA = kAffine ? Affine::kShared : Affine::kNone;
    const int npairs = (words + 1) >> 1;     // P = 1: 16-byte pairs of words per row
    uint64_t *Ws = reinterpret_cast<uint64_t *>(smem);      // F x pitch packed columns
    uint64_t *As = Ws + size_t(F) * pitch;                   // R x pitch packed rows
    float2 *sST = reinterpret_cast<float2 *>(As + size_t(kSplitWarps) * pitch);
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int rr = tid / T, tt = tid % T, sub = tt % P;
    const int cstep = T / P;                 // columns per pass
    const int Fw = D16 != nullptr ? int(ldd16) : F;   // columns written (with padding)
    const int passes = (Fw + cstep - 1) / cstep;
    if (kAffine) {
        for (int k0 = tid; k0 < K; k0 += 4 * kSplitThreads) {
            float2 v[4];
#pragma unroll
            for (int u = 0; u < 4; ++u) {
                const int k = k0 + u * kSplitThreads;
                if (k < K) v[u] = make_float2(__ldg(scale + k), __ldg(shift + k));
            }
#pragma unroll
            for (int u = 0; u < 4; ++u)
                if (k0 + u * kSplitThreads < K) sST[k0 + u * kSplitThreads] = v[u];
        }
        __syncthreads();
    }
    bool staged = false;
    for (int64_t group = blockIdx.x; group * R < N; group += gridDim.x) {
        const int64_t row = group * R + warp / G;
        uint32_t *a32 = reinterpret_cast<uint32_t *>(As + size_t(warp / G) * pitch);
        const float l1 = (row < N) ? pack_share<G, kFrontUnroll, kA>(X + row * ldx, K, nullptr,
                                                                     nullptr, sST, a32,
                                                                     P == 1 ? 4 * npairs
                                                                            : 2 * words,
                                                                     warp % G)
                                   : 0.0f;
        if (lane == 0) part[warp] = l1;
        if (!staged) {
            grid_dependency_wait();     // the packed weight columns come from the previous kernel
            const int n = F * words;
            for (int q0 = tid; q0 < n; q0 += 4 * kSplitThreads) {
                uint64_t v[4];
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int q = q0 + u * kSplitThreads;
                    if (q < n) v[u] = __ldg(wbits + q);
                }
#pragma unroll
                for (int u = 0; u < 4; ++u) {
                    const int q = q0 + u * kSplitThreads;
                    if (q < n) Ws[(q / words) * pitch + (q % words)] = v[u];
                }
            }
            if (P == 1 && (words & 1))      // the zero word that completes the last pair
                for (int c = tid; c < F; c += kSplitThreads) Ws[c * pitch + words] = 0ull;
            staged = true;
        }
        __syncthreads();
        const int64_t row2 = group * R + rr;
        if (row2 < N) {                      // uniform over each warp (T is a multiple of 32)
            float t = 0.0f;
#pragma unroll
            for (int g = 0; g < G; ++g) t += part[rr * G + g];
            const float ai =
                rowptr == nullptr
                    ? t / float(K)
                    : (t / float(K)) *
                          inv_sqrt_degree(__ldg(rowptr + row2 + 1) - __ldg(rowptr + row2));
            if (D16 != nullptr && tt == 0) rowscale[row2] = ai;
            const uint64_t *a = As + size_t(rr) * pitch;
            const ulonglong2 *a2 = reinterpret_cast<const ulonglong2 *>(a);
            for (int j = 0; j < passes; ++j) {
                const int c = tt / P + j * cstep;
                int mism = 0;
                if (c < F) {
                    if (P == 1) {    // a lane per column: two words per 16-byte load
                        const ulonglong2 *w2 =
                            reinterpret_cast<const ulonglong2 *>(Ws + size_t(c) * pitch);
#pragma unroll 4
                        for (int q = 0; q < npairs; ++q) {
                            const ulonglong2 x = a2[q], y = w2[q];
                            mism += __popcll(x.x ^ y.x) + __popcll(x.y ^ y.y);
                        }
                    } else {
                        for (int w = sub; w < words; w += P)
                            mism += __popcll(a[w] ^ Ws[c * pitch + w]);
                    }
                }
                for (int o = 1; o < P; o <<= 1) mism += __shfl_xor_sync(kFullMask, mism, o);
                if (sub != 0 || c >= Fw) continue;
                if (D16 != nullptr)
                    D16[row2 * ldd16 + c] = encode_dot(K - 2 * mism, c < F, f16);
                else
                    Z[row2 * ldz + c] = ai * (__ldg(beta + c) * float(K - 2 * mism));
            }
        }
        __syncthreads();                     // As and part are rewritten by the next rows
    }
    if (!staged) grid_dependency_wait();
}

bool split_supported(int64_t N, int K, int F, const DeviceInfo &dev) {
    const int words = (K + 63) / 64;
    const int pitch = split_pitch(words, 1) > split_pitch(words, 2) ? split_pitch(words, 1)
                                                                     : split_pitch(words, 2);
    const size_t smem = split_smem(F, K, pitch, true);
    return F >= 1 && F <= 128 && split_warps(N, K, dev) > 1 && smem <= kSplitMaxSmem &&
           smem <= size_t(dev.max_smem_optin);
}

void launch_split(const FrontArgs &a, const DeviceInfo &dev, cudaStream_t s, bool pdl) {
    const int G = split_warps(a.N, a.K, dev);
    int fp = 1;
    while (fp < a.F) fp *= 2;
    int P = 32 * G / fp;
    if (P < 1) P = 1;
    if (P > 32) P = 32;
    const bool affine = a.scale != nullptr;
    const int pitch = split_pitch(a.words, P);
    const size_t smem = split_smem(a.F, a.K, pitch, affine);
    void (*kernel)(const float *, int64_t, int, int64_t, const float *, const float *,
                   const uint64_t *, const float *, int, int, const int64_t *, float *, int64_t,
                   uint16_t *, int64_t, float *, int, int, bool);
    if (G == 2) kernel = affine ? front_split_kernel<2, true> : front_split_kernel<2, false>;
    else if (G == 4) kernel = affine ? front_split_kernel<4, true> : front_split_kernel<4, false>;
    else kernel = affine ? front_split_kernel<8, true> : front_split_kernel<8, false>;
    cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kSplitThreads, smem) !=
            cudaSuccess ||
        per_sm < 1)
        per_sm = 1;
    const int64_t groups = (a.N + kSplitWarps / G - 1) / (kSplitWarps / G);
    const int64_t resident = int64_t(per_sm) * dev.sm_count;
    launch_kernel(kernel, dim3(unsigned(groups < resident ? groups : resident)),
                  dim3(kSplitThreads), smem, s, pdl, dim3(1, 1, 1), a.X, a.N, a.K, a.ldx, a.scale,
                  a.shift, a.wbits, a.beta, a.F, a.words, a.rowptr, a.Z, a.ldz, a.D16, a.ldd16,
                  a.rowscale, P, pitch, a.dots_f16);
}

}  // namespace

bool front_supported(int64_t N, int K, int F, const DeviceInfo &dev) {
    if (split_supported(N, K, F, dev)) return true;
    if (F < 1 || F > 128 || K < 1 || K > kFrontMaxK) return false;
    const size_t smem = front_smem(front_rows(N, dev), F, (K + 63) / 64);
    return smem <= kFrontMaxSmem && smem <= size_t(dev.max_smem_optin);
}

bool front_split_supported(int64_t N, int K, int F, const DeviceInfo &dev) {
    return split_supported(N, K, F, dev);
}

void launch_front(const FrontArgs &a, const DeviceInfo &dev, cudaStream_t s, bool pdl) {
    if (a.N == 0) return;
    if (split_supported(a.N, a.K, a.F, dev)) {
        launch_split(a, dev, s, pdl);
        return;
    }
    const int BM = front_rows(a.N, dev);
    const size_t smem = front_smem(BM, a.F, a.words);
    if (BM == 64) launch_ri<4>(a, BM, smem, s, pdl);
    else if (BM == 32) launch_ri<2>(a, BM, smem, s, pdl);
    else launch_ri<1>(a, BM, smem, s, pdl);
}

}  // namespace bigcn
