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
// The packed weight columns and beta come from the weight-packing kernel
// that runs first; the kernel is used when both packed tiles fit in shared
// memory and rows are at most 2048 features (front_supported): a warp streams
// whole rows one batch after another, so with long rows and few rows per SM
// the separate row-packing kernel, which shares long rows between warps,
// keeps more bytes in flight.
#include "launch.cuh"

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
             const int64_t *__restrict__ rowptr, float *__restrict__ Z, int64_t ldz) {
    constexpr int BM = 16 * RI;
    extern __shared__ __align__(16) unsigned char smem[];
    const int pitch = words + 1;
    uint64_t *As = reinterpret_cast<uint64_t *>(smem);             // BM x pitch
    uint64_t *Bs = As + size_t(BM) * pitch;                          // F x pitch
    float *sAlpha = reinterpret_cast<float *>(Bs + size_t(F) * pitch);

    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int64_t m0 = int64_t(blockIdx.x) * BM;

    // Phase A: centre + sign + pack + |y| sums, rows warp, warp + 8, ...
    const int nchunks = (K + 31) >> 5;
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
        float l1 = 0.0f;
        for (int c0 = 0; c0 < nchunks; c0 += kFrontUnroll) {
            float v[kFrontUnroll];
#pragma unroll
            for (int u = 0; u < kFrontUnroll; ++u) {
                const int k = (c0 + u) * 32 + lane;
                v[u] = (k < K) ? __ldcs(x + k) : 0.0f;
            }
#pragma unroll
            for (int u = 0; u < kFrontUnroll; ++u) {
                const int k = (c0 + u) * 32 + lane;
                const bool in = k < K;
                float y = v[u];
                if (scale != nullptr && in) y = __fmaf_rn(y, __ldg(scale + k), __ldg(shift + k));
                const unsigned m = __ballot_sync(kFullMask, in && y >= 0.0f);
                if (lane == 0 && c0 + u < nchunks) a32[c0 + u] = m;
                l1 += in ? fabsf(y) : 0.0f;
            }
        }
        for (int q = nchunks + lane; q < nhalf; q += 32) a32[q] = 0u;
        l1 = warp_sum(l1);
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
        const float ai = sAlpha[rg + 16 * i] *
                         inv_sqrt_degree(__ldg(rowptr + row + 1) - __ldg(rowptr + row));
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
                  a.words, a.rowptr, a.Z, a.ldz);
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

}  // namespace

bool front_supported(int64_t N, int K, int F, const DeviceInfo &dev) {
    if (F < 1 || F > 128 || K < 1 || K > kFrontMaxK) return false;
    const size_t smem = front_smem(front_rows(N, dev), F, (K + 63) / 64);
    return smem <= kFrontMaxSmem && smem <= size_t(dev.max_smem_optin);
}

void launch_front(const FrontArgs &a, const DeviceInfo &dev, cudaStream_t s, bool pdl) {
    if (a.N == 0) return;
    const int BM = front_rows(a.N, dev);
    const size_t smem = front_smem(BM, a.F, a.words);
    if (BM == 64) launch_ri<4>(a, BM, smem, s, pdl);
    else if (BM == 32) launch_ri<2>(a, BM, smem, s, pdl);
    else launch_ri<1>(a, BM, smem, s, pdl);
}

}  // namespace bigcn
