// One warp's share of packing a row (Sec. 6.2 centring, Eq. 8 signs, the
// |y| sum of Eq. 7), shared by the row-packing and fused front kernels.
#pragma once

#include "bigcn_internal.cuh"

namespace bigcn {

constexpr int kPackUnroll = 8;

// Packs chunks sub, sub + G, ... of row `row` (lane l of chunk c owns
// feature 32c + l) and returns this warp's sum of |y| (all lanes).
template <bool kAffine>
__device__ __forceinline__ float pack_row_chunks(const float *__restrict__ x, int K,
                                                 const float *__restrict__ scale,
                                                 const float *__restrict__ shift,
                                                 uint32_t *__restrict__ out, int64_t ld32, int sub,
                                                 int G) {
    const int lane = threadIdx.x & 31;
    const int nchunks = (K + 31) >> 5;          // 32-bit half-words that carry signs
    float l1 = 0.0f;
    for (int m0 = sub; m0 < nchunks; m0 += G * kPackUnroll) {
        // All of a batch's loads (features and, when centring, the affine's
        // two factors) are issued before any is consumed.
        float v[kPackUnroll], sc[kPackUnroll], sh[kPackUnroll];
#pragma unroll
        for (int u = 0; u < kPackUnroll; ++u) {
            const int k = (m0 + u * G) * 32 + lane;
            v[u] = (k < K) ? __ldcs(x + k) : 0.0f;
            if (kAffine) {
                sc[u] = (k < K) ? __ldg(scale + k) : 1.0f;
                sh[u] = (k < K) ? __ldg(shift + k) : 0.0f;
            }
        }
#pragma unroll
        for (int u = 0; u < kPackUnroll; ++u) {
            const int c = m0 + u * G;
            const int k = c * 32 + lane;
            const bool in = k < K;
            float y = v[u];
            if (kAffine && in) y = __fmaf_rn(y, sc[u], sh[u]);
            const unsigned m = __ballot_sync(kFullMask, in && y >= 0.0f);
            if (c < nchunks && lane == 0) out[c] = m;
            l1 += in ? fabsf(y) : 0.0f;
        }
    }
    // Pad half-words past the last one that carries signs are zero.
    if (sub == 0)
        for (int64_t q = nchunks + lane; q < ld32; q += 32) out[q] = 0u;
    return warp_sum(l1);
}

}  // namespace bigcn
