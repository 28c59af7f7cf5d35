// One warp's share of packing a row (Sec. 6.2 centring, Eq. 8 signs, the
// |y| sum of Eq. 7), shared by the row-packing and fused front kernels.
//
// Lane l of chunk c owns feature 32c + l, so one __ballot_sync yields the
// chunk's 32-bit half-word of the packed row (LSB first). A warp takes
// chunks q, q + G, q + 2G, ... of the row (G warps share it), UNR chunks per
// batch: every load of a batch is issued before any is consumed. G and UNR
// are compile-time constants and each lane walks pointers to its own
// feature, so the batch's loads and stores carry immediate offsets; only
// the row's last batch checks bounds.
#pragma once

#include "bigcn_internal.cuh"

namespace bigcn {

// Where the centring affine y = x * scale + shift comes from: global memory
// (loaded with the batch's features, or, kGlobalLate, as each is consumed:
// fewer registers, for kernels that need full occupancy), shared memory
// (float2 pairs), or nowhere (identity).
enum class Affine { kNone, kGlobal, kGlobalLate, kShared };

template <int G, int UNR, Affine kA>
__device__ __forceinline__ float pack_share(const float *__restrict__ x, int K,
                                            const float *__restrict__ scale,
                                            const float *__restrict__ shift,
                                            const float2 *__restrict__ st,
                                            uint32_t *__restrict__ out, int64_t ld32, int q) {
    const int lane = threadIdx.x & 31;
    const int nchunks = (K + 31) >> 5;          // 32-bit half-words that carry signs
    const int full = K >> 5;                    // chunks with all 32 features inside
    constexpr int kStep = G * 32;               // features between a lane's chunks
    const int off = q * 32 + lane;
    const float *xl = x + off;
    constexpr bool kG = kA == Affine::kGlobal || kA == Affine::kGlobalLate;
    const float *sl = kG ? scale + off : nullptr;
    const float *tl = kG ? shift + off : nullptr;
    const float2 *pl = kA == Affine::kShared ? st + off : nullptr;
    uint32_t *ol = out + q;
    const bool writer = lane == 0;
    float l1 = 0.0f;
    int c0 = q;
    for (; c0 + (UNR - 1) * G < full; c0 += UNR * G) {
        float v[UNR], a[UNR], b[UNR];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            v[u] = __ldcs(xl + u * kStep);
            if (kA == Affine::kGlobal) {
                a[u] = __ldg(sl + u * kStep);
                b[u] = __ldg(tl + u * kStep);
            }
        }
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            float y = v[u];
            if (kA == Affine::kGlobal) y = __fmaf_rn(y, a[u], b[u]);
            if (kA == Affine::kGlobalLate)
                y = __fmaf_rn(y, __ldg(sl + u * kStep), __ldg(tl + u * kStep));
            if (kA == Affine::kShared) {
                const float2 p = pl[u * kStep];
                y = __fmaf_rn(y, p.x, p.y);
            }
            const unsigned m = __ballot_sync(kFullMask, y >= 0.0f);
            if (writer) ol[u * G] = m;
            l1 += fabsf(y);
        }
        xl += UNR * kStep;
        if (kG) {
            sl += UNR * kStep;
            tl += UNR * kStep;
        }
        if (kA == Affine::kShared) pl += UNR * kStep;
        ol += UNR * G;
    }
    if (c0 < nchunks) {                         // the last, partial batch
        float v[UNR], a[UNR], b[UNR];
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            const bool in = (c0 + u * G) * 32 + lane < K;
            v[u] = in ? __ldcs(xl + u * kStep) : 0.0f;
            if (kA == Affine::kGlobal) {
                a[u] = in ? __ldg(sl + u * kStep) : 0.0f;
                b[u] = in ? __ldg(tl + u * kStep) : 0.0f;
            }
        }
#pragma unroll
        for (int u = 0; u < UNR; ++u) {
            const int c = c0 + u * G;
            const bool in = c * 32 + lane < K;
            float y = v[u];
            if (kA == Affine::kGlobal) y = __fmaf_rn(y, a[u], b[u]);
            if (kA == Affine::kGlobalLate && in)
                y = __fmaf_rn(y, __ldg(sl + u * kStep), __ldg(tl + u * kStep));
            if (kA == Affine::kShared && in) {
                const float2 p = pl[u * kStep];
                y = __fmaf_rn(y, p.x, p.y);
            }
            const unsigned m = __ballot_sync(kFullMask, in && y >= 0.0f);
            if (writer && c < nchunks) ol[u * G] = m;
            l1 += in ? fabsf(y) : 0.0f;
        }
    }
    // Pad half-words past the last one that carries signs are zero.
    if (q == 0)
        for (int64_t h = nchunks + lane; h < ld32; h += 32) out[h] = 0u;
    return warp_sum(l1);
}

}  // namespace bigcn
