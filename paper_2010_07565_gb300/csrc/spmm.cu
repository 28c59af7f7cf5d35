// Step 5 of the Bi-GCN layer forward (Wang et al., CVPR 2021, Eq. 13 with
// the operator of Eq. 1): H = D^-1/2 (A + I) D^-1/2 Z over a CSR graph.
//
// One warp per output row. The warp is split into P = 32 / L groups of L
// lanes; each group gathers a different neighbour's row of Z, lane by lane
// in VEC-wide vectors (NV per lane), so that rows narrower than a warp still
// keep all 32 lanes busy. Neighbour indices (and, unless Z is pre-scaled,
// their 1/sqrt(dhat_j)) are fetched 32 at a time, one per lane, then
// broadcast with shuffles. The self-loop that A + I adds is the first entry
// of every row's list. Partial sums are combined across groups with xor
// shuffles and group 0 writes H_i scaled by 1/sqrt(dhat_i). A grid y
// dimension splits wide rows into column slabs of L * NV * VEC features.
//
// Bounds: the row range is clamped to [0, nnz] and column indices outside
// [0, N) are skipped, so a malformed CSR cannot make the kernel read out of
// bounds.
#include "launch.cuh"

namespace bigcn {
namespace {

constexpr int kSpmmThreads = 256;
constexpr int kUnroll = 4;

template <int VEC> struct Vec;
template <> struct Vec<1> {
    using T = float;
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) { acc[0] = fmaf(w, v, acc[0]); }
    static __device__ __forceinline__ void set(float *acc, T &v) { v = acc[0]; }
};
template <> struct Vec<2> {
    using T = float2;
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) {
        acc[0] = fmaf(w, v.x, acc[0]);
        acc[1] = fmaf(w, v.y, acc[1]);
    }
    static __device__ __forceinline__ void set(float *acc, T &v) { v = make_float2(acc[0], acc[1]); }
};
template <> struct Vec<4> {
    using T = float4;
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) {
        acc[0] = fmaf(w, v.x, acc[0]);
        acc[1] = fmaf(w, v.y, acc[1]);
        acc[2] = fmaf(w, v.z, acc[2]);
        acc[3] = fmaf(w, v.w, acc[3]);
    }
    static __device__ __forceinline__ void set(float *acc, T &v) {
        v = make_float4(acc[0], acc[1], acc[2], acc[3]);
    }
};

template <int VEC, int L, int NV, bool kPrescaled>
__global__ void __launch_bounds__(kSpmmThreads)
spmm_norm_kernel(const int64_t *__restrict__ rowptr, const int32_t *__restrict__ colidx,
                 int64_t N, int64_t nnz, const float *__restrict__ Z, int64_t ldz, int F,
                 float *__restrict__ H, int64_t ldh) {
    using V = typename Vec<VEC>::T;
    constexpr int P = 32 / L;                 // neighbours gathered in parallel
    constexpr int SLAB = L * NV * VEC;        // features per column slab

    const int lane = threadIdx.x & 31;
    const int64_t i = (int64_t(blockIdx.x) * kSpmmThreads + threadIdx.x) >> 5;
    if (i >= N) return;
    const int g = lane / L, sl = lane % L;
    const int f0 = blockIdx.y * SLAB;

    const int64_t rb = __ldg(rowptr + i), re = __ldg(rowptr + i + 1);
    const int64_t b = min(max(rb, int64_t(0)), nnz);
    const int64_t e = min(max(re, b), nnz);
    const float dinv_i = inv_sqrt_degree(e - b);
    const int64_t total = (e - b) + 1;        // + the self-loop

    float acc[NV][VEC];
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int c = 0; c < VEC; ++c) acc[v][c] = 0.0f;

    for (int64_t base = 0; base < total; base += 32) {
        // Lane q fetches entry base + q of the row's list (entry 0 = self).
        int j = -1;
        float wj = 0.0f;
        const int64_t q = base + lane;
        if (q < total) {
            j = (q == 0) ? int(i) : __ldg(colidx + b + q - 1);
            if (j < 0 || j >= N) j = -1;
            if (j >= 0)
                wj = kPrescaled ? 1.0f
                                : inv_sqrt_degree(__ldg(rowptr + j + 1) - __ldg(rowptr + j));
        }
        const int cnt = int(min(total - base, int64_t(32)));
        for (int t0 = 0; t0 < cnt; t0 += P * kUnroll) {
            V val[kUnroll][NV];
            float w[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int src = t0 + u * P + g;          // < 32 always
                const int jj = __shfl_sync(kFullMask, j, src & 31);
                w[u] = __shfl_sync(kFullMask, wj, src & 31);
                const bool live = src < cnt && jj >= 0;
                if (!live) w[u] = 0.0f;
                const float *zr = Z + int64_t(live ? jj : 0) * ldz;
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int f = f0 + (v * L + sl) * VEC;
                    if (live && f < F) val[u][v] = __ldg(reinterpret_cast<const V *>(zr + f));
                    else val[u][v] = V{};
                }
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u)
#pragma unroll
                for (int v = 0; v < NV; ++v) Vec<VEC>::fma(acc[v], val[u][v], w[u]);
        }
    }

#pragma unroll
    for (int o = L; o < 32; o <<= 1)
#pragma unroll
        for (int v = 0; v < NV; ++v)
#pragma unroll
            for (int c = 0; c < VEC; ++c) acc[v][c] += __shfl_xor_sync(kFullMask, acc[v][c], o);

    if (g == 0) {
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int f = f0 + (v * L + sl) * VEC;
            if (f < F) {
#pragma unroll
                for (int c = 0; c < VEC; ++c) acc[v][c] *= dinv_i;
                V out;
                Vec<VEC>::set(acc[v], out);
                *reinterpret_cast<V *>(H + i * ldh + f) = out;
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Layer-1 aggregation fused with layer 2's binarization and product.
//
// Each warp computes H1_i = dinv_i * sum_j Z1'_j exactly as the kernel above
// (VEC = 4, one vector per lane, pre-scaled rows), then, without writing H1
// (unless asked to), takes layer 2's steps on the row while it is still in
// registers: the signs of its Fh <= 128 features become one or two 64-bit
// words (four ballots, one per vector component, spread into place), the
// row scale alpha2_i = mean |H1_i| is one warp reduction, and the XNOR
// popcount against the (shared-memory) packed columns of W2 gives
//   Z2'_ij = (alpha2_i * dinv_i) * (beta2_j * (Fh - 2 popc(h_i ^ w_j))),
// the same expression the product's degree-scaled epilogue evaluates.

// Spreads 16 bits so that bit i lands on bit 4i of a 64-bit word.
__device__ __forceinline__ uint64_t spread16by4(uint32_t x) {
    uint64_t v = x & 0xFFFFu;
    v = (v | (v << 24)) & 0x000000FF000000FFull;
    v = (v | (v << 12)) & 0x000F000F000F000Full;
    v = (v | (v << 6)) & 0x0303030303030303ull;
    v = (v | (v << 3)) & 0x1111111111111111ull;
    return v;
}

template <int L>
__global__ void __launch_bounds__(kSpmmThreads, 4)
spmm_pack_gemm_kernel(const int64_t *__restrict__ rowptr, const int32_t *__restrict__ colidx,
                      int64_t N, int64_t nnz, const float *__restrict__ Z1, int Fh,
                      float *__restrict__ H1, int64_t ldh, const uint64_t *__restrict__ wbits2,
                      const float *__restrict__ beta2, int Fo, int words2,
                      float *__restrict__ Z2, int64_t ldz2) {
    constexpr int P = 32 / L;
    __shared__ uint64_t sW[kMaxFusedOut * 2];
    __shared__ float sBeta[kMaxFusedOut];
    for (int q = threadIdx.x; q < Fo * words2; q += kSpmmThreads) sW[q] = __ldg(wbits2 + q);
    for (int q = threadIdx.x; q < Fo; q += kSpmmThreads) sBeta[q] = __ldg(beta2 + q);
    __syncthreads();

    const int lane = threadIdx.x & 31;
    const int64_t i = (int64_t(blockIdx.x) * kSpmmThreads + threadIdx.x) >> 5;
    if (i >= N) return;
    const int g = lane / L, sl = lane % L;
    const int f = sl * 4;                      // this lane's first feature

    const int64_t rb = __ldg(rowptr + i), re = __ldg(rowptr + i + 1);
    const int64_t b = min(max(rb, int64_t(0)), nnz);
    const int64_t e = min(max(re, b), nnz);
    const float dinv_i = inv_sqrt_degree(e - b);
    const int64_t total = (e - b) + 1;

    float acc[4] = {0.0f, 0.0f, 0.0f, 0.0f};
    for (int64_t base = 0; base < total; base += 32) {
        int j = -1;
        const int64_t q = base + lane;
        if (q < total) {
            j = (q == 0) ? int(i) : __ldg(colidx + b + q - 1);
            if (j < 0 || j >= N) j = -1;
        }
        const int cnt = int(min(total - base, int64_t(32)));
        for (int t0 = 0; t0 < cnt; t0 += P * kUnroll) {
            float4 val[kUnroll];
            bool live[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                const int src = t0 + u * P + g;
                const int jj = __shfl_sync(kFullMask, j, src & 31);
                live[u] = src < cnt && jj >= 0 && f < Fh;
                val[u] = live[u] ? __ldg(reinterpret_cast<const float4 *>(Z1 + int64_t(jj) * Fh + f))
                                 : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < kUnroll; ++u) {
                acc[0] += val[u].x;
                acc[1] += val[u].y;
                acc[2] += val[u].z;
                acc[3] += val[u].w;
            }
        }
    }
#pragma unroll
    for (int o = L; o < 32; o <<= 1)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[c] += __shfl_xor_sync(kFullMask, acc[c], o);

    float h[4];
#pragma unroll
    for (int c = 0; c < 4; ++c) h[c] = acc[c] * dinv_i;
    if (H1 != nullptr && g == 0) {
#pragma unroll
        for (int c = 0; c < 4; ++c)
            if (f + c < Fh) H1[i * ldh + f + c] = h[c];
    }

    // Layer 2, Eqs. 7-8: signs of H1_i packed LSB-first, and its mean |.|.
    uint64_t w0 = 0, w1 = 0;
    float l1 = 0.0f;
#pragma unroll
    for (int c = 0; c < 4; ++c) {
        const bool in = g == 0 && f + c < Fh;
        const unsigned m = __ballot_sync(kFullMask, in && h[c] >= 0.0f);
        w0 |= spread16by4(m) << c;
        w1 |= spread16by4(m >> 16) << c;
        l1 += in ? fabsf(h[c]) : 0.0f;
    }
    l1 = warp_sum(l1);
    const float a = (l1 / float(Fh)) * dinv_i;

    // Layer 2, Eqs. 11-12, pre-scaled by this row's 1/sqrt(dhat_i).
    for (int jo = lane; jo < Fo; jo += 32) {
        int mism = __popcll(w0 ^ sW[jo * words2]);
        if (words2 > 1) mism += __popcll(w1 ^ sW[jo * words2 + 1]);
        const int d = Fh - 2 * mism;
        Z2[i * ldz2 + jo] = a * (sBeta[jo] * float(d));
    }
}

template <int VEC, int L, int NV, bool kPre>
void launch_cfg(const SpmmArgs &a, cudaStream_t s) {
    constexpr int SLAB = L * NV * VEC;
    const int64_t rows_per_block = kSpmmThreads / 32;
    dim3 grid(unsigned((a.N + rows_per_block - 1) / rows_per_block),
              unsigned((a.F + SLAB - 1) / SLAB));
    spmm_norm_kernel<VEC, L, NV, kPre><<<grid, kSpmmThreads, 0, s>>>(
        a.rowptr, a.colidx, a.N, a.nnz, a.Z, a.ldz, a.F, a.H, a.ldh);
}

// Lanes per neighbour L = the power of two >= the row's vector count (at
// least 4, at most 32); NV = 2 vectors per lane once a row exceeds 32.
template <int VEC, bool kPre>
void launch_vec(const SpmmArgs &a, cudaStream_t s) {
    const int nvec = (a.F + VEC - 1) / VEC;
    if (nvec <= 4) launch_cfg<VEC, 4, 1, kPre>(a, s);
    else if (nvec <= 8) launch_cfg<VEC, 8, 1, kPre>(a, s);
    else if (nvec <= 16) launch_cfg<VEC, 16, 1, kPre>(a, s);
    else if (nvec <= 32) launch_cfg<VEC, 32, 1, kPre>(a, s);
    else launch_cfg<VEC, 32, 2, kPre>(a, s);
}

template <bool kPre>
void launch_pre(const SpmmArgs &a, cudaStream_t s) {
    auto al = [](const void *p, int n) { return aligned_to(p, size_t(n) * 4); };
    if (a.F % 4 == 0 && a.ldz % 4 == 0 && a.ldh % 4 == 0 && al(a.Z, 4) && al(a.H, 4))
        launch_vec<4, kPre>(a, s);
    else if (a.F % 2 == 0 && a.ldz % 2 == 0 && a.ldh % 2 == 0 && al(a.Z, 2) && al(a.H, 2))
        launch_vec<2, kPre>(a, s);
    else
        launch_vec<1, kPre>(a, s);
}

}  // namespace

void launch_spmm_norm(const SpmmArgs &a, const DeviceInfo &, cudaStream_t stream) {
    if (a.N == 0) return;
    if (a.prescaled) launch_pre<true>(a, stream);
    else launch_pre<false>(a, stream);
}

bool spmm_pack_gemm_supported(int Fh, int Fo) {
    return Fh >= 1 && Fh <= 128 && Fh % 4 == 0 && Fo >= 1 && Fo <= kMaxFusedOut;
}

void launch_spmm_pack_gemm(const SpmmPackGemmArgs &a, cudaStream_t s) {
    if (a.N == 0) return;
    const int nvec = a.Fh / 4;
    const dim3 grid(unsigned((a.N + kSpmmThreads / 32 - 1) / (kSpmmThreads / 32)));
    const int words2 = (a.Fh + 63) / 64;
#define BIGCN_LAUNCH_SPG(LL)                                                                  \
    spmm_pack_gemm_kernel<LL><<<grid, kSpmmThreads, 0, s>>>(a.rowptr, a.colidx, a.N, a.nnz,   \
                                                            a.Z1, a.Fh, a.H1, a.ldh, a.wbits2, \
                                                            a.beta2, a.Fo, words2, a.Z2, a.ldz2)
    if (nvec <= 4) BIGCN_LAUNCH_SPG(4);
    else if (nvec <= 8) BIGCN_LAUNCH_SPG(8);
    else if (nvec <= 16) BIGCN_LAUNCH_SPG(16);
    else BIGCN_LAUNCH_SPG(32);
#undef BIGCN_LAUNCH_SPG
}

}  // namespace bigcn

using namespace bigcn;

namespace {
bigcn_status spmm_entry(const int64_t *rowptr, const int32_t *colidx, int64_t N, int64_t nnz,
                        const float *Z, int64_t ldz, int32_t F, float *H, int64_t ldh,
                        bool prescaled, void *stream) {
    if (N < 0 || N > int64_t(INT32_MAX) || nnz < 0 || F < 1 || ldz < F || ldh < F)
        return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldz || N > kMaxElems / ldh)) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!rowptr || !Z || !H || (nnz > 0 && !colidx)) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(rowptr, 8) || (colidx && !aligned_to(colidx, 4)) || !aligned_to(Z, 4) ||
        !aligned_to(H, 4))
        return BIGCN_ERR_MISALIGNED;
    const size_t hb = span_bytes(N, F, ldh, 4);
    if (overlaps(H, hb, Z, span_bytes(N, F, ldz, 4)) ||
        overlaps(H, hb, rowptr, size_t(N + 1) * 8) ||
        overlaps(H, hb, colidx, size_t(nnz) * 4))
        return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    SpmmArgs a{rowptr, colidx, N, nnz, Z, ldz, F, H, ldh, prescaled};
    launch_spmm_norm(a, dev, as_stream(stream));
    return launch_status();
}
}  // namespace

extern "C" bigcn_status bigcn_spmm_norm(const int64_t *rowptr, const int32_t *colidx,
                                        int64_t N, int64_t nnz, const float *Z, int64_t ldz,
                                        int32_t F, float *H, int64_t ldh, void *stream) {
    return spmm_entry(rowptr, colidx, N, nnz, Z, ldz, F, H, ldh, false, stream);
}

extern "C" bigcn_status bigcn_spmm_prescaled(const int64_t *rowptr, const int32_t *colidx,
                                             int64_t N, int64_t nnz, const float *Z,
                                             int64_t ldz, int32_t F, float *H, int64_t ldh,
                                             void *stream) {
    return spmm_entry(rowptr, colidx, N, nnz, Z, ldz, F, H, ldh, true, stream);
}
