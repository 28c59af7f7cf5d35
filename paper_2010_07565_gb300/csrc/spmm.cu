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
