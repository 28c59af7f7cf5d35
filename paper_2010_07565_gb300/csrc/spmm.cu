// Step 5 of the Bi-GCN layer forward (Wang et al., CVPR 2021, Eq. 13 with
// the operator of Eq. 1): H = D^-1/2 (A + I) D^-1/2 Z over a CSR graph.
//
// Light rows: one warp per output row. The warp is split into P = 32 / L
// groups of L lanes; each group gathers a different neighbour's row of Z,
// lane by lane in VEC-wide vectors (NV per lane), so rows narrower than a
// warp still keep all 32 lanes busy, and U such gathers are issued before any
// is consumed (U = 4, or 2 when each lane holds two vectors; twice that for
// compressed rows spread over all 32 lanes). Neighbour indices (and, unless Z is pre-scaled, their
// 1/sqrt(dhat_j)) are fetched 32 at a time, one per lane, then broadcast with
// shuffles. The self-loop that A + I adds is entry 0 of every row's list.
// Partial sums are combined across groups with xor shuffles and group 0
// writes H_i scaled by 1/sqrt(dhat_i).
//
// Heavy rows (the hubs of a power-law graph) would make one warp the
// critical path of the whole launch: a warp walks its row U * 32 / L
// neighbours per round trip. A row is heavy when it has more than
// max(32, 4 * that width, 4 * the mean degree) neighbours, i.e. when its walk
// would take several times longer than a typical row's. The first `heavy_blocks` blocks of every launch therefore scan the
// row pointers in chunks of 32 rows (so that the hubs of a small graph land
// on many blocks), skip light rows, and give each heavy row to all 8 warps of
// the block: warp w gathers the w-th eighth of the row's list, the eight
// partial rows meet in shared memory and warp 0 adds them in warp order
// (deterministic) before the same epilogue. Light warps skip heavy rows.
//
// Rows of Z come in one of three forms (template S): fp32 rows weighted by
// 1/sqrt(dhat_j) per neighbour (kDinv), fp32 rows that already carry it
// (kPre), or compressed rows (kDots16) of integer dots stored as uint16 with
// a bias of 32768, weighted per neighbour by the row scale s_j = alpha_j /
// sqrt(dhat_j) and, in the epilogue, per column by beta_f:
//   H_if = (1/sqrt(dhat_i)) * beta_f * sum_j s_j * dot_jf.
// A compressed row is half the bytes of an fp32 row, and a dot is turned
// back into a float exactly by placing its 16 bits under the exponent of
// 2^23 (one byte permute) and subtracting 2^23 + 32768. (The row scale costs
// one more random 4-byte read per neighbour, which pays off for wide rows:
// the fused forward compresses layer 1's rows, not layer 2's narrow ones.)
//
// A grid y dimension splits wide rows into column slabs of L * NV * VEC
// features. Bounds: the row range is clamped to [0, nnz] and column indices
// outside [0, N) are skipped, so a malformed CSR cannot make the kernel read
// out of bounds.
#include "launch.cuh"

namespace bigcn {
namespace {

constexpr int kSpmmThreads = 256;
constexpr int kSpmmWarps = kSpmmThreads / 32;

template <int VEC> struct Vec;
template <> struct Vec<1> {
    using T = float;
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) {
        acc[0] = fmaf(w, v, acc[0]);
    }
    static __device__ __forceinline__ T make(const float *a) { return a[0]; }
};
template <> struct Vec<2> {
    using T = float2;
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) {
        acc[0] = fmaf(w, v.x, acc[0]);
        acc[1] = fmaf(w, v.y, acc[1]);
    }
    static __device__ __forceinline__ T make(const float *a) { return make_float2(a[0], a[1]); }
};
template <> struct Vec<4> {
    using T = float4;
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) {
        acc[0] = fmaf(w, v.x, acc[0]);
        acc[1] = fmaf(w, v.y, acc[1]);
        acc[2] = fmaf(w, v.z, acc[2]);
        acc[3] = fmaf(w, v.w, acc[3]);
    }
    static __device__ __forceinline__ T make(const float *a) {
        return make_float4(a[0], a[1], a[2], a[3]);
    }
};

enum : int { kDinv = 0, kPre = 1, kDots16 = 2 };

struct SpmmParams {
    const int64_t *rowptr;
    const int32_t *colidx;
    int64_t N;
    int64_t nnz;
    const void *Z;           // float rows, or uint16 rows for kDots16
    int64_t ldz;
    int Fload;               // features gathered per row (a multiple of VEC, <= ldz)
    int F;                   // features stored per row (<= Fload)
    float *H;
    int64_t ldh;
    int heavy_blocks;        // leading blocks that take the heavy rows
    int64_t heavy_degree;    // rows with more neighbours are heavy
    bool vec_store;          // H rows start VEC-aligned: whole vectors may be stored
    const float *rowscale;   // kDots16: s_j
    const float *colscale;   // kDots16: beta_f
    int32_t *pred;           // nullable: argmax of each output row (one column slab only)
    // Aggregator (kAggGcn, kAggMean, kAggSage). kAggSage: Z (or the dots)
    // holds the neighbour half of each row and Zs the self half (same row
    // stride), with colscale_s the self half's column scales (kDots16).
    int agg = 0;
    const void *Zs = nullptr;
    const float *colscale_s = nullptr;
    int64_t ncols = 0;       // rows of Z (column indices must lie below); N when 0
    const float *values = nullptr;   // kAggWeighted: a_ij per CSR entry
    const float *dinv = nullptr;     // kAggWeighted: 1/sqrt(dhat) per node
};

// How a lane loads VEC consecutive entries of a row of Z and adds them,
// weighted, into its accumulators.
template <int VEC, int S>
struct RowSrc {
    using T = typename Vec<VEC>::T;
    static __device__ __forceinline__ T load(const void *Z, int64_t row, int64_t ldz, int f) {
        return __ldg(reinterpret_cast<const T *>(static_cast<const float *>(Z) + row * ldz + f));
    }
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) {
        Vec<VEC>::fma(acc, v, w);
    }
};

// A dot stored as uint16 with a bias of 32768, back to an exact float.
__device__ __forceinline__ float dot16_lo(uint32_t w) {
    return __int_as_float(int(__byte_perm(w, 0x4B000000u, 0x7410))) - 8421376.0f;
}
__device__ __forceinline__ float dot16_hi(uint32_t w) {
    return __int_as_float(int(__byte_perm(w, 0x4B000000u, 0x7432))) - 8421376.0f;
}

template <>
struct RowSrc<4, kDots16> {
    using T = uint2;
    static __device__ __forceinline__ T load(const void *Z, int64_t row, int64_t ldz, int f) {
        return __ldg(reinterpret_cast<const uint2 *>(static_cast<const uint16_t *>(Z) + row * ldz + f));
    }
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) {
        acc[0] = fmaf(w, dot16_lo(v.x), acc[0]);
        acc[1] = fmaf(w, dot16_hi(v.x), acc[1]);
        acc[2] = fmaf(w, dot16_lo(v.y), acc[2]);
        acc[3] = fmaf(w, dot16_hi(v.y), acc[3]);
    }
};

// Eight dots (16 bytes) per vector: half the lanes per row of the 4-wide form,
// so a warp gathers twice the neighbours per load instruction.
template <>
struct RowSrc<8, kDots16> {
    using T = uint4;
    static __device__ __forceinline__ T load(const void *Z, int64_t row, int64_t ldz, int f) {
        return __ldg(reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(Z) + row * ldz + f));
    }
    static __device__ __forceinline__ void fma(float *acc, const T &v, float w) {
        acc[0] = fmaf(w, dot16_lo(v.x), acc[0]);
        acc[1] = fmaf(w, dot16_hi(v.x), acc[1]);
        acc[2] = fmaf(w, dot16_lo(v.y), acc[2]);
        acc[3] = fmaf(w, dot16_hi(v.y), acc[3]);
        acc[4] = fmaf(w, dot16_lo(v.z), acc[4]);
        acc[5] = fmaf(w, dot16_hi(v.z), acc[5]);
        acc[6] = fmaf(w, dot16_lo(v.w), acc[6]);
        acc[7] = fmaf(w, dot16_hi(v.w), acc[7]);
    }
};

// Row i's neighbour list: CSR entries [b, b + total - 1) plus the self-loop
// (entry 0); `first` is the first entry the aggregator sums (1 when the self
// row is added separately), `dinv` the factor applied to the sum: Eq. 1's
// 1/sqrt(dhat_i) (for a weighted A read from `wdinv`), the mean's 1/dhat_i,
// or GraphSAGE's 1/|N(i)| (0 without neighbours).
struct RowSpan {
    int64_t b;
    int64_t total;
    int64_t first;
    float dinv;
};

__device__ __forceinline__ RowSpan row_span(const int64_t *__restrict__ rowptr, int64_t nnz,
                                            int64_t i, int agg = kAggGcn,
                                            const float *wdinv = nullptr) {
    const int64_t rb = __ldg(rowptr + i), re = __ldg(rowptr + i + 1);
    const int64_t b = min(max(rb, int64_t(0)), nnz);
    const int64_t e = min(max(re, b), nnz);
    const int64_t deg = e - b;
    const float norm = agg == kAggWeighted ? __ldg(wdinv + i)
                       : agg == kAggGcn    ? inv_sqrt_degree(deg)
                       : agg == kAggMean ? 1.0f / (1.0f + float(deg))
                       : deg > 0         ? 1.0f / float(deg)
                                         : 0.0f;
    return RowSpan{b, deg + 1, agg == kAggSage ? 1 : 0, norm};
}

// Adds, into acc, the Z rows of entries [q0, q1) of row i's list (entry 0 is
// the self-loop), weighted by 1/sqrt(dhat_j) (kDinv), 1 (kPre) or s_j (kDots16),
// and for a weighted A (kAggWeighted) also by the entry's a_ij (1 for the
// self-loop), with dhat_j read from p.dinv.
template <int VEC, int L, int NV, int U, int S, int AGG = kAggGcn>
__device__ __forceinline__ void gather(const SpmmParams &p, int64_t i, int64_t b, int64_t q0,
                                       int64_t q1, int f0, float (&acc)[NV][VEC]) {
    using Src = RowSrc<VEC, S>;
    using V = typename Src::T;
    constexpr int P = 32 / L;
    const int lane = threadIdx.x & 31;
    const int g = lane / L, sl = lane % L;
    for (int64_t base = q0; base < q1; base += 32) {
        int j = -1;
        float wj = 0.0f;
        const int64_t q = base + lane;
        if (q < q1) {
            j = (q == 0) ? int(i) : __ldg(p.colidx + b + q - 1);
            if (j < 0 || j >= p.ncols) j = -1;
            if (j >= 0) {
                wj = S == kPre              ? 1.0f
                     : S == kDots16         ? __ldg(p.rowscale + j)
                     : AGG == kAggWeighted  ? __ldg(p.dinv + j)
                                            : inv_sqrt_degree(__ldg(p.rowptr + j + 1) -
                                                              __ldg(p.rowptr + j));
                if (AGG == kAggWeighted && q > 0) wj *= __ldg(p.values + b + q - 1);
            }
        }
        const int cnt = int(min(q1 - base, int64_t(32)));
        for (int t0 = 0; t0 < cnt; t0 += P * U) {
            V val[U][NV];
            float w[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int src = t0 + u * P + g;
                const int jj = __shfl_sync(kFullMask, j, src & 31);
                w[u] = __shfl_sync(kFullMask, wj, src & 31);
                const bool live = src < cnt && jj >= 0;
                if (!live) w[u] = 0.0f;
                const int64_t zrow = live ? jj : 0;
#pragma unroll
                for (int v = 0; v < NV; ++v) {
                    const int f = f0 + (v * L + sl) * VEC;
                    if (live && f < p.Fload) val[u][v] = Src::load(p.Z, zrow, p.ldz, f);
                    else val[u][v] = V{};
                }
            }
#pragma unroll
            for (int u = 0; u < U; ++u)
#pragma unroll
                for (int v = 0; v < NV; ++v) Src::fma(acc[v], val[u][v], w[u]);
        }
    }
}

template <int VEC, int L, int NV>
__device__ __forceinline__ void reduce_groups(float (&acc)[NV][VEC]) {
#pragma unroll
    for (int o = L; o < 32; o <<= 1)
#pragma unroll
        for (int v = 0; v < NV; ++v)
#pragma unroll
            for (int c = 0; c < VEC; ++c) acc[v][c] += __shfl_xor_sync(kFullMask, acc[v][c], o);
}

// Epilogue of the plain aggregation: H_i = dinv_i * acc, or for compressed
// rows H_if = dinv_i * (beta_f * acc_f) (lanes of group 0).
template <int VEC, int L, int NV, int S, int AGG = kAggGcn>
struct StoreRow {
    __device__ __forceinline__ void prologue() const {}
    __device__ __forceinline__ void operator()(const SpmmParams &p, int64_t i, float dinv,
                                               int f0, float (&acc)[NV][VEC]) const {
        const int lane = threadIdx.x & 31;
        if (lane / L != 0) return;
        const int sl = lane % L;
        float bestv = 0.0f;
        int best = -1;              // this lane's argmax candidate (lowest index on ties)
#pragma unroll
        for (int v = 0; v < NV; ++v) {
            const int f = f0 + (v * L + sl) * VEC;
            float o[VEC];
#pragma unroll
            for (int c = 0; c < VEC; ++c) {
                if (S == kDots16)
                    o[c] = f + c < p.F ? dinv * (__ldg(p.colscale + f + c) * acc[v][c]) : 0.0f;
                else
                    o[c] = acc[v][c] * dinv;
            }
            if constexpr (AGG == kAggSage) {   // GraphSAGE: the node's own (self-half) product
                const float si = S == kDots16 ? __ldg(p.rowscale + i) : 0.0f;
#pragma unroll
                for (int c = 0; c < VEC; ++c) {
                    if (f + c >= p.F) continue;
                    if (S == kDots16) {
                        const uint32_t d = __ldg(static_cast<const uint16_t *>(p.Zs) + i * p.ldz + f + c);
                        o[c] += si * (__ldg(p.colscale_s + f + c) * (float(d) - 32768.0f));
                    } else {
                        o[c] += __ldg(static_cast<const float *>(p.Zs) + i * p.ldz + f + c);
                    }
                }
            }
            if (p.pred != nullptr) {
#pragma unroll
                for (int c = 0; c < VEC; ++c)
                    if (f + c < p.F && (best < 0 || o[c] > bestv)) {
                        bestv = o[c];
                        best = f + c;
                    }
            }
            float *h = p.H + i * p.ldh + f;
            if (p.vec_store && f + VEC <= p.F) {
                if constexpr (VEC == 8) {
                    reinterpret_cast<float4 *>(h)[0] = make_float4(o[0], o[1], o[2], o[3]);
                    reinterpret_cast<float4 *>(h)[1] = make_float4(o[4], o[5], o[6], o[7]);
                } else {
                    *reinterpret_cast<typename Vec<VEC>::T *>(h) = Vec<VEC>::make(o);
                }
            } else {
#pragma unroll
                for (int c = 0; c < VEC; ++c)
                    if (f + c < p.F) h[c] = o[c];
            }
        }
        if (p.pred != nullptr) {    // the row's argmax over the L lanes of group 0
            const unsigned gm = L == 32 ? kFullMask : (1u << L) - 1u;
#pragma unroll
            for (int o = L / 2; o > 0; o >>= 1) {
                const float ov = __shfl_xor_sync(gm, bestv, o);
                const int oi = __shfl_xor_sync(gm, best, o);
                if (oi >= 0 && (best < 0 || ov > bestv || (ov == bestv && oi < best))) {
                    bestv = ov;
                    best = oi;
                }
            }
            if (sl == 0) p.pred[i] = best;
        }
    }
};

// Argmax of each row of H (F columns, row stride ldh; lowest index on ties),
// one warp per row: for outputs too wide for the aggregation's epilogue.
__global__ void __launch_bounds__(kSpmmThreads)
argmax_rows_kernel(const float *__restrict__ H, int64_t N, int F, int64_t ldh,
                   int32_t *__restrict__ pred) {
    grid_dependency_wait();     // H is the previous kernel's output
    const int lane = threadIdx.x & 31;
    const int64_t i = int64_t(blockIdx.x) * kSpmmWarps + (threadIdx.x >> 5);
    if (i >= N) return;
    float bestv = 0.0f;
    int best = -1;
    for (int f = lane; f < F; f += 32) {
        const float v = __ldg(H + i * ldh + f);
        if (best < 0 || v > bestv) {
            bestv = v;
            best = f;
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float ov = __shfl_xor_sync(kFullMask, bestv, o);
        const int oi = __shfl_xor_sync(kFullMask, best, o);
        if (oi >= 0 && (best < 0 || ov > bestv || (ov == bestv && oi < best))) {
            bestv = ov;
            best = oi;
        }
    }
    if (lane == 0) pred[i] = best;
}

template <int VEC, int L, int NV, int U, int S, class Epi, int AGG = kAggGcn>
__device__ __forceinline__ void light_rows(const SpmmParams &p, const Epi &epi, int f0) {
    const int warp = threadIdx.x >> 5;
    const int64_t i = int64_t(blockIdx.x - p.heavy_blocks) * kSpmmWarps + warp;
    if (i >= p.N) return;
    const RowSpan sp = row_span(p.rowptr, p.nnz, i, AGG, p.dinv);
    if (p.heavy_blocks > 0 && sp.total - 1 > p.heavy_degree) return;   // a heavy block's row
    float acc[NV][VEC];
#pragma unroll
    for (int v = 0; v < NV; ++v)
#pragma unroll
        for (int c = 0; c < VEC; ++c) acc[v][c] = 0.0f;
    gather<VEC, L, NV, U, S, AGG>(p, i, sp.b, sp.first, sp.total, f0, acc);
    reduce_groups<VEC, L, NV>(acc);
    epi(p, i, sp.dinv, f0, acc);
}

template <int VEC, int L, int NV, int U, int S, class Epi, int AGG = kAggGcn>
__device__ __forceinline__ void heavy_rows(const SpmmParams &p, const Epi &epi, int f0,
                                           float *part) {
    constexpr int SLAB = L * NV * VEC;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = lane / L, sl = lane % L;
    // Chunks of 32 rows: every warp takes the same ballot over the chunk's
    // row lengths, so the loop below is uniform over the block.
    for (int64_t base = int64_t(blockIdx.x) * 32; base < p.N;
         base += int64_t(p.heavy_blocks) * 32) {
        const int64_t r = base + lane;
        bool heavy = false;
        if (r < p.N) heavy = row_span(p.rowptr, p.nnz, r).total - 1 > p.heavy_degree;
        unsigned mm = __ballot_sync(kFullMask, heavy);
        while (mm != 0u) {
            const int bit = __ffs(mm) - 1;
            mm &= mm - 1u;
            const int64_t i = base + bit;
            const RowSpan sp = row_span(p.rowptr, p.nnz, i, AGG, p.dinv);
            float acc[NV][VEC];
#pragma unroll
            for (int v = 0; v < NV; ++v)
#pragma unroll
                for (int c = 0; c < VEC; ++c) acc[v][c] = 0.0f;
            const int64_t span = sp.total - sp.first;
            const int64_t q0 = sp.first + span * warp / kSpmmWarps;
            const int64_t q1 = sp.first + span * (warp + 1) / kSpmmWarps;
            gather<VEC, L, NV, U, S, AGG>(p, i, sp.b, q0, q1, f0, acc);
            reduce_groups<VEC, L, NV>(acc);
            if (g == 0) {
#pragma unroll
                for (int v = 0; v < NV; ++v)
#pragma unroll
                    for (int c = 0; c < VEC; ++c)
                        part[warp * SLAB + (v * L + sl) * VEC + c] = acc[v][c];
            }
            __syncthreads();
            if (warp == 0) {
#pragma unroll
                for (int v = 0; v < NV; ++v)
#pragma unroll
                    for (int c = 0; c < VEC; ++c) {
                        float t = 0.0f;
                        if (g == 0)
                            for (int q = 0; q < kSpmmWarps; ++q)
                                t += part[q * SLAB + (v * L + sl) * VEC + c];
                        acc[v][c] = t;
                    }
                epi(p, i, sp.dinv, f0, acc);
            }
            __syncthreads();    // part[] is rewritten by the next heavy row
        }
    }
}

template <int VEC, int L, int NV, int U, int S, int AGG>
__global__ void __launch_bounds__(kSpmmThreads, 4)
spmm_norm_kernel(SpmmParams p) {
    constexpr int SLAB = L * NV * VEC;
    __shared__ float part[kSpmmWarps * SLAB];
    grid_dependency_wait();     // Z is the output of the previous kernel
    const int f0 = blockIdx.y * SLAB;
    using Epi = StoreRow<VEC, L, NV, S, AGG>;
    Epi epi;
    if (int(blockIdx.x) < p.heavy_blocks)
        heavy_rows<VEC, L, NV, U, S, Epi, AGG>(p, epi, f0, part);
    else
        light_rows<VEC, L, NV, U, S, Epi, AGG>(p, epi, f0);
}

// ---------------------------------------------------------------------------
// Layer-1 aggregation fused with layer 2's binarization and product.
//
// Each row's H1_i is computed exactly as above (one vector per lane), from
// layer 1's Z' as pre-scaled fp32 rows (VEC = 4) or, compressed, as uint16
// dots weighted by s1_j with beta1 applied per column (VEC = 8 when the row
// stride is a multiple of 8, else 4). Then, without writing
// H1 (unless asked to), layer 2's steps run on the row while it is in
// registers: the signs of its Fh <= 128 features become one or two 64-bit
// words (VEC ballots, one per vector component, spread into place), the row
// scale alpha2_i = mean |H1_i| is one warp reduction, and the XNOR popcount
// against the (shared-memory) packed columns of W2 gives the dots of Eq. 11.
// The result is written as Z2'_ij = (alpha2_i * dinv_i) * (beta2_j * dot_ij),
// the expression the product's degree-scaled epilogue evaluates; columns of
// Z2' from Fo up to its row stride are written as zeros, so the layer-2
// aggregation can gather whole 4-wide vectors.

// Spreads 16 bits so that bit i lands on bit 4i of a 64-bit word.
__device__ __forceinline__ uint64_t spread16by4(uint32_t x) {
    uint64_t v = x & 0xFFFFu;
    v = (v | (v << 24)) & 0x000000FF000000FFull;
    v = (v | (v << 12)) & 0x000F000F000F000Full;
    v = (v | (v << 6)) & 0x0303030303030303ull;
    v = (v | (v << 3)) & 0x1111111111111111ull;
    return v;
}

// Spreads 8 bits so that bit i lands on bit 8i of a 64-bit word.
__device__ __forceinline__ uint64_t spread8by8(uint32_t x) {
    uint64_t v = x & 0xFFu;
    v = (v | (v << 28)) & 0x0000000F0000000Full;
    v = (v | (v << 14)) & 0x0003000300030003ull;
    v = (v | (v << 7)) & 0x0101010101010101ull;
    return v;
}

struct FusedLayer2 {
    float *H1;
    int64_t ldh;
    const uint64_t *sW;       // shared: Fo x words2 packed columns of W2
    const float *sBeta1;      // shared: Fh (compressed input only)
    const float *sBeta2;      // shared: Fo
    int Fo;
    int words2;
    float *Z2;
    int64_t ldz2;
};

template <int VEC, int L, int S>
struct PackGemmRow {
    FusedLayer2 f;
    __device__ __forceinline__ void operator()(const SpmmParams &p, int64_t i, float dinv,
                                               int, float (&acc)[1][VEC]) const {
        const int lane = threadIdx.x & 31;
        const int g = lane / L, sl = lane % L;
        const int fb = sl * VEC;
        const int Fh = p.F;
        float h[VEC];
#pragma unroll
        for (int c = 0; c < VEC; ++c) {
            if (S == kDots16)
                h[c] = fb + c < Fh ? dinv * (f.sBeta1[fb + c] * acc[0][c]) : 0.0f;
            else
                h[c] = acc[0][c] * dinv;
        }
        if (f.H1 != nullptr && g == 0) {
#pragma unroll
            for (int c = 0; c < VEC; ++c)
                if (fb + c < Fh) f.H1[i * f.ldh + fb + c] = h[c];
        }
        // Layer 2, Eqs. 7-8: signs of H1_i packed LSB-first, and its mean |.|.
        // Ballot c holds component c of every lane's vector: feature VEC l + c.
        uint64_t w0 = 0, w1 = 0;
        float l1 = 0.0f;
#pragma unroll
        for (int c = 0; c < VEC; ++c) {
            const bool in = g == 0 && fb + c < Fh;
            const unsigned m = __ballot_sync(kFullMask, in && h[c] >= 0.0f);
            if (VEC == 4) {
                w0 |= spread16by4(m) << c;
                w1 |= spread16by4(m >> 16) << c;
            } else {
                w0 |= spread8by8(m) << c;
                w1 |= spread8by8(m >> 8) << c;
            }
            l1 += in ? fabsf(h[c]) : 0.0f;
        }
        l1 = warp_sum(l1);
        const float a = (l1 / float(Fh)) * dinv;
        // Layer 2, Eqs. 11-12, pre-scaled by this row's 1/sqrt(dhat_i).
        for (int jo = lane; jo < f.ldz2; jo += 32) {
            float z = 0.0f;
            if (jo < f.Fo) {
                int mism = __popcll(w0 ^ f.sW[jo * f.words2]);
                if (f.words2 > 1) mism += __popcll(w1 ^ f.sW[jo * f.words2 + 1]);
                z = a * (f.sBeta2[jo] * float(Fh - 2 * mism));
            }
            f.Z2[i * f.ldz2 + jo] = z;
        }
    }
};

template <int VEC, int L, int S>
__global__ void __launch_bounds__(kSpmmThreads, 3)
spmm_pack_gemm_kernel(SpmmParams p, FusedLayer2 f, const uint64_t *__restrict__ wbits2,
                      const float *__restrict__ beta1, const float *__restrict__ beta2) {
    constexpr int SLAB = L * VEC;
    constexpr int U = S == kDots16 && VEC == 4 && L == 32 ? 8 : 4;
    __shared__ float part[kSpmmWarps * SLAB];
    __shared__ uint64_t sW[kMaxFusedOut * 2];
    __shared__ float sBeta1[128];
    __shared__ float sBeta2[kMaxFusedOut];
    grid_dependency_wait();     // layer 1's Z' and the packed W2 come from earlier kernels
    for (int q = threadIdx.x; q < f.Fo * f.words2; q += kSpmmThreads) sW[q] = __ldg(wbits2 + q);
    for (int q = threadIdx.x; q < f.Fo; q += kSpmmThreads) sBeta2[q] = __ldg(beta2 + q);
    if (S == kDots16)
        for (int q = threadIdx.x; q < p.F; q += kSpmmThreads) sBeta1[q] = __ldg(beta1 + q);
    __syncthreads();
    f.sW = sW;
    f.sBeta1 = sBeta1;
    f.sBeta2 = sBeta2;
    PackGemmRow<VEC, L, S> epi{f};
    if (int(blockIdx.x) < p.heavy_blocks)
        heavy_rows<VEC, L, 1, U, S>(p, epi, 0, part);
    else
        light_rows<VEC, L, 1, U, S>(p, epi, 0);
}

// Leading blocks that look for heavy rows: up to two per SM, one per 32 rows.
int heavy_block_count(int64_t N, const DeviceInfo &dev) {
    const int64_t chunks = (N + 31) / 32;
    const int64_t cap = 2 * int64_t(dev.sm_count);
    return int(chunks < cap ? chunks : cap);
}

// The heavy-row threshold for a walk of `per_iter` neighbours per round trip.
int64_t heavy_degree(int64_t N, int64_t nnz, int per_iter) {
    const int64_t mean = N > 0 ? nnz / N : 0;
    int64_t h = 4 * int64_t(per_iter);
    if (4 * mean > h) h = 4 * mean;
    return h > 32 ? h : 32;
}

// Eight dots per lane halve the gather instructions per neighbour but double
// the per-row reduction and epilogue work: worth it from a mean degree of 8.
bool wide_dots(int64_t N, int64_t nnz) { return N > 0 && nnz >= 8 * N; }

template <int VEC, int L, int NV, int S, int AGG>
void launch_cfg(const SpmmArgs &a, const DeviceInfo &dev, int Fload, cudaStream_t s, bool pdl) {
    constexpr int SLAB = L * NV * VEC;
    // Rows in flight per group. A compressed row costs half the registers, so
    // where a warp holds only a few rows at a time (one row across all 32
    // lanes) it takes twice as many.
    constexpr int U = VEC == 8 ? (NV == 1 ? 4 : 2)
                               : (S == kDots16 && L == 32 ? 2 : 1) * (NV == 1 ? 4 : 2);
    constexpr int kStoreVec = VEC < 4 ? VEC : 4;    // 8-wide rows are stored as two float4
    const bool vec_store = a.ldh % kStoreVec == 0 && aligned_to(a.H, size_t(kStoreVec) * 4);
    const void *Z = S == kDots16 ? static_cast<const void *>(a.D16) : a.Z;
    const bool one_slab = a.F <= SLAB;
    SpmmParams p{a.rowptr, a.colidx, a.N, a.nnz, Z, a.ldz, Fload, a.F, a.H, a.ldh,
                 heavy_block_count(a.N, dev), heavy_degree(a.N, a.nnz, (32 / L) * U), vec_store,
                 a.rowscale, a.colscale, one_slab ? a.pred : nullptr, a.agg, a.Zs,
                 a.colscale_s, a.ncols > 0 ? a.ncols : a.N, a.values, a.dinv};
    dim3 grid(unsigned(p.heavy_blocks + (a.N + kSpmmWarps - 1) / kSpmmWarps),
              unsigned((a.F + SLAB - 1) / SLAB));
    launch_kernel(spmm_norm_kernel<VEC, L, NV, U, S, AGG>, grid, dim3(kSpmmThreads), 0, s, pdl,
                  dim3(1, 1, 1), p);
    if (a.pred != nullptr && !one_slab)
        launch_kernel(argmax_rows_kernel, dim3(unsigned((a.N + kSpmmWarps - 1) / kSpmmWarps)),
                      dim3(kSpmmThreads), 0, s, pdl, dim3(1, 1, 1), static_cast<const float *>(a.H),
                      a.N, a.F, a.ldh, a.pred);
}

// Lanes per neighbour L = the power of two >= the row's vector count (at
// least 4, at most 32); NV = 2 vectors per lane once a row exceeds 32.
// fp32 rows of Z larger than this in all are gathered in column slabs of at
// most 16 vectors per lane group: the slabs (grid y) run mostly one after the
// other, so each keeps only its share of Z in L2 (measured on 119 MB of
// 128-wide rows: 7.17 -> 6.49 ms; 16-bit dots, at 8 per lane, lose by it).
constexpr int64_t kSlabL2Bytes = int64_t(64) << 20;

template <int VEC, int S, int AGG = kAggGcn>
void launch_vec(const SpmmArgs &a, const DeviceInfo &dev, int Fload, cudaStream_t s, bool pdl) {
    const int nvec = Fload / VEC;
    const int64_t zbytes = S == kDots16 ? 0 : a.N * int64_t(Fload) * 4;
    if (nvec <= 4) launch_cfg<VEC, 4, 1, S, AGG>(a, dev, Fload, s, pdl);
    else if (nvec <= 8) launch_cfg<VEC, 8, 1, S, AGG>(a, dev, Fload, s, pdl);
    else if (nvec <= 16 || zbytes > kSlabL2Bytes) launch_cfg<VEC, 16, 1, S, AGG>(a, dev, Fload, s, pdl);
    else if (nvec <= 32) launch_cfg<VEC, 32, 1, S, AGG>(a, dev, Fload, s, pdl);
    else launch_cfg<VEC, 32, 2, S, AGG>(a, dev, Fload, s, pdl);
}

template <int S, int AGG = kAggGcn>
void launch_src(const SpmmArgs &a, const DeviceInfo &dev, cudaStream_t s, bool pdl) {
    auto al = [](const void *p, int n) { return aligned_to(p, size_t(n) * 4); };
    // Gathers may read whole vectors past F when the padding up to a multiple
    // of 4 lies inside the row stride and is declared readable (a.z_pad4).
    const int F4 = (a.F + 3) / 4 * 4;
    if (a.ldz % 4 == 0 && al(a.Z, 4) && (a.F % 4 == 0 || (a.z_pad4 && F4 <= a.ldz)))
        launch_vec<4, S, AGG>(a, dev, F4, s, pdl);
    else if (a.F % 2 == 0 && a.ldz % 2 == 0 && a.ldh % 2 == 0 && al(a.Z, 2) && al(a.H, 2))
        launch_vec<2, S, AGG>(a, dev, a.F, s, pdl);
    else
        launch_vec<1, S, AGG>(a, dev, a.F, s, pdl);
}

// Inductive aggregators: fp32 rows without a per-neighbour factor, or dots.
template <int AGG>
void launch_inductive(const SpmmArgs &a, const DeviceInfo &dev, cudaStream_t stream, bool pdl) {
    if (a.D16 != nullptr) {
        if (a.ldz % 8 == 0 && aligned_to(a.D16, 16) && wide_dots(a.N, a.nnz))
            launch_vec<8, kDots16, AGG>(a, dev, (a.F + 7) / 8 * 8, stream, pdl);
        else
            launch_vec<4, kDots16, AGG>(a, dev, (a.F + 3) / 4 * 4, stream, pdl);
        return;
    }
    launch_src<kPre, AGG>(a, dev, stream, pdl);
}

// A weighted A: dots with their row scale, or plain fp32 rows whose source
// factor dinv_j is read per neighbour (kDinv).
void launch_weighted(const SpmmArgs &a, const DeviceInfo &dev, cudaStream_t stream, bool pdl) {
    if (a.D16 != nullptr) {
        if (a.ldz % 8 == 0 && aligned_to(a.D16, 16) && wide_dots(a.N, a.nnz))
            launch_vec<8, kDots16, kAggWeighted>(a, dev, (a.F + 7) / 8 * 8, stream, pdl);
        else
            launch_vec<4, kDots16, kAggWeighted>(a, dev, (a.F + 3) / 4 * 4, stream, pdl);
        return;
    }
    launch_src<kDinv, kAggWeighted>(a, dev, stream, pdl);
}

}  // namespace

void launch_spmm_norm(const SpmmArgs &a, const DeviceInfo &dev, cudaStream_t stream, bool pdl) {
    if (a.N == 0) return;
    if (a.agg == kAggMean) return launch_inductive<kAggMean>(a, dev, stream, pdl);
    if (a.agg == kAggSage) return launch_inductive<kAggSage>(a, dev, stream, pdl);
    if (a.agg == kAggWeighted) return launch_weighted(a, dev, stream, pdl);
    if (a.D16 != nullptr) {
        // Compressed rows: eight dots (16 bytes) per vector when the row
        // stride and base allow and rows are long, else four (8 bytes);
        // padding columns up to the stride hold a zero dot.
        if (a.ldz % 8 == 0 && aligned_to(a.D16, 16) && wide_dots(a.N, a.nnz))
            launch_vec<8, kDots16>(a, dev, (a.F + 7) / 8 * 8, stream, pdl);
        else
            launch_vec<4, kDots16>(a, dev, (a.F + 3) / 4 * 4, stream, pdl);
        return;
    }
    if (a.prescaled) launch_src<kPre>(a, dev, stream, pdl);
    else launch_src<kDinv>(a, dev, stream, pdl);
}

bool spmm_pack_gemm_supported(int Fh, int Fo) {
    return Fh >= 1 && Fh <= 128 && Fh % 4 == 0 && Fo >= 1 && Fo <= kMaxFusedOut;
}

void launch_spmm_pack_gemm(const SpmmPackGemmArgs &a, const DeviceInfo &dev, cudaStream_t s,
                           bool pdl) {
    if (a.N == 0) return;
    const bool c16 = a.D1 != nullptr;
    // Compressed rows take eight dots per lane when their stride allows and
    // the rows are long enough to repay it.
    const int VEC = c16 && a.ldz1 % 8 == 0 && aligned_to(a.D1, 16) && wide_dots(a.N, a.nnz) ? 8 : 4;
    const int Fload = (a.Fh + VEC - 1) / VEC * VEC;
    const int nvec = Fload / VEC;
    int L = 4;
    while (L < 32 && L < nvec) L *= 2;
    const int U = c16 && VEC == 4 && L == 32 ? 8 : 4;
    const void *Z1 = c16 ? static_cast<const void *>(a.D1) : static_cast<const void *>(a.Z1);
    SpmmParams p{a.rowptr, a.colidx, a.N, a.nnz, Z1, c16 ? a.ldz1 : a.Fh, Fload, a.Fh, nullptr, 0,
                 heavy_block_count(a.N, dev), heavy_degree(a.N, a.nnz, (32 / L) * U), false,
                 a.s1, nullptr, nullptr};
    p.ncols = a.N;
    FusedLayer2 f{a.H1, a.ldh, nullptr, nullptr, nullptr, a.Fo, (a.Fh + 63) / 64, a.Z2, a.ldz2};
    const dim3 grid(unsigned(p.heavy_blocks + (a.N + kSpmmWarps - 1) / kSpmmWarps));
    const dim3 one(1, 1, 1), block(kSpmmThreads);
    auto run = [&](auto kernel) {
        launch_kernel(kernel, grid, block, 0, s, pdl, one, p, f, a.wbits2, a.beta1, a.beta2);
    };
    if (c16 && VEC == 8) {
        if (L == 4) run(spmm_pack_gemm_kernel<8, 4, kDots16>);
        else if (L == 8) run(spmm_pack_gemm_kernel<8, 8, kDots16>);
        else run(spmm_pack_gemm_kernel<8, 16, kDots16>);
    } else if (c16) {
        if (L == 4) run(spmm_pack_gemm_kernel<4, 4, kDots16>);
        else if (L == 8) run(spmm_pack_gemm_kernel<4, 8, kDots16>);
        else if (L == 16) run(spmm_pack_gemm_kernel<4, 16, kDots16>);
        else run(spmm_pack_gemm_kernel<4, 32, kDots16>);
    } else {
        if (L == 4) run(spmm_pack_gemm_kernel<4, 4, kPre>);
        else if (L == 8) run(spmm_pack_gemm_kernel<4, 8, kPre>);
        else if (L == 16) run(spmm_pack_gemm_kernel<4, 16, kPre>);
        else run(spmm_pack_gemm_kernel<4, 32, kPre>);
    }
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
    SpmmArgs a{rowptr, colidx, N, nnz, Z, ldz, F, H, ldh, prescaled, false};
    launch_spmm_norm(a, dev, as_stream(stream));
    return launch_status();
}
}  // namespace

extern "C" bigcn_status bigcn_spmm_prescaled_rows(const int64_t *rowptr, const int32_t *colidx,
                                                  int64_t n_rows, int64_t n_cols, int64_t nnz,
                                                  const float *Z, int64_t ldz, int32_t F,
                                                  float *H, int64_t ldh, void *stream) {
    if (n_rows < 0 || n_rows > int64_t(INT32_MAX) || n_cols < n_rows ||
        n_cols > int64_t(INT32_MAX) || nnz < 0 || F < 1 || ldz < F || ldh < F)
        return BIGCN_ERR_INVALID_ARG;
    if (n_rows > 0 && (n_cols > kMaxElems / ldz || n_rows > kMaxElems / ldh))
        return BIGCN_ERR_INVALID_ARG;
    if (n_rows == 0) return BIGCN_OK;
    if (!rowptr || !Z || !H || (nnz > 0 && !colidx)) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(rowptr, 8) || (colidx && !aligned_to(colidx, 4)) || !aligned_to(Z, 4) ||
        !aligned_to(H, 4))
        return BIGCN_ERR_MISALIGNED;
    const size_t hb = span_bytes(n_rows, F, ldh, 4);
    if (overlaps(H, hb, Z, span_bytes(n_cols, F, ldz, 4)) ||
        overlaps(H, hb, rowptr, size_t(n_rows + 1) * 8) ||
        overlaps(H, hb, colidx, size_t(nnz) * 4))
        return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    SpmmArgs a{rowptr, colidx, n_rows, nnz, Z, ldz, F, H, ldh, true, false};
    a.ncols = n_cols;
    launch_spmm_norm(a, dev, as_stream(stream));
    return launch_status();
}

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
