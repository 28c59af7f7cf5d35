// Ablation variants of step 4 (Sec. 6.3, the transductive table's rows
// "binarize weights only" and "binarize features only"): one operand of
// Eq. 11's product keeps its real fp32 values, the other is binarized.
//
//   weights binarized:  Z[i,j] = beta_j  * sum_k y_ik * s(b_jk)   (A real)
//   features binarized: Z[i,j] = alpha_i * sum_k s(a_ik) * W_kj   (B real)
//
// Both are dense contractions and run on the tcgen05 tensor cores (kind::f16,
// bf16 operands, fp32 accumulators in tensor memory). A sign +-1 is exact in
// bf16; the real operand v is split into three bf16 parts
//   hi = bf16(v), mid = bf16(v - hi), lo = bf16(v - hi - mid)
// (each subtraction exact in fp32), so |v - (hi + mid + lo)| <= 2^-24 |v|
// roughly, and the three products are accumulated into the same fp32 tile:
// the result is an fp32-accurate evaluation of the sum.
//
// CTA tile: 128 node rows (UMMA M) x NT output columns (UMMA N), k-blocks of
// 64 elements (one 128-byte bf16 row of a 128B-swizzled K-major operand, and
// exactly one 64-bit word of packed signs). All 256 threads build a stage --
// the real operand's three part tiles and the sign tile -- while the tensor
// core works on the previous one; each thread loads the next k-block's inputs
// into registers before the barrier. A stage is reused only after the
// tcgen05.commit of the MMAs that read it has arrived on its mbarrier; every
// such wait is bounded (a wait that runs out is counted, the CTA writes
// nothing and returns).
//
// Few row tiles: the k-blocks are split between the KS CTAs of a cluster
// (KS <= 8). Each CTA moves its partial tile from tensor memory to its shared
// memory; after a cluster barrier CTA r adds the KS partials of rows
// [128 r / KS, 128 (r + 1) / KS) in rank order through distributed shared
// memory, scales and stores them; a second cluster barrier keeps every CTA's
// shared memory alive until its peers have read it.
//
// Epilogue scale: weights binarized, Z = rs_i * (beta_j * acc); features
// binarized, Z = rs_i * acc with rs_i = alpha_i; with the degree form (rowptr
// given) rs_i also carries 1/sqrt(dhat_i).
#include <cuda_bf16.h>

#include "async.cuh"
#include "launch.cuh"
#include "tc.cuh"

namespace bigcn {

namespace {

__device__ unsigned int g_mix_timeouts;

constexpr int kMixThreads = 256;
constexpr int kMixK = 64;        // elements per k-block
constexpr int kParts = 3;        // bf16 parts of the real operand
constexpr int kMaxSplit = 8;     // CTAs of a cluster sharing one tile's k-blocks

// Instruction descriptor: BF16 x BF16 -> F32, both K-major, M = 128, N = n.
__host__ __device__ constexpr uint32_t bf16_idesc(int n) {
    return (1u << 4) | (1u << 7) | (1u << 10) | (uint32_t(n >> 3) << 17) |
           (uint32_t(kUmmaM >> 4) << 24);
}

__device__ __forceinline__ void mma_bf16(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n.reg .pred p;\n"
        "setp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate));
}

// Eight signs (bits 0..7 of `byte`) as eight bf16 values, +1 (0x3F80) for a
// set bit and -1 (0xBF80) otherwise, element e in the e-th 16-bit half.
__device__ __forceinline__ uint4 signs8_to_bf16(uint32_t byte) {
    uint32_t u[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        const uint32_t b = byte >> (2 * w);
        u[w] = 0xBF80BF80u ^ ((b & 1u) << 15) ^ ((b & 2u) << 30);
    }
    return make_uint4(u[0], u[1], u[2], u[3]);
}

// The three bf16 parts of v, as 16-bit patterns.
__device__ __forceinline__ void split3(float v, uint32_t &hi, uint32_t &mid, uint32_t &lo) {
    const __nv_bfloat16 h = __float2bfloat16_rn(v);
    const float r1 = v - __bfloat162float(h);
    const __nv_bfloat16 m = __float2bfloat16_rn(r1);
    const float r2 = r1 - __bfloat162float(m);
    const __nv_bfloat16 l = __float2bfloat16_rn(r2);
    hi = __bfloat16_as_ushort(h);
    mid = __bfloat16_as_ushort(m);
    lo = __bfloat16_as_ushort(l);
}

__device__ __forceinline__ uint32_t cluster_rank() {
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

__device__ __forceinline__ void cluster_sync() {
    asm volatile("barrier.cluster.arrive.release.aligned;\n"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t map_to_rank(uint32_t saddr, uint32_t rank) {
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(saddr), "r"(rank));
    return r;
}

__device__ __forceinline__ float4 ld_cluster_f4(uint32_t addr) {
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(addr)
                 : "memory");
    return v;
}

__device__ __forceinline__ uint32_t ld_cluster_u32(uint32_t addr) {
    uint32_t v;
    asm volatile("ld.shared::cluster.u32 %0, [%1];" : "=r"(v) : "r"(addr) : "memory");
    return v;
}

struct MixParams {
    // A real (weights binarized): X, centring, packed weight columns.
    const float *X;
    int64_t ldx;
    const float *scale;
    const float *shift;
    const uint64_t *b_bits;
    const float *beta;
    // B real (features binarized): packed node rows and the parts of W,
    // wparts[p][j][k] (p < 3, j < F, k < words * 64; zero at k >= K).
    const uint64_t *a_bits;
    const float *alpha;
    const uint16_t *wparts;
    int64_t N;
    int K;
    int F;
    int words;
    float *Z;
    int64_t ldz;
    const int64_t *rowptr;   // nullable: rows scaled by 1/sqrt(dhat_i)
    int split;               // KS: CTAs of a cluster sharing a tile's k-blocks
};

template <int NT, bool kRealA>
struct MixShape {
    static constexpr int kTileA = kUmmaM * 128;           // bytes of one 128-row bf16 tile
    static constexpr int kTileB = NT * 128;
    static constexpr int kStage = kRealA ? kParts * kTileA + kTileB : kTileA + kParts * kTileB;
    static constexpr int kStages = (kStage <= 48 * 1024) ? 4 : (kStage <= 64 * 1024 ? 3 : 2);
    static constexpr int kRedStride = NT + 4;              // floats per partial row
    static constexpr size_t kSmem = 1024 + size_t(kStages) * kStage;
    static_assert(size_t(kUmmaM) * kRedStride * 4 <= size_t(kStages) * kStage,
                  "the partial tile reuses the stage buffers");
};

template <int NT, bool kRealA>
__global__ void __launch_bounds__(kMixThreads)
mixed_gemm_tc_kernel(const MixParams p) {
    using S = MixShape<NT, kRealA>;
    constexpr int kStages = S::kStages;
    constexpr int kBRows = NT / 32;                        // B rows per thread
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bars[kStages];
    __shared__ uint32_t tmem_base;
    __shared__ uint32_t s_ok;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int KS = p.split;
    const int rank = KS > 1 ? int(cluster_rank()) : 0;
    const int64_t m0 = int64_t(blockIdx.x / KS) * kUmmaM;
    const int n0 = blockIdx.y * NT;
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t tile0 = (raw + 1023u) & ~1023u;
    unsigned char *tiles = smem_raw + (tile0 - raw);

    // This CTA's k-blocks.
    const int KB = p.words;
    const int per = (KB + KS - 1) / KS;
    const int kb0 = min(KB, rank * per), kb1 = min(KB, kb0 + per);

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_addr(&tmem_base)),
                     "r"(NT));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) mbar_init(smem_addr(&bars[s]), 1);
        mbar_fence_init();
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base;
    grid_dependency_wait();     // packed operands and parts come from earlier kernels

    // Thread t builds 16-byte chunk c = t & 7 (elements 8c .. 8c + 7 of the
    // k-block) of rows r0 + 32 q of each tile.
    const int c = tid & 7, r0 = tid >> 3;
    const bool vec_x = kRealA && (p.ldx & 3) == 0 && (reinterpret_cast<uintptr_t>(p.X) & 15) == 0;

    float xv[kRealA ? 4 : 1][8];       // A real: 4 rows x 8 elements
    float sv[8], tv[8];                // centring of those elements
    uint64_t wsign[kRealA ? kBRows : 4];   // packed words of the sign tile's rows
    uint4 wpart[kRealA ? 1 : kBRows][kParts];

    auto load = [&](int kb) {
        const int k = kb * kMixK + 8 * c;
        if constexpr (kRealA) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int64_t row = m0 + r0 + 32 * q;
                const float *x = p.X + row * p.ldx + k;
                if (row < p.N && vec_x && k + 8 <= p.K) {
                    const float4 a = __ldg(reinterpret_cast<const float4 *>(x));
                    const float4 b = __ldg(reinterpret_cast<const float4 *>(x) + 1);
                    xv[q][0] = a.x; xv[q][1] = a.y; xv[q][2] = a.z; xv[q][3] = a.w;
                    xv[q][4] = b.x; xv[q][5] = b.y; xv[q][6] = b.z; xv[q][7] = b.w;
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e)
                        xv[q][e] = (row < p.N && k + e < p.K) ? __ldg(x + e) : 0.0f;
                }
            }
            if (p.scale != nullptr) {
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const bool in = k + e < p.K;     // y = fmaf(0, 0, 0) = 0 past K
                    sv[e] = in ? __ldg(p.scale + k + e) : 0.0f;
                    tv[e] = in ? __ldg(p.shift + k + e) : 0.0f;
                }
            }
#pragma unroll
            for (int q = 0; q < kBRows; ++q) {
                const int col = n0 + r0 + 32 * q;
                wsign[q] = col < p.F ? __ldg(p.b_bits + int64_t(col) * p.words + kb) : 0ull;
            }
        } else {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int64_t row = m0 + r0 + 32 * q;
                wsign[q] = row < p.N ? __ldg(p.a_bits + row * p.words + kb) : 0ull;
            }
            const int64_t kp = int64_t(p.words) * kMixK;
#pragma unroll
            for (int q = 0; q < kBRows; ++q) {
                const int col = n0 + r0 + 32 * q;
#pragma unroll
                for (int part = 0; part < kParts; ++part)
                    wpart[q][part] =
                        col < p.F ? __ldg(reinterpret_cast<const uint4 *>(
                                        p.wparts + (int64_t(part) * p.F + col) * kp + k))
                                  : make_uint4(0u, 0u, 0u, 0u);
            }
        }
    };

    auto store = [&](unsigned char *sa, unsigned char *sb) {
        if constexpr (kRealA) {
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                uint32_t h[4], m[4], l[4];
#pragma unroll
                for (int w = 0; w < 4; ++w) {
                    uint32_t h0, m0_, l0, h1, m1, l1;
                    float y0 = xv[q][2 * w], y1 = xv[q][2 * w + 1];
                    if (p.scale != nullptr) {
                        y0 = __fmaf_rn(y0, sv[2 * w], tv[2 * w]);
                        y1 = __fmaf_rn(y1, sv[2 * w + 1], tv[2 * w + 1]);
                    }
                    split3(y0, h0, m0_, l0);
                    split3(y1, h1, m1, l1);
                    h[w] = h0 | (h1 << 16);
                    m[w] = m0_ | (m1 << 16);
                    l[w] = l0 | (l1 << 16);
                }
                const uint32_t off = sw128_offset(r0 + 32 * q, c);
                *reinterpret_cast<uint4 *>(sa + off) = make_uint4(h[0], h[1], h[2], h[3]);
                *reinterpret_cast<uint4 *>(sa + S::kTileA + off) = make_uint4(m[0], m[1], m[2], m[3]);
                *reinterpret_cast<uint4 *>(sa + 2 * S::kTileA + off) =
                    make_uint4(l[0], l[1], l[2], l[3]);
            }
#pragma unroll
            for (int q = 0; q < kBRows; ++q)
                *reinterpret_cast<uint4 *>(sb + sw128_offset(r0 + 32 * q, c)) =
                    signs8_to_bf16(uint32_t(wsign[q] >> (8 * c)) & 0xFFu);
        } else {
#pragma unroll
            for (int q = 0; q < 4; ++q)
                *reinterpret_cast<uint4 *>(sa + sw128_offset(r0 + 32 * q, c)) =
                    signs8_to_bf16(uint32_t(wsign[q] >> (8 * c)) & 0xFFu);
#pragma unroll
            for (int q = 0; q < kBRows; ++q) {
                const uint32_t off = sw128_offset(r0 + 32 * q, c);
#pragma unroll
                for (int part = 0; part < kParts; ++part)
                    *reinterpret_cast<uint4 *>(sb + part * S::kTileB + off) = wpart[q][part];
            }
        }
    };

    constexpr uint32_t idesc = bf16_idesc(NT);
    bool ok = true;
    int committed = -1;          // last local k-block whose MMAs were committed
    if (kb0 < kb1) load(kb0);
    for (int kb = kb0; kb < kb1; ++kb) {
        const int it = kb - kb0;
        const int s = it % kStages;
        if (it >= kStages) {
            const bool done = mbar_wait(smem_addr(&bars[s]), uint32_t(it / kStages - 1) & 1u);
            if (!__syncthreads_and(done)) {
                ok = false;
                break;
            }
        }
        unsigned char *sa = tiles + s * S::kStage;
        unsigned char *sb = sa + (kRealA ? kParts * S::kTileA : S::kTileA);
        store(sa, sb);
        if (kb + 1 < kb1) load(kb + 1);      // in flight across the barrier and MMAs
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (tid == 0) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t a0 = smem_addr(sa), b0 = smem_addr(sb);
#pragma unroll
            for (int k = 0; k < kMixK / 16; ++k)
#pragma unroll
                for (int part = 0; part < kParts; ++part) {
                    const uint32_t a = a0 + (kRealA ? part * S::kTileA : 0) + 32u * k;
                    const uint32_t b = b0 + (kRealA ? 0 : part * S::kTileB) + 32u * k;
                    mma_bf16(tmem, sw128_desc(a), sw128_desc(b), idesc,
                             (it > 0 || k > 0 || part > 0) ? 1u : 0u);
                }
            asm volatile(
                "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                    smem_addr(&bars[s]))
                : "memory");
        }
        committed = it;
    }
    bool done = true;
    if (committed >= 0)
        done = mbar_wait(smem_addr(&bars[committed % kStages]),
                         uint32_t(committed / kStages) & 1u);
    ok = __syncthreads_and(ok && done) != 0;
    if (!ok && tid == 0) atomicAdd(&g_mix_timeouts, 1u);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");

    const int quad = warp & 3;
    const uint32_t taddr = tmem + (uint32_t(32 * quad) << 16);
    auto row_scale = [&](int64_t row) {
        float rs = kRealA ? 1.0f : __ldg(p.alpha + row);
        if (p.rowptr != nullptr) {
            const float d = inv_sqrt_degree(__ldg(p.rowptr + row + 1) - __ldg(p.rowptr + row));
            rs = kRealA ? d : rs * d;
        }
        return rs;
    };
    auto scaled = [&](float rs, int col, float acc) {
        return kRealA ? rs * (__ldg(p.beta + col) * acc) : rs * acc;
    };
    const bool vec_z = (p.ldz & 3) == 0 && (reinterpret_cast<uintptr_t>(p.Z) & 15) == 0;

    if (KS == 1) {
        if (ok) {
            const int64_t row = m0 + 32 * quad + lane;
            const float rs = row < p.N ? row_scale(row) : 0.0f;
#pragma unroll 1
            for (int c0 = 16 * (warp >> 2); c0 < NT; c0 += 32) {
                uint32_t acc[16];
                tmem_ld16(taddr + uint32_t(c0), acc);
                if (row >= p.N) continue;
                const int col0 = n0 + c0;
                float z[16];
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    z[j] = scaled(rs, min(col0 + j, p.F - 1), __uint_as_float(acc[j]));
                float *zr = p.Z + row * p.ldz + col0;
                if (vec_z && col0 + 16 <= p.F) {
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        reinterpret_cast<float4 *>(zr)[q] =
                            make_float4(z[4 * q], z[4 * q + 1], z[4 * q + 2], z[4 * q + 3]);
                } else {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        if (col0 + j < p.F) zr[j] = z[j];
                }
            }
        }
    } else {
        // Partial tile -> this CTA's shared memory (all stages are idle now).
        float *red = reinterpret_cast<float *>(tiles);
        const int rl = 32 * quad + lane;
#pragma unroll 1
        for (int c0 = 16 * (warp >> 2); c0 < NT; c0 += 32) {
            uint32_t acc[16];
            if (committed >= 0 && ok) tmem_ld16(taddr + uint32_t(c0), acc);
            else {
#pragma unroll
                for (int j = 0; j < 16; ++j) acc[j] = 0u;
            }
            float4 *dst = reinterpret_cast<float4 *>(red + rl * S::kRedStride + c0);
#pragma unroll
            for (int q = 0; q < 4; ++q)
                dst[q] = make_float4(__uint_as_float(acc[4 * q]), __uint_as_float(acc[4 * q + 1]),
                                     __uint_as_float(acc[4 * q + 2]),
                                     __uint_as_float(acc[4 * q + 3]));
        }
        if (tid == 0) s_ok = ok ? 1u : 0u;
        cluster_sync();
        uint32_t peer_ok = 1u;
        if (tid < KS) peer_ok = ld_cluster_u32(map_to_rank(smem_addr(&s_ok), uint32_t(tid)));
        const bool all_ok = __syncthreads_and(peer_ok != 0u) != 0;
        if (all_ok) {
            const int lo = (kUmmaM * rank) / KS, hi = (kUmmaM * (rank + 1)) / KS;
            constexpr int kC4 = NT / 4;
            const uint32_t red0 = smem_addr(red);
            for (int idx = tid; idx < (hi - lo) * kC4; idx += kMixThreads) {
                const int r = lo + idx / kC4, c4 = idx % kC4;
                const int64_t row = m0 + r;
                const int col0 = n0 + 4 * c4;
                if (row >= p.N || col0 >= p.F) continue;
                const uint32_t off = red0 + uint32_t(r * S::kRedStride + 4 * c4) * 4u;
                float4 v = ld_cluster_f4(map_to_rank(off, 0));
                for (int q = 1; q < KS; ++q) {
                    const float4 w = ld_cluster_f4(map_to_rank(off, uint32_t(q)));
                    v.x += w.x; v.y += w.y; v.z += w.z; v.w += w.w;
                }
                const float rs = row_scale(row);
                const float a[4] = {v.x, v.y, v.z, v.w};
                float *zr = p.Z + row * p.ldz + col0;
                if (vec_z && col0 + 4 <= p.F) {
                    *reinterpret_cast<float4 *>(zr) =
                        make_float4(scaled(rs, col0, a[0]), scaled(rs, col0 + 1, a[1]),
                                    scaled(rs, col0 + 2, a[2]), scaled(rs, col0 + 3, a[3]));
                } else {
#pragma unroll
                    for (int e = 0; e < 4; ++e)
                        if (col0 + e < p.F) zr[e] = scaled(rs, col0 + e, a[e]);
                }
            }
        }
        cluster_sync();          // peers have finished reading this CTA's partials
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(NT));
}

// W (K x F, row stride ldw) -> wparts[p][j][k], the three bf16 parts of
// W[k][j], zero for k >= K (k < words * 64). Thread (j, 8-element chunk).
__global__ void __launch_bounds__(256)
split_weights_kernel(const float *__restrict__ Wt, int K, int F, int64_t ldw, int words,
                     uint16_t *__restrict__ wparts) {
    const int64_t kp = int64_t(words) * kMixK;
    const int64_t chunks = kp / 8;
    const int64_t idx = int64_t(blockIdx.x) * blockDim.x + threadIdx.x;
    if (idx >= chunks * F) return;
    const int j = int(idx % F);
    const int64_t k0 = (idx / F) * 8;
    uint32_t h[4], m[4], l[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) {
        uint32_t hh[2], mm[2], ll[2];
#pragma unroll
        for (int e = 0; e < 2; ++e) {
            const int64_t k = k0 + 2 * w + e;
            const float v = k < K ? __ldg(Wt + k * ldw + j) : 0.0f;
            split3(v, hh[e], mm[e], ll[e]);
        }
        h[w] = hh[0] | (hh[1] << 16);
        m[w] = mm[0] | (mm[1] << 16);
        l[w] = ll[0] | (ll[1] << 16);
    }
    uint4 *dst = reinterpret_cast<uint4 *>(wparts + int64_t(j) * kp + k0);
    const int64_t part = int64_t(F) * kp / 8;     // uint4s per part
    dst[0] = make_uint4(h[0], h[1], h[2], h[3]);
    dst[part] = make_uint4(m[0], m[1], m[2], m[3]);
    dst[2 * part] = make_uint4(l[0], l[1], l[2], l[3]);
}

template <int NT, bool kRealA>
void launch_mix(MixParams p, const DeviceInfo &dev, cudaStream_t stream, bool pdl) {
    using S = MixShape<NT, kRealA>;
    const int64_t tiles = (p.N + kUmmaM - 1) / kUmmaM;
    const int ctiles = (p.F + NT - 1) / NT;
    // Split the k-blocks over a cluster while the tiles leave SMs idle.
    int ks = 1;
    while (ks < kMaxSplit && ks < p.words && tiles * ctiles * (ks + 1) <= dev.sm_count) ++ks;
    p.split = ks;
    cudaFuncSetAttribute(mixed_gemm_tc_kernel<NT, kRealA>,
                         cudaFuncAttributeMaxDynamicSharedMemorySize, int(S::kSmem));
    const dim3 grid(unsigned(tiles * ks), unsigned(ctiles));
    launch_kernel(mixed_gemm_tc_kernel<NT, kRealA>, grid, dim3(kMixThreads), S::kSmem, stream, pdl,
                  dim3(unsigned(ks), 1, 1), p);
}

}  // namespace

size_t weight_parts_bytes(int K, int F) {
    return size_t(kParts) * size_t(F) * size_t(bigcn_words(K)) * kMixK * 2;
}

void launch_real_binary_gemm(const RealBinaryArgs &g, const DeviceInfo &dev, cudaStream_t stream,
                             bool pdl) {
    if (g.N == 0) return;
    MixParams p{};
    p.X = g.X;
    p.ldx = g.ldx;
    p.scale = g.scale;
    p.shift = g.shift;
    p.b_bits = g.b_bits;
    p.beta = g.beta;
    p.N = g.N;
    p.K = g.K;
    p.F = g.F;
    p.words = g.words;
    p.Z = g.Z;
    p.ldz = g.ldz;
    p.rowptr = g.rowptr;
    if (g.F <= 64) launch_mix<64, true>(p, dev, stream, pdl);
    else if (g.F <= 128) launch_mix<128, true>(p, dev, stream, pdl);
    else launch_mix<256, true>(p, dev, stream, pdl);
}

void launch_split_weights(const float *Wt, int K, int F, int64_t ldw, uint16_t *wparts,
                          cudaStream_t stream) {
    const int64_t n = int64_t(bigcn_words(K)) * kMixK / 8 * F;
    split_weights_kernel<<<unsigned((n + 255) / 256), 256, 0, stream>>>(Wt, K, F, ldw,
                                                                         bigcn_words(K), wparts);
}

void launch_binary_real_gemm(const BinaryRealArgs &g, const DeviceInfo &dev, cudaStream_t stream,
                             bool pdl) {
    if (g.N == 0) return;
    MixParams p{};
    p.a_bits = g.a_bits;
    p.alpha = g.alpha;
    p.wparts = g.wparts;
    p.N = g.N;
    p.K = g.K;
    p.F = g.F;
    p.words = g.words;
    p.Z = g.Z;
    p.ldz = g.ldz;
    p.rowptr = g.rowptr;
    if (g.F <= 64) launch_mix<64, false>(p, dev, stream, pdl);
    else launch_mix<128, false>(p, dev, stream, pdl);
}

uint32_t take_mix_timeouts() {
    unsigned int n = 0;
    const unsigned int zero = 0;
    if (cudaMemcpyFromSymbol(&n, g_mix_timeouts, sizeof(n)) != cudaSuccess ||
        cudaMemcpyToSymbol(g_mix_timeouts, &zero, sizeof(zero)) != cudaSuccess) {
        cudaGetLastError();
        return ~0u;
    }
    return n;
}

}  // namespace bigcn

using namespace bigcn;

namespace {

constexpr size_t kWsAlign = 256;
size_t ws_round(size_t x) { return (x + kWsAlign - 1) / kWsAlign * kWsAlign; }

// Workspace of bigcn_layer_forward_ablation (weights / features binarized):
// the packed operand and its scales, the parts of W (features binarized), and
// Z' (N x F fp32).
struct AblationWorkspace {
    size_t bits, scales, parts, z, total;
};

bool ablation_workspace(int32_t binarize, int64_t N, int32_t K, int32_t F, AblationWorkspace *w) {
    if (N < 0 || K < 1 || F < 1) return false;
    if (binarize != BIGCN_BINARIZE_WEIGHTS && binarize != BIGCN_BINARIZE_FEATURES) return false;
    const int64_t words = bigcn_words(K);
    if (N > kMaxElems / (words > F ? words : F)) return false;
    const bool rows = binarize == BIGCN_BINARIZE_FEATURES;     // pack node rows, else W's columns
    const int64_t packed = rows ? N : F;
    size_t off = 0;
    w->bits = off;   off = ws_round(off + size_t(packed) * size_t(words) * 8);
    w->scales = off; off = ws_round(off + size_t(packed) * 4);
    w->parts = off;  if (rows) off = ws_round(off + weight_parts_bytes(K, F));
    w->z = off;      off = ws_round(off + size_t(N) * size_t(F) * 4);
    w->total = off;
    return true;
}

}  // namespace

extern "C" bigcn_status bigcn_real_binary_gemm(const float *X, int64_t N, int32_t K, int64_t ldx,
                                               const float *scale, const float *shift,
                                               const uint64_t *b_bits, const float *beta,
                                               int32_t F, int32_t words, float *Z, int64_t ldz,
                                               void *stream) {
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || ldx < K || ldz < F ||
        words != bigcn_words(K))
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / ldz)) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!X || !b_bits || !beta || !Z) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(b_bits, 8) || !aligned_to(beta, 4) || !aligned_to(Z, 4) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t zb = span_bytes(N, F, ldz, 4);
    const void *in[] = {X, b_bits, beta, scale, shift};
    const size_t inb[] = {span_bytes(N, K, ldx, 4), size_t(F) * size_t(words) * 8, size_t(F) * 4,
                          size_t(K) * 4, size_t(K) * 4};
    for (int q = 0; q < 5; ++q)
        if (overlaps(Z, zb, in[q], inb[q])) return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    RealBinaryArgs g{X, ldx, scale, shift, b_bits, beta, N, K, F, words, Z, ldz, nullptr};
    launch_real_binary_gemm(g, dev, as_stream(stream));
    return launch_status();
}

extern "C" size_t bigcn_binary_real_gemm_workspace_bytes(int32_t K, int32_t F) {
    if (K < 1 || F < 1) return 0;
    return ws_round(weight_parts_bytes(K, F));
}

extern "C" bigcn_status bigcn_binary_real_gemm(const uint64_t *a_bits, const float *alpha,
                                               int64_t N, int32_t K, int32_t words,
                                               const float *Wt, int32_t F, int64_t ldw,
                                               void *workspace, size_t ws_bytes, float *Z,
                                               int64_t ldz, void *stream) {
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || ldw < F || ldz < F ||
        words != bigcn_words(K))
        return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldz || N > kMaxElems / words)) return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    const size_t need = bigcn_binary_real_gemm_workspace_bytes(K, F);
    if (!a_bits || !alpha || !Wt || !Z || !workspace || ws_bytes < need)
        return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(a_bits, 8) || !aligned_to(alpha, 4) || !aligned_to(Wt, 4) ||
        !aligned_to(Z, 4) || !aligned_to(workspace, kWsAlign))
        return BIGCN_ERR_MISALIGNED;
    const size_t zb = span_bytes(N, F, ldz, 4);
    const void *in[] = {a_bits, alpha, Wt};
    const size_t inb[] = {size_t(N) * size_t(words) * 8, size_t(N) * 4, span_bytes(K, F, ldw, 4)};
    for (int q = 0; q < 3; ++q)
        if (overlaps(Z, zb, in[q], inb[q]) || overlaps(workspace, need, in[q], inb[q]))
            return BIGCN_ERR_INVALID_ARG;
    if (overlaps(Z, zb, workspace, need)) return BIGCN_ERR_INVALID_ARG;
    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    uint16_t *parts = static_cast<uint16_t *>(workspace);
    cudaStream_t s = as_stream(stream);
    launch_split_weights(Wt, K, F, ldw, parts, s);
    BinaryRealArgs g{a_bits, alpha, parts, N, K, F, words, Z, ldz, nullptr};
    launch_binary_real_gemm(g, dev, s);
    return launch_status();
}

extern "C" size_t bigcn_layer_ablation_workspace_bytes(int32_t binarize, int64_t N, int32_t K,
                                                       int32_t F) {
    if (binarize == BIGCN_BINARIZE_BOTH) return bigcn_layer_workspace_bytes(N, K, F);
    AblationWorkspace w;
    return ablation_workspace(binarize, N, K, F, &w) ? w.total : 0;
}

extern "C" bigcn_status bigcn_layer_forward_ablation(int32_t binarize, const float *X, int64_t N,
                                                     int32_t K, int64_t ldx, const float *scale,
                                                     const float *shift, const float *Wt,
                                                     int32_t F, int64_t ldw,
                                                     const int64_t *rowptr, const int32_t *colidx,
                                                     int64_t nnz, void *workspace,
                                                     size_t ws_bytes, float *H, int64_t ldh,
                                                     void *stream) {
    if (binarize == BIGCN_BINARIZE_BOTH)
        return bigcn_layer_forward(X, N, K, ldx, scale, shift, Wt, F, ldw, rowptr, colidx, nnz,
                                   workspace, ws_bytes, H, ldh, stream);
    AblationWorkspace w;
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || ldx < K || ldw < F || ldh < F ||
        nnz < 0)
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (!ablation_workspace(binarize, N, K, F, &w)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / ldh)) return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!X || !Wt || !rowptr || !H || !workspace || (nnz > 0 && !colidx))
        return BIGCN_ERR_INVALID_ARG;
    if (ws_bytes < w.total) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(Wt, 4) || !aligned_to(rowptr, 8) ||
        (colidx && !aligned_to(colidx, 4)) || !aligned_to(H, 4) ||
        !aligned_to(workspace, kWsAlign) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t xb = span_bytes(N, K, ldx, 4), hb = span_bytes(N, F, ldh, 4);
    const void *inputs[] = {X, Wt, rowptr, colidx, scale, shift};
    const size_t in_bytes[] = {xb, span_bytes(K, F, ldw, 4), size_t(N + 1) * 8, size_t(nnz) * 4,
                               size_t(K) * 4, size_t(K) * 4};
    for (int q = 0; q < 6; ++q) {
        if (overlaps(workspace, w.total, inputs[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
        if (overlaps(H, hb, inputs[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
    }
    if (overlaps(H, hb, workspace, w.total)) return BIGCN_ERR_INVALID_ARG;

    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    char *ws = static_cast<char *>(workspace);
    uint64_t *bits = reinterpret_cast<uint64_t *>(ws + w.bits);
    float *scales = reinterpret_cast<float *>(ws + w.scales);
    float *Zs = reinterpret_cast<float *>(ws + w.z);
    const int words = bigcn_words(K);
    cudaStream_t s = as_stream(stream);
    if (binarize == BIGCN_BINARIZE_WEIGHTS) {
        launch_pack_weights(Wt, K, F, ldw, bits, words, scales, s);
        RealBinaryArgs g{X, ldx, scale, shift, bits, scales, N, K, F, words, Zs, F, rowptr};
        launch_real_binary_gemm(g, dev, s);
    } else {
        uint16_t *parts = reinterpret_cast<uint16_t *>(ws + w.parts);
        launch_pack_rows(X, N, K, ldx, scale, shift, bits, words, scales, dev, s);
        launch_split_weights(Wt, K, F, ldw, parts, s);
        BinaryRealArgs g{bits, scales, parts, N, K, F, words, Zs, F, rowptr};
        launch_binary_real_gemm(g, dev, s);
    }
    SpmmArgs a{rowptr, colidx, N, nnz, Zs, F, F, H, ldh, true, false};
    launch_spmm_norm(a, dev, s);
    return launch_status();
}
