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

constexpr int kProducerWarps = 16;
constexpr int kProducers = 32 * kProducerWarps;     // threads that build the operand tiles
constexpr int kMmaWarp = kProducerWarps;            // the warp that issues the MMAs
constexpr int kMixThreads = kProducers + 32;
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

__device__ __forceinline__ void commit_to(uint64_t *bar) {
    asm volatile(
        "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
            smem_addr(bar))
        : "memory");
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

// Three bf16 parts of two values v0, v1, packed as pairs (v0 in the low half).
// hi keeps the top 16 bits of v (a bf16 by truncation), so r = v - hi is
// exact in fp32 (v's low 16 mantissa bits) with |r| < 2^-7 |v|; mid is r
// truncated the same way, q = r - mid exact with |q| < 2^-14 |v|; lo is q
// rounded to nearest bf16, so |v - (hi + mid + lo)| <= 2^-9 |q| < 2^-23 |v|.
__device__ __forceinline__ void split3x2(float v0, float v1, uint32_t &hi, uint32_t &mid,
                                         uint32_t &lo) {
    const uint32_t u0 = __float_as_uint(v0), u1 = __float_as_uint(v1);
    const float r0 = v0 - __uint_as_float(u0 & 0xFFFF0000u);
    const float r1 = v1 - __uint_as_float(u1 & 0xFFFF0000u);
    const uint32_t w0 = __float_as_uint(r0), w1 = __float_as_uint(r1);
    const float q0 = r0 - __uint_as_float(w0 & 0xFFFF0000u);
    const float q1 = r1 - __uint_as_float(w1 & 0xFFFF0000u);
    hi = __byte_perm(u0, u1, 0x7632);
    mid = __byte_perm(w0, w1, 0x7632);
    const __nv_bfloat162 l = __floats2bfloat162_rn(q0, q1);
    lo = *reinterpret_cast<const uint32_t *>(&l);
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

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, uint32_t src_bytes) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(src_bytes)
                 : "memory");
}

__device__ __forceinline__ void cp_async8(uint32_t dst, const void *src, uint32_t src_bytes) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 8, %2;" ::"r"(dst), "l"(src),
                 "r"(src_bytes)
                 : "memory");
}

__device__ __forceinline__ void cp_async4(uint32_t dst, const void *src, uint32_t src_bytes) {
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(dst), "l"(src),
                 "r"(src_bytes)
                 : "memory");
}

__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}

// Waits until at most N of this thread's most recent copy groups are pending.
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

// mbar_wait that also gives up as soon as another thread of the CTA has
// raised *abort (after its own wait ran out); false if it gave up.
__device__ __forceinline__ bool wait_or_abort(uint32_t bar, uint32_t parity,
                                              const volatile uint32_t *abort) {
    for (uint32_t it = 0; it < kWaitLimit; ++it) {
        uint32_t done;
        asm volatile(
            "{\n.reg .pred p;\n"
            "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n"
            "selp.u32 %0, 1, 0, p;\n}"
            : "=r"(done)
            : "r"(bar), "r"(parity)
            : "memory");
        if (done) return true;
        if (*abort) return false;
    }
    return false;
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
    bool clip;               // store z where |z| < 1, else 0 (Eq. bp-H)
};

// Shared-memory plan. Weights binarized (A real): kStages operand stages of
// three 128-row part tiles plus the NT-row sign tile, then a ring of kRaw raw
// fp32 k-blocks of X (128 rows x 64). Features binarized (B real): kHalves = 2
// row tiles of 128 (256 node rows per CTA, so that each copy of W's parts
// serves twice the rows): stages of the two sign tiles plus W's three NT-row
// part tiles.
template <int NT, bool kRealA>
struct MixShape {
    static constexpr int kHalves = kRealA ? 1 : 2;
    static constexpr int kRows = kUmmaM * kHalves;                 // node rows per CTA
    static constexpr int kTileA = kUmmaM * 128;                    // one 128-row bf16 tile
    static constexpr int kTileB = NT * 128;
    static constexpr int kStage =
        kRealA ? kParts * kTileA + kTileB : kHalves * kTileA + kParts * kTileB;
    static constexpr int kRawBlock = kUmmaM * kMixK * 4;           // 32 KB of X
    static constexpr int kRaw = kRealA ? (NT <= 128 ? 3 : 2) : 0;
    static constexpr int kStages = kRealA ? 2 : 4;
    static constexpr int kRedStride = NT + 4;                      // floats per partial row
    static constexpr size_t kBytes = size_t(kRaw) * kRawBlock + size_t(kStages) * kStage;
    static constexpr size_t kSmem = 1024 + kBytes;
    static_assert(kSmem <= 227 * 1024, "shared memory per CTA");
    static_assert(size_t(kRows) * kRedStride * 4 <= size_t(kStages) * kStage,
                  "the partial tile reuses the stage buffers");
};

// Barriers and flags of one CTA: stage s is full once every producer thread
// has arrived on full[s], and empty again once the MMAs that read it commit
// to empty[s]; `done` receives the commit that follows the last MMA.
template <int kStages>
struct MixSync {
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t done;
    uint32_t tmem_base;
    uint32_t abort;
    uint32_t ok;
};

template <int kCols, int kStages>
__device__ __forceinline__ uint32_t mix_setup(MixSync<kStages> &sy) {
    const int tid = threadIdx.x;
    if ((tid >> 5) == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_addr(&sy.tmem_base)),
                     "r"(kCols));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (tid == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(smem_addr(&sy.full[s]), kProducers);
            mbar_init(smem_addr(&sy.empty[s]), 1);
        }
        mbar_init(smem_addr(&sy.done), 1);
        sy.abort = 0u;
        mbar_fence_init();
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    return sy.tmem_base;
}

template <int kCols>
__device__ __forceinline__ void mix_teardown(uint32_t tmem) {
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if ((threadIdx.x >> 5) == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(kCols));
}

// The MMA warp: for each k-block, wait until its stage is full, issue the
// MMAs (lane 0) and commit them to the stage's `empty` barrier; finally commit
// to `done`, which then tracks every MMA issued.
template <int kStages, typename Issue>
__device__ __forceinline__ void mma_loop(MixSync<kStages> &sy, int nkb, Issue issue) {
    const int lane = threadIdx.x & 31;
    bool any = false;
#pragma unroll 1
    for (int it = 0; it < nkb; ++it) {
        const int s = it % kStages;
        if (!wait_or_abort(smem_addr(&sy.full[s]), uint32_t(it / kStages) & 1u, &sy.abort)) {
            sy.abort = 1u;
            break;
        }
        asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
        if (lane == 0) {
            issue(it, s);
            commit_to(&sy.empty[s]);
        }
        any = true;
        __syncwarp();
    }
    if (lane == 0) {
        if (any) commit_to(&sy.done);
        else mbar_arrive(smem_addr(&sy.done));
    }
    __syncwarp();
}

// After the main loop: move the accumulators out of tensor memory and store
// Z (KS == 1), or add the KS partials of the cluster in rank order first.
// Accumulator h (h < kHalves) holds rows 128 h .. 128 h + 127 in tensor-memory
// columns h NT .. h NT + NT - 1. The producer warps read it: warp w may read
// lanes 32 (w % 4) ..; group g = w / 4 takes a share of the columns.
template <int NT, bool kRealA, int kStages>
__device__ __forceinline__ void mix_epilogue(const MixParams &p, unsigned char *tiles,
                                             uint32_t tmem, int64_t m0, int n0, int rank,
                                             bool ok, bool has_acc, MixSync<kStages> &sy) {
    using S = MixShape<NT, kRealA>;
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int KS = p.split;
    const bool reader = warp < kProducerWarps;
    const int quad = warp & 3, group = (warp >> 2) & 3;
    const int half = S::kHalves == 2 ? (group & 1) : 0;
    const int cfirst = S::kHalves == 2 ? 16 * (group >> 1) : 16 * group;
    const int cstep = S::kHalves == 2 ? 32 : 64;
    const int rl = 128 * half + 32 * quad + lane;                 // row within the CTA
    const uint32_t taddr = tmem + (uint32_t(32 * quad) << 16) + uint32_t(half * NT);
    auto row_scale = [&](int64_t row) {
        float rs = kRealA ? 1.0f : __ldg(p.alpha + row);
        if (p.rowptr != nullptr) {
            const float d = inv_sqrt_degree(__ldg(p.rowptr + row + 1) - __ldg(p.rowptr + row));
            rs = kRealA ? d : rs * d;
        }
        return rs;
    };
    auto scaled = [&](float rs, int col, float acc) {
        float z = kRealA ? rs * ((p.beta != nullptr ? __ldg(p.beta + col) : 1.0f) * acc)
                         : rs * acc;
        if (p.clip && !(fabsf(z) < 1.0f)) z = 0.0f;
        return z;
    };
    const bool vec_z = (p.ldz & 3) == 0 && (reinterpret_cast<uintptr_t>(p.Z) & 15) == 0;

    if (KS == 1) {
        if (!ok || !reader) return;
        const int64_t row = m0 + rl;
        const float rs = row < p.N ? row_scale(row) : 0.0f;
#pragma unroll 1
        for (int c0 = cfirst; c0 < NT; c0 += cstep) {
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
        return;
    }
    // Partial tile -> this CTA's shared memory (every stage is idle now).
    float *red = reinterpret_cast<float *>(tiles);
    if (reader) {
#pragma unroll 1
        for (int c0 = cfirst; c0 < NT; c0 += cstep) {
            uint32_t acc[16];
            if (has_acc && ok) tmem_ld16(taddr + uint32_t(c0), acc);
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
    }
    if (tid == 0) sy.ok = ok ? 1u : 0u;
    cluster_sync();
    uint32_t peer_ok = 1u;
    if (tid < KS) peer_ok = ld_cluster_u32(map_to_rank(smem_addr(&sy.ok), uint32_t(tid)));
    if (__syncthreads_and(peer_ok != 0u)) {
        const int lo = (S::kRows * rank) / KS, hi = (S::kRows * (rank + 1)) / KS;
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

// Common end of both kernels: wait for the last MMA (`done`), count a wait
// that ran out, then the epilogue and the release of tensor memory.
template <int NT, bool kRealA, int kStages>
__device__ __forceinline__ void mix_finish(const MixParams &p, unsigned char *tiles, uint32_t tmem,
                                           int64_t m0, int n0, int rank, bool has_acc,
                                           MixSync<kStages> &sy) {
    cp_async_wait<0>();            // no copy of this thread is left in flight
    const bool done = mbar_wait(smem_addr(&sy.done), 0u);
    const bool ok = __syncthreads_and(done && sy.abort == 0u) != 0;
    if (!ok && threadIdx.x == 0) atomicAdd(&g_mix_timeouts, 1u);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    mix_epilogue<NT, kRealA, kStages>(p, tiles, tmem, m0, n0, rank, ok, has_acc, sy);
    mix_teardown<MixShape<NT, kRealA>::kHalves * NT>(tmem);
}

// ---- weights binarized: Z = Y W~ (A = centred X, real; B = signs of W) ----
//
// Producer thread t owns 16-byte chunk c = t & 7 (elements 8c .. 8c + 7 of a
// k-block) of rows r0 + 64 q (r0 = t >> 3, q < 2) of the A tiles and of rows
// r0 + 64 q (q < NT / 64) of the sign tile. It copies its own 64 elements of
// X for k-block kb + kRaw - 1 into the raw ring with cp.async (zero-filled
// past N and K) while it converts k-block kb, so kRaw - 1 k-blocks of X are in
// flight per thread; it reads back only what it copied itself, so the wait on
// its own copy group suffices. Odd rows take their two 16-byte halves in the
// other order, which spreads each copy and read instruction over all banks.
template <int NT>
__global__ void __launch_bounds__(kMixThreads, 1)
real_binary_tc_kernel(const MixParams p) {
    using S = MixShape<NT, true>;
    constexpr int kStages = S::kStages, kRaw = S::kRaw;
    constexpr int kARows = kUmmaM / 64, kBRows = NT / 64;
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) MixSync<kStages> sy;

    const int tid = threadIdx.x, warp = tid >> 5;
    const int KS = p.split;
    const int rank = KS > 1 ? int(cluster_rank()) : 0;
    const int64_t m0 = int64_t(blockIdx.x / KS) * kUmmaM;
    const int n0 = blockIdx.y * NT;
    const uint32_t raw_addr = smem_addr(smem_raw);
    const uint32_t base = (raw_addr + 1023u) & ~1023u;
    unsigned char *tiles = smem_raw + (base - raw_addr);          // stages, then the raw ring
    unsigned char *ring = tiles + kStages * S::kStage;
    const uint32_t ring_addr = base + kStages * S::kStage;

    const int KB = p.words;
    const int per = (KB + KS - 1) / KS;
    const int kb0 = min(KB, rank * per), kb1 = min(KB, kb0 + per);

    const uint32_t tmem = mix_setup<NT, kStages>(sy);
    grid_dependency_wait();     // the packed weights come from an earlier kernel

    if (warp == kMmaWarp) {
        constexpr uint32_t idesc = bf16_idesc(NT);
        mma_loop<kStages>(sy, kb1 - kb0, [&](int it, int s) {
            const uint32_t a0 = base + s * S::kStage, b0 = a0 + kParts * S::kTileA;
#pragma unroll
            for (int k = 0; k < kMixK / 16; ++k)
#pragma unroll
                for (int part = 0; part < kParts; ++part)
                    mma_bf16(tmem, sw128_desc(a0 + part * S::kTileA + 32u * k),
                             sw128_desc(b0 + 32u * k), idesc,
                             (it > 0 || k > 0 || part > 0) ? 1u : 0u);
        });
    } else {
        const int c = tid & 7, r0 = tid >> 3;
        const int odd = r0 & 1;
        // Widest copy every row start allows: 16, 8 or 4 bytes.
        const uintptr_t xa = reinterpret_cast<uintptr_t>(p.X);
        const int width = ((p.ldx & 3) == 0 && (xa & 15) == 0) ? 16
                          : ((p.ldx & 1) == 0 && (xa & 7) == 0) ? 8 : 4;

        auto issue = [&](int kb) {      // this thread's 64 elements of X for k-block kb
            const uint32_t slot = ring_addr + uint32_t(((kb - kb0) % kRaw) * S::kRawBlock);
#pragma unroll
            for (int q = 0; q < kARows; ++q) {
                const int r = r0 + 64 * q;
                const int64_t row = m0 + r;
                const int k = kb * kMixK + 8 * c;
                const uint32_t dst = slot + uint32_t(r * kMixK + 8 * c) * 4u;
                const float *src = p.X + (row < p.N ? row : 0) * p.ldx;
                if (width == 16) {
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        const int hh = h ^ odd;
                        const int kk = k + 4 * hh;
                        const int n = row < p.N ? min(max(p.K - kk, 0), 4) : 0;
                        cp_async16(dst + 16u * hh, n > 0 ? src + kk : p.X, uint32_t(4 * n));
                    }
                } else if (width == 8) {
#pragma unroll
                    for (int h = 0; h < 4; ++h) {
                        const int hh = h ^ (2 * odd);
                        const int kk = k + 2 * hh;
                        const int n = row < p.N ? min(max(p.K - kk, 0), 2) : 0;
                        cp_async8(dst + 8u * hh, n > 0 ? src + kk : p.X, uint32_t(4 * n));
                    }
                } else {
#pragma unroll
                    for (int e = 0; e < 8; ++e) {
                        const bool in = row < p.N && k + e < p.K;
                        cp_async4(dst + 4u * e, in ? src + k + e : p.X, in ? 4u : 0u);
                    }
                }
            }
        };
        uint64_t wsign[kBRows];
        float sv[8], tv[8];
        auto load_small = [&](int kb) {     // sign words and centring of k-block kb
#pragma unroll
            for (int q = 0; q < kBRows; ++q) {
                const int col = n0 + r0 + 64 * q;
                wsign[q] = col < p.F ? __ldg(p.b_bits + int64_t(col) * p.words + kb) : 0ull;
            }
            if (p.scale != nullptr) {
                const int k = kb * kMixK + 8 * c;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const bool in = k + e < p.K;      // y = fmaf(0, 0, 0) = 0 past K
                    sv[e] = in ? __ldg(p.scale + k + e) : 0.0f;
                    tv[e] = (in && p.shift != nullptr) ? __ldg(p.shift + k + e) : 0.0f;
                }
            }
        };

#pragma unroll 1
        for (int d = 0; d < kRaw - 1; ++d) {
            if (kb0 + d < kb1) issue(kb0 + d);
            cp_async_commit();
        }
        if (kb0 < kb1) load_small(kb0);
#pragma unroll 1
        for (int kb = kb0; kb < kb1; ++kb) {
            const int it = kb - kb0;
            const int s = it % kStages;
            if (kb + kRaw - 1 < kb1) issue(kb + kRaw - 1);
            cp_async_commit();
            if (it >= kStages &&
                !wait_or_abort(smem_addr(&sy.empty[s]), uint32_t(it / kStages - 1) & 1u,
                               &sy.abort)) {
                sy.abort = 1u;
                break;
            }
            cp_async_wait<kRaw - 1>();     // this thread's copy of k-block kb has landed
            unsigned char *sa = tiles + s * S::kStage;
            unsigned char *sb = sa + kParts * S::kTileA;
            const unsigned char *slot = ring + (it % kRaw) * S::kRawBlock;
#pragma unroll
            for (int q = 0; q < kARows; ++q) {
                const int r = r0 + 64 * q;
                const float4 *xr =
                    reinterpret_cast<const float4 *>(slot + (r * kMixK + 8 * c) * 4);
                const float4 xa = xr[odd], xb = xr[odd ^ 1];
                const float4 x0 = odd ? xb : xa, x1 = odd ? xa : xb;
                float y[8] = {x0.x, x0.y, x0.z, x0.w, x1.x, x1.y, x1.z, x1.w};
                if (p.scale != nullptr) {
#pragma unroll
                    for (int e = 0; e < 8; ++e) y[e] = __fmaf_rn(y[e], sv[e], tv[e]);
                }
                uint32_t h[4], m[4], l[4];
#pragma unroll
                for (int w = 0; w < 4; ++w) split3x2(y[2 * w], y[2 * w + 1], h[w], m[w], l[w]);
                const uint32_t off = sw128_offset(r, c);
                *reinterpret_cast<uint4 *>(sa + off) = make_uint4(h[0], h[1], h[2], h[3]);
                *reinterpret_cast<uint4 *>(sa + S::kTileA + off) =
                    make_uint4(m[0], m[1], m[2], m[3]);
                *reinterpret_cast<uint4 *>(sa + 2 * S::kTileA + off) =
                    make_uint4(l[0], l[1], l[2], l[3]);
            }
#pragma unroll
            for (int q = 0; q < kBRows; ++q)
                *reinterpret_cast<uint4 *>(sb + sw128_offset(r0 + 64 * q, c)) =
                    signs8_to_bf16(uint32_t(wsign[q] >> (8 * c)) & 0xFFu);
            if (kb + 1 < kb1) load_small(kb + 1);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            mbar_arrive(smem_addr(&sy.full[s]));
        }
    }
    mix_finish<NT, true, kStages>(p, tiles, tmem, m0, n0, rank, kb1 > kb0, sy);
}

// ---- features binarized: Z = H~ W (A = signs of the node rows; B = W real) ----
//
// 256 node rows per CTA (two 128-row accumulators sharing each B tile). W's
// bf16 parts (already split, K-contiguous per column) are copied with
// cp.async straight into their 128B-swizzled places, two k-blocks ahead: the
// copies for k-block kb + 2 go into the stage of kb - 2 once its MMAs have
// completed. The sign tiles are expanded from the packed words (loaded one
// k-block ahead) by the same threads.
template <int NT>
__global__ void __launch_bounds__(kMixThreads, 1)
binary_real_tc_kernel(const MixParams p) {
    using S = MixShape<NT, false>;
    constexpr int kStages = S::kStages;
    constexpr int kAhead = kStages - 2;
    constexpr int kARows = S::kRows / 64;                  // sign rows per thread
    constexpr int kBRows = NT / 64;
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) MixSync<kStages> sy;

    const int tid = threadIdx.x, warp = tid >> 5;
    const int KS = p.split;
    const int rank = KS > 1 ? int(cluster_rank()) : 0;
    const int64_t m0 = int64_t(blockIdx.x / KS) * S::kRows;
    const int n0 = blockIdx.y * NT;
    const uint32_t raw_addr = smem_addr(smem_raw);
    const uint32_t base = (raw_addr + 1023u) & ~1023u;
    unsigned char *tiles = smem_raw + (base - raw_addr);

    const int KB = p.words;
    const int per = (KB + KS - 1) / KS;
    const int kb0 = min(KB, rank * per), kb1 = min(KB, kb0 + per);

    const uint32_t tmem = mix_setup<S::kHalves * NT, kStages>(sy);
    grid_dependency_wait();     // packed rows and W's parts come from earlier kernels

    if (warp == kMmaWarp) {
        constexpr uint32_t idesc = bf16_idesc(NT);
        mma_loop<kStages>(sy, kb1 - kb0, [&](int it, int s) {
            const uint32_t a0 = base + s * S::kStage, b0 = a0 + S::kHalves * S::kTileA;
#pragma unroll
            for (int k = 0; k < kMixK / 16; ++k)
#pragma unroll
                for (int h = 0; h < S::kHalves; ++h)
#pragma unroll
                    for (int part = 0; part < kParts; ++part)
                        mma_bf16(tmem + uint32_t(h * NT),
                                 sw128_desc(a0 + h * S::kTileA + 32u * k),
                                 sw128_desc(b0 + part * S::kTileB + 32u * k), idesc,
                                 (it > 0 || k > 0 || part > 0) ? 1u : 0u);
        });
    } else {
        const int c = tid & 7, r0 = tid >> 3;
        const int64_t kp = int64_t(p.words) * kMixK;
        auto issue = [&](int kb) {          // W's parts of k-block kb into its stage
            const uint32_t sb = base + uint32_t(((kb - kb0) % kStages) * S::kStage +
                                                S::kHalves * S::kTileA);
#pragma unroll
            for (int q = 0; q < kBRows; ++q) {
                const int r = r0 + 64 * q;
                const int col = n0 + r;
                const uint32_t off = sw128_offset(r, c);
#pragma unroll
                for (int part = 0; part < kParts; ++part) {
                    const uint16_t *src = p.wparts +
                                          (int64_t(part) * p.F + (col < p.F ? col : 0)) * kp +
                                          int64_t(kb) * kMixK + 8 * c;
                    cp_async16(sb + part * S::kTileB + off, src, col < p.F ? 16u : 0u);
                }
            }
        };
        uint64_t wsign[kARows];
        auto load_signs = [&](int kb) {
#pragma unroll
            for (int q = 0; q < kARows; ++q) {
                const int64_t row = m0 + r0 + 64 * q;
                wsign[q] = row < p.N ? __ldg(p.a_bits + row * p.words + kb) : 0ull;
            }
        };

#pragma unroll 1
        for (int d = 0; d < kAhead; ++d) {
            if (kb0 + d < kb1) issue(kb0 + d);
            cp_async_commit();
        }
        if (kb0 < kb1) load_signs(kb0);
#pragma unroll 1
        for (int kb = kb0; kb < kb1; ++kb) {
            const int it = kb - kb0;
            const int s = it % kStages;
            // The stage of k-block kb + kAhead last held k-block kb - 2: its
            // MMAs (committed to that stage's `empty`) must be complete; those
            // of k-block kb - 4, which last used stage s, are then too.
            if (it >= 2) {
                const int prev = it - 2;
                if (!wait_or_abort(smem_addr(&sy.empty[prev % kStages]),
                                   uint32_t(prev / kStages) & 1u, &sy.abort)) {
                    sy.abort = 1u;
                    break;
                }
            }
            if (kb + kAhead < kb1) issue(kb + kAhead);
            cp_async_commit();
            unsigned char *sa = tiles + s * S::kStage;
#pragma unroll
            for (int q = 0; q < kARows; ++q) {
                const int r = r0 + 64 * q;             // row within the CTA's 256
                *reinterpret_cast<uint4 *>(sa + (r >> 7) * S::kTileA + sw128_offset(r & 127, c)) =
                    signs8_to_bf16(uint32_t(wsign[q] >> (8 * c)) & 0xFFu);
            }
            if (kb + 1 < kb1) load_signs(kb + 1);
            cp_async_wait<kAhead>();       // this thread's part copies of k-block kb have landed
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            mbar_arrive(smem_addr(&sy.full[s]));
        }
    }
    mix_finish<NT, false, kStages>(p, tiles, tmem, m0, n0, rank, kb1 > kb0, sy);
}

// ---- transposed signs x real: P_s = sum over nodes i of chunk s of
//      (alpha_i sign(y_ik)) G_ij  (dL/dW~ = H~^T G of Algorithm 1) ----
//
// M = the features k (128 per tile), N = the columns j (NT per tile), the
// contraction over nodes in k-blocks of 64, split over S CTAs (grid z) that
// each write a fp32 partial; the partials are added in order afterwards.
// A (K-major: a row per feature, 64 nodes along it) is built from the nodes'
// packed words: a producer warp takes 32 consecutive features of one 8-node
// chunk, so its eight word loads are broadcasts, and gathers bit k of each
// node into a byte of signs. B holds alpha_i G_ij (rounded once) as three
// bf16 parts, read coalesced across the columns. Warp roles and barriers are
// those of the ablation products.
template <int NT>
struct SignTShape {
    static constexpr int kTileA = kUmmaM * 128;
    static constexpr int kTileB = NT * 128;
    static constexpr int kStage = kTileA + kParts * kTileB;
    static constexpr int kStages = NT <= 64 ? 4 : (NT <= 128 ? 3 : 2);
    static constexpr size_t kSmem = 1024 + size_t(kStages) * kStage;
    static_assert(kSmem <= 227 * 1024, "shared memory per CTA");
};

struct SignTParams {
    const uint64_t *bits;    // N x words packed node signs (K features)
    int words;
    const float *alpha;      // N
    const float *G;          // N x F (row stride ldg)
    int64_t ldg;
    int64_t N;
    int K;
    int F;
    float *partial;          // S x K x F (row stride F)
    int per;                 // k-blocks (of 64 nodes) per split
};

template <int NT>
__global__ void __launch_bounds__(kMixThreads, 1)
sign_t_real_tc_kernel(const SignTParams p) {
    using S = SignTShape<NT>;
    constexpr int kStages = S::kStages;
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) MixSync<kStages> sy;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int m0 = blockIdx.x * kUmmaM;         // first feature of the tile
    const int n0 = blockIdx.y * NT;             // first column
    const int split = blockIdx.z;
    const int64_t KB = (p.N + kMixK - 1) / kMixK;
    const int64_t kb0 = min(KB, int64_t(split) * p.per), kb1 = min(KB, kb0 + p.per);
    const uint32_t raw_addr = smem_addr(smem_raw);
    const uint32_t base = (raw_addr + 1023u) & ~1023u;
    unsigned char *tiles = smem_raw + (base - raw_addr);

    const uint32_t tmem = mix_setup<NT, kStages>(sy);
    grid_dependency_wait();     // packed rows and G come from earlier kernels

    if (warp == kMmaWarp) {
        constexpr uint32_t idesc = bf16_idesc(NT);
        mma_loop<kStages>(sy, int(kb1 - kb0), [&](int it, int s) {
            const uint32_t a0 = base + s * S::kStage, b0 = a0 + S::kTileA;
#pragma unroll
            for (int k = 0; k < kMixK / 16; ++k)
#pragma unroll
                for (int part = 0; part < kParts; ++part)
                    mma_bf16(tmem, sw128_desc(a0 + 32u * k),
                             sw128_desc(b0 + part * S::kTileB + 32u * k), idesc,
                             (it > 0 || k > 0 || part > 0) ? 1u : 0u);
        });
    } else {
#pragma unroll 1
        for (int64_t kb = kb0; kb < kb1; ++kb) {
            const int it = int(kb - kb0);
            const int s = it % kStages;
            if (it >= kStages &&
                !wait_or_abort(smem_addr(&sy.empty[s]), uint32_t(it / kStages - 1) & 1u,
                               &sy.abort)) {
                sy.abort = 1u;
                break;
            }
            unsigned char *sa = tiles + s * S::kStage;
            unsigned char *sb = sa + S::kTileA;
            const int64_t i0 = kb * kMixK;
            // A: 4 x 8 (feature group, node chunk) tasks of 32 features x 8 nodes.
            for (int t = warp; t < 32; t += kProducerWarps) {
                const int c = t & 7, mh = t >> 3;
                const int m = 32 * mh + lane, f = m0 + m;
                const int wi = (m0 + 32 * mh) / 64;          // the same word for the warp
                uint32_t byte = 0;
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const int64_t i = i0 + 8 * c + e;
                    const uint64_t w =
                        (i < p.N && wi < p.words) ? __ldg(p.bits + i * p.words + wi) : 0ull;
                    byte |= uint32_t((w >> (f & 63)) & 1ull) << e;
                }
                *reinterpret_cast<uint4 *>(sa + sw128_offset(m, c)) = signs8_to_bf16(byte);
            }
            // B: (NT / 32) x 8 (column group, node chunk) tasks of 32 columns x 8 nodes.
            for (int t = warp; t < (NT / 32) * 8; t += kProducerWarps) {
                const int c = t & 7, jh = t >> 3;
                const int r = 32 * jh + lane, j = n0 + r;
                float v[8];
#pragma unroll
                for (int e = 0; e < 8; ++e) {
                    const int64_t i = i0 + 8 * c + e;
                    v[e] = (i < p.N && j < p.F) ? __ldg(p.alpha + i) * __ldg(p.G + i * p.ldg + j)
                                                : 0.0f;
                }
                uint32_t h[4], mi[4], lo[4];
#pragma unroll
                for (int w = 0; w < 4; ++w) split3x2(v[2 * w], v[2 * w + 1], h[w], mi[w], lo[w]);
                const uint32_t off = sw128_offset(r, c);
                *reinterpret_cast<uint4 *>(sb + off) = make_uint4(h[0], h[1], h[2], h[3]);
                *reinterpret_cast<uint4 *>(sb + S::kTileB + off) =
                    make_uint4(mi[0], mi[1], mi[2], mi[3]);
                *reinterpret_cast<uint4 *>(sb + 2 * S::kTileB + off) =
                    make_uint4(lo[0], lo[1], lo[2], lo[3]);
            }
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            mbar_arrive(smem_addr(&sy.full[s]));
        }
    }
    // The last MMA is done once `done` completes; then warps 0-15 move the
    // partial tile (rows = features, zeros for an empty split) to memory.
    const bool done = mbar_wait(smem_addr(&sy.done), 0u);
    const bool ok = __syncthreads_and(done && sy.abort == 0u) != 0;
    if (!ok && tid == 0) atomicAdd(&g_mix_timeouts, 1u);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    if (ok && warp < kProducerWarps) {
        const int quad = warp & 3, group = warp >> 2;
        const int f = m0 + 32 * quad + lane;
        const uint32_t taddr = tmem + (uint32_t(32 * quad) << 16);
        const bool has_acc = kb1 > kb0;
        float *prow = p.partial + (int64_t(split) * p.K + f) * p.F;
#pragma unroll 1
        for (int c0 = 16 * group; c0 < NT; c0 += 64) {
            uint32_t acc[16];
            if (has_acc) tmem_ld16(taddr + uint32_t(c0), acc);
            else {
#pragma unroll
                for (int j = 0; j < 16; ++j) acc[j] = 0u;
            }
            if (f >= p.K) continue;
#pragma unroll
            for (int j = 0; j < 16; ++j)
                if (n0 + c0 + j < p.F) prow[n0 + c0 + j] = __uint_as_float(acc[j]);
        }
    }
    mix_teardown<NT>(tmem);
}

template <int NT>
int launch_sign_t(SignTParams p, int max_split, const DeviceInfo &dev, cudaStream_t stream) {
    using S = SignTShape<NT>;
    const int mt = (p.K + kUmmaM - 1) / kUmmaM, nt = (p.F + NT - 1) / NT;
    const int64_t KB = (p.N + kMixK - 1) / kMixK;
    int64_t want = (int64_t(dev.sm_count) + int64_t(mt) * nt - 1) / (int64_t(mt) * nt);
    if (want > max_split) want = max_split;
    if (want > KB) want = KB;
    if (want < 1) want = 1;
    p.per = int((KB + want - 1) / want);
    const int splits = int((KB + p.per - 1) / p.per);
    cudaFuncSetAttribute(sign_t_real_tc_kernel<NT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                         int(S::kSmem));
    launch_kernel(sign_t_real_tc_kernel<NT>, dim3(unsigned(mt), unsigned(nt), unsigned(splits)),
                  dim3(kMixThreads), S::kSmem, stream, false, dim3(1, 1, 1), p);
    return splits;
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
    float v[8];
#pragma unroll
    for (int e = 0; e < 8; ++e) v[e] = k0 + e < K ? __ldg(Wt + (k0 + e) * ldw + j) : 0.0f;
    uint32_t h[4], m[4], l[4];
#pragma unroll
    for (int w = 0; w < 4; ++w) split3x2(v[2 * w], v[2 * w + 1], h[w], m[w], l[w]);
    uint4 *dst = reinterpret_cast<uint4 *>(wparts + int64_t(j) * kp + k0);
    const int64_t part = int64_t(F) * kp / 8;     // uint4s per part
    dst[0] = make_uint4(h[0], h[1], h[2], h[3]);
    dst[part] = make_uint4(m[0], m[1], m[2], m[3]);
    dst[2 * part] = make_uint4(l[0], l[1], l[2], l[3]);
}

template <int NT, bool kRealA>
void launch_mix(MixParams p, const DeviceInfo &dev, cudaStream_t stream, bool pdl) {
    using S = MixShape<NT, kRealA>;
    void (*kernel)(const MixParams);
    if constexpr (kRealA) kernel = real_binary_tc_kernel<NT>;
    else kernel = binary_real_tc_kernel<NT>;
    const int64_t tiles = (p.N + S::kRows - 1) / S::kRows;
    const int ctiles = (p.F + NT - 1) / NT;
    // Split the k-blocks over a cluster while the tiles leave SMs idle.
    int ks = 1;
    while (ks < kMaxSplit && ks < p.words && tiles * ctiles * (ks + 1) <= dev.sm_count) ++ks;
    p.split = ks;
    cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(S::kSmem));
    const dim3 grid(unsigned(tiles * ks), unsigned(ctiles));
    launch_kernel(kernel, grid, dim3(kMixThreads), S::kSmem, stream, pdl, dim3(unsigned(ks), 1, 1),
                  p);
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
    p.clip = g.clip;
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
    launch_mix<64, false>(p, dev, stream, pdl);
}

int launch_sign_t_real_gemm(const SignTRealArgs &a, int max_split, const DeviceInfo &dev,
                            cudaStream_t stream) {
    if (a.N == 0) return 0;
    SignTParams p{a.bits, a.words, a.alpha, a.G, a.ldg, a.N, a.K, a.F, a.partial, 0};
    if (a.F <= 64) return launch_sign_t<64>(p, max_split, dev, stream);
    if (a.F <= 128) return launch_sign_t<128>(p, max_split, dev, stream);
    return launch_sign_t<256>(p, max_split, dev, stream);
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
