// Step 4 of the Bi-GCN layer forward (Wang et al., CVPR 2021, Eqs. 11-12) on
// the fifth-generation tensor cores (tcgen05) of sm_103a.
//
// Eq. 11's inner product of two sign vectors is a dense contraction of +-1
// values, and FP8 E4M3 represents +-1 exactly (+1 = 0x38, -1 = 0xB8): each
// CTA expands its packed bits into FP8 bytes in shared memory and lets
// tcgen05.mma (kind::f8f6f4, fp32 accumulators in tensor memory) sum the
// products. Every product is +-1 and every partial sum an integer of
// magnitude <= K < 2^24, so the fp32 accumulator holds the dot exactly:
// dot = K - 2 popc(a XOR b), the same integer the XNOR/popcount form gives.
// Elements of A at k >= K are written as 0.0, so padding adds nothing.
//
// CTA tile: 128 rows (UMMA M) x NT output columns (UMMA N = 64, 128 or 256),
// k-blocks of 128 signs (one 128-byte row of a 128B-swizzled K-major
// operand). Two shared-memory stages: while the tensor core works on one,
// the CTA's 256 threads expand the next -- each thread owns one 16-sign chunk
// position of several rows, issues all its packed-word loads for a k-block at
// once (and the next k-block's while the MMAs are issued), and turns every
// four signs into four E4M3 bytes with one multiply and three logic ops.
// A stage is reused only after the tcgen05.commit of the MMAs that read it
// has arrived on its mbarrier. With a caller's scratch for it, B's signs are
// instead expanded once per launch (expand_b_kernel) into the stage images of
// every (column tile, k-block), and thread 0 copies each k-block's image into
// its stage with one bulk copy (completion counted on a second mbarrier per
// stage) while the CTA expands only A. For 256-column tiles with pre-expanded
// weights, xnor_gemm_tc_ws_kernel (below) runs the same product with 256-row
// CTAs and separate expander, copy and MMA warps (2^20 x 8192 x 256: 2.39 ->
// 1.80 ms).
// Every mbarrier wait is bounded; a wait that runs out is counted in
// g_tc_timeouts (see bigcn_device_timeouts), the CTA skips its epilogue,
// frees its tensor memory and returns.
//
// Epilogue: warp w reads tensor-memory lanes 32w..32w+31 (its rows) with
// tcgen05.ld, converts the exact fp32 dots to integers and writes
//   Z = (alpha_i * beta_j) * dot     or, degree-scaled,
//   Z = (alpha_i / sqrt(dhat_i)) * (beta_j * dot).
#include "async.cuh"
#include "launch.cuh"
#include "tc.cuh"

namespace bigcn {

__device__ unsigned int g_tc_timeouts;

namespace {

constexpr int kTcThreads = 256;
constexpr int kTcKBytes = 128;
constexpr int kTcStages = 2;

// Epilogue of a product tile by kWarps warps: warp w reads tensor-memory lanes
// 32 (w % 4) .. (its rows) of accumulator h = (w / 4) % kHalves (rows 128 h
// on, NT columns further on) with tcgen05.ld, converts the exact fp32 dots to
// integers and writes Z (or the 16-bit dots and the row scale); the warps
// sharing rows take alternate 16-column slices. Rows of Z / dots take 16-byte
// stores when their starts are 16-byte aligned.
template <int NT, int kHalves, int kWarps, bool kDeg>
__device__ __forceinline__ void tc_epilogue(uint32_t tmem, int warp, int lane, int64_t m0, int n0,
                                            int64_t N, const float *__restrict__ alpha,
                                            const int64_t *__restrict__ rowptr,
                                            const float *__restrict__ beta, int F,
                                            float *__restrict__ Z, int64_t ldz,
                                            int32_t *__restrict__ dots,
                                            uint16_t *__restrict__ dots16, int64_t ldd16,
                                            float *__restrict__ rowscale, bool f16) {
    const bool vec_z = (ldz & 3) == 0 && (reinterpret_cast<uintptr_t>(Z) & 15) == 0;
    const bool vec_d = (F & 3) == 0 && (reinterpret_cast<uintptr_t>(dots) & 15) == 0;
    {
        constexpr int kSplit = kWarps / (4 * kHalves);     // warps sharing a row
        const int quad = warp & 3;
        const int hsel = (warp >> 2) % kHalves;
        const int cs = warp / (4 * kHalves);
        const int64_t row = m0 + kUmmaM * hsel + 32 * quad + lane;
        float ai = 0.0f;
        if (row < N) {
            ai = __ldg(alpha + row);
            if (kDeg) ai *= inv_sqrt_degree(__ldg(rowptr + row + 1) - __ldg(rowptr + row));
        }
        const uint32_t taddr = tmem + (uint32_t(32 * quad) << 16) + uint32_t(hsel * NT);
        if (dots16 != nullptr && row < N && n0 == 0 && cs == 0) rowscale[row] = ai;
#pragma unroll 1
        for (int c0 = 16 * cs; c0 < NT; c0 += 16 * kSplit) {
            uint32_t acc[16];
            tmem_ld16(taddr + uint32_t(c0), acc);
            if (row >= N) continue;
            const int col0 = n0 + c0;
            if (dots16 != nullptr) {        // compressed output: 16-bit dots, 4 per store
                uint16_t *dr = dots16 + row * ldd16 + col0;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    if (col0 + 4 * q >= ldd16) break;
                    uint32_t u[4];
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const int col = col0 + 4 * q + e;
                        u[e] = encode_dot(__float2int_rn(__uint_as_float(acc[4 * q + e])), col < F,
                                          f16);
                    }
                    *reinterpret_cast<uint2 *>(dr + 4 * q) =
                        make_uint2(u[0] | (u[1] << 16), u[2] | (u[3] << 16));
                }
                continue;
            }
            float z[16];
            int d[16];
#pragma unroll
            for (int j = 0; j < 16; ++j) {
                const int col = col0 + j < F ? col0 + j : F - 1;
                d[j] = __float2int_rn(__uint_as_float(acc[j]));
                const float bj = __ldg(beta + col);
                z[j] = kDeg ? ai * (bj * float(d[j])) : (ai * bj) * float(d[j]);
            }
            float *zr = Z + row * ldz + col0;
            int32_t *dr = dots != nullptr ? dots + row * F + col0 : nullptr;
            if (vec_z && col0 + 16 <= F) {
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    reinterpret_cast<float4 *>(zr)[q] =
                        make_float4(z[4 * q], z[4 * q + 1], z[4 * q + 2], z[4 * q + 3]);
            } else {
#pragma unroll
                for (int j = 0; j < 16; ++j)
                    if (col0 + j < F) zr[j] = z[j];
            }
            if (dr != nullptr) {
                if (vec_d && col0 + 16 <= F) {
#pragma unroll
                    for (int q = 0; q < 4; ++q)
                        reinterpret_cast<int4 *>(dr)[q] =
                            make_int4(d[4 * q], d[4 * q + 1], d[4 * q + 2], d[4 * q + 3]);
                } else {
#pragma unroll
                    for (int j = 0; j < 16; ++j)
                        if (col0 + j < F) dr[j] = d[j];
                }
            }
        }
    }
}

template <int NT, bool kDeg, bool kBexp>
__global__ void __launch_bounds__(kTcThreads, NT == 256 ? 2 : 4)
xnor_gemm_tc_kernel(const uint64_t *__restrict__ A, const float *__restrict__ alpha, int64_t N,
                    const uint64_t *__restrict__ B, const float *__restrict__ beta, int F, int K,
                    int words, float *__restrict__ Z, int64_t ldz, int32_t *__restrict__ dots,
                    const int64_t *__restrict__ rowptr, uint16_t *__restrict__ dots16,
                    int64_t ldd16, float *__restrict__ rowscale, bool f16,
                    const uint8_t *__restrict__ bexp) {
    constexpr int kStageA = kUmmaM * kTcKBytes;
    constexpr int kStageB = NT * kTcKBytes;
    constexpr int kStage = kStageA + kStageB;
    constexpr int kRowsPerPass = kTcThreads / 8;         // 32: thread t owns chunk t & 7
    constexpr int kAChunks = kUmmaM / kRowsPerPass;         // 4 rows of A per thread
    constexpr int kBChunks = NT / kRowsPerPass;           // 2, 4 or 8 rows of B per thread
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bars[kTcStages];
    __shared__ __align__(8) uint64_t full[kTcStages];       // B tile landed (kBexp)
    __shared__ uint32_t tmem_base;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t m0 = int64_t(blockIdx.x) * kUmmaM;
    const int n0 = blockIdx.y * NT;
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t tile0 = (raw + 1023u) & ~1023u;          // 1024-byte aligned stages
    unsigned char *tiles = smem_raw + (tile0 - raw);

    if (warp == 0) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_addr(&tmem_base)),
                     "r"(NT));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (tid == 0) {
        for (int s = 0; s < kTcStages; ++s) {
            mbar_init(smem_addr(&bars[s]), 1);
            mbar_init(smem_addr(&full[s]), 1);
        }
        mbar_fence_init();
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base;
    grid_dependency_wait();     // the packed operands come from earlier kernels

    // Thread t expands chunk c = t & 7 (16 signs) of rows (t >> 3) + 32 q.
    const int c = tid & 7, r0 = tid >> 3;
    const int KB = (K + kTcKBytes - 1) / kTcKBytes;
    uint64_t wa[kAChunks], wb[kBChunks];
    auto load_words = [&](int kb) {
        const int k0 = kb * kTcKBytes + c * 16;
#pragma unroll
        for (int q = 0; q < kAChunks; ++q) {
            const int64_t row = m0 + r0 + kRowsPerPass * q;
            wa[q] = (row < N && k0 < K) ? __ldg(A + row * words + (k0 >> 6)) : 0ull;
        }
#pragma unroll
        for (int q = 0; q < kBChunks; ++q) {
            const int col = n0 + r0 + kRowsPerPass * q;
            wb[q] = (!kBexp && col < F && k0 < K)
                        ? __ldg(B + int64_t(col) * words + (k0 >> 6)) : 0ull;
        }
    };
    const uint8_t *btiles = kBexp ? bexp + size_t(blockIdx.y) * KB * kStageB : nullptr;
    int issued = -1, landed = -1;       // thread 0: last k-block copied / seen landing
    // 16 signs from bit `sh` of w as E4M3 bytes, zero past `valid` signs.
    auto expand = [&](uint64_t w, int sh, int valid) {
        const uint32_t bits = uint32_t(w >> sh);
        uint4 v = make_uint4(signs4_to_e4m3(bits & 15u), signs4_to_e4m3((bits >> 4) & 15u),
                             signs4_to_e4m3((bits >> 8) & 15u), signs4_to_e4m3((bits >> 12) & 15u));
        if (valid < 16) {
            uint32_t *e = reinterpret_cast<uint32_t *>(&v);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const int keep = valid - 4 * q;
                if (keep <= 0) e[q] = 0u;
                else if (keep < 4) e[q] &= (1u << (8 * keep)) - 1u;
            }
        }
        return v;
    };

    constexpr uint32_t idesc = e4m3_idesc(NT);
    bool ok = true;
    int committed = -1;          // last k-block whose MMAs were committed
    load_words(0);
    for (int kb = 0; kb < KB; ++kb) {
        const int s = kb & 1;
        if (kb >= kTcStages) {
            const bool done = mbar_wait(smem_addr(&bars[s]), uint32_t((kb - kTcStages) >> 1) & 1u);
            if (!__syncthreads_and(done)) {
                ok = false;
                break;
            }
        }
        unsigned char *sa = tiles + s * kStage;
        unsigned char *sb = sa + kStageA;
        if (kBexp && tid == 0) {    // B's tile of this k-block: one bulk copy
            const uint32_t fb = smem_addr(&full[s]);
            asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb),
                         "r"(uint32_t(kStageB))
                         : "memory");
            asm volatile(
                "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], "
                "%2, [%3];" ::"r"(smem_addr(sb)),
                "l"(btiles + size_t(kb) * kStageB), "r"(uint32_t(kStageB)), "r"(fb)
                : "memory");
            issued = kb;
        }
        const int k0 = kb * kTcKBytes + c * 16;
        const int sh = k0 & 63;
        const int valid = min(max(K - k0, 0), 16);
#pragma unroll
        for (int q = 0; q < kAChunks; ++q) {
            const int r = r0 + kRowsPerPass * q;
            const bool live = m0 + r < N && valid > 0;
            *reinterpret_cast<uint4 *>(sa + sw128_offset(r, c)) =
                live ? expand(wa[q], sh, valid) : make_uint4(0u, 0u, 0u, 0u);
        }
        if (!kBexp) {
#pragma unroll
            for (int q = 0; q < kBChunks; ++q) {
                const int r = r0 + kRowsPerPass * q;
                *reinterpret_cast<uint4 *>(sb + sw128_offset(r, c)) = expand(wb[q], sh, 16);
            }
        }
        if (kb + 1 < KB) load_words(kb + 1);      // in flight across the barrier and MMAs
        asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
        __syncthreads();
        if (kBexp) {                // B's tile has landed (bounded wait, as for the MMAs)
            bool here = true;
            if (tid == 0) {
                here = mbar_wait(smem_addr(&full[s]), uint32_t(kb >> 1) & 1u);
                if (here) landed = kb;
            }
            if (!__syncthreads_and(here)) {
                ok = false;
                break;
            }
        }
        if (tid == 0) {
            asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
            const uint32_t a0 = smem_addr(sa), b0 = smem_addr(sb);
#pragma unroll
            for (int k = 0; k < kTcKBytes / 32; ++k)
                mma_e4m3(tmem, sw128_desc(a0 + 32u * k), sw128_desc(b0 + 32u * k), idesc,
                         (kb > 0 || k > 0) ? 1u : 0u);
            asm volatile(
                "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(
                    smem_addr(&bars[s]))
                : "memory");
        }
        committed = kb;
    }
    // Every MMA issued is done once the last commit has arrived (waited for
    // even after a failed wait, so that no MMA is in flight at deallocation).
    // B copies whose landing was not seen (a wait ran out, or the loop ended
    // early) are waited for too, bounded, before the shared memory is given up.
    if (kBexp && tid == 0)
        for (int kbp = landed + 1; kbp <= issued; ++kbp)
            mbar_wait(smem_addr(&full[kbp & 1]), uint32_t(kbp >> 1) & 1u);
    bool done = true;
    if (committed >= 0)
        done = mbar_wait(smem_addr(&bars[committed & 1]), uint32_t(committed >> 1) & 1u);
    ok = __syncthreads_and(ok && done) != 0;
    if (!ok && tid == 0) atomicAdd(&g_tc_timeouts, 1u);
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");

    if (ok)
        tc_epilogue<NT, 1, kTcThreads / 32, kDeg>(tmem, warp, lane, m0, n0, N, alpha, rowptr, beta, F,
                                                  Z, ldz, dots,
                                 dots16, ldd16, rowscale, f16);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == 0)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(NT));
}

// Warp-specialised form for 256-column tiles whose weight tiles are
// pre-expanded (expand_b_kernel): a CTA of 256 rows (two M = 128 accumulators
// of 256 columns share each weight tile, all 512 TMEM columns, one CTA per
// SM) runs a three-stage ring with three roles that meet only on per-stage
// mbarriers:
//   warps 0-15  expand A's packed words (loaded two k-blocks ahead) into the
//               stage's FP8 rows (4 rows of 16 signs per thread) once the
//               stage is empty, then arrive on afull[s] (one arrival per warp);
//               they also run the epilogue;
//   warp 16     (one lane) bulk-copies the k-block's weight tile into the stage
//               as soon as it is empty (completion counted on bfull[s]) -- up to
//               two k-blocks ahead of the MMAs;
//   warp 17     (one lane) waits for afull[s] and bfull[s], issues the 8 MMAs of
//               the k-block and commits them to empty[s].
// No role waits on a CTA barrier inside the loop. Every wait is bounded; a
// wait that runs out sets `err`, the other roles stop at their next wait or
// step, and the CTA skips its epilogue (after waiting, bounded, for its copies
// and MMAs in flight) and counts the failure in g_tc_timeouts.
constexpr int kWsExpWarps = 16;
constexpr int kWsThreads = (kWsExpWarps + 2) * 32;
constexpr int kWsStages = 3;
constexpr int kWsRows = 256;
constexpr int kWsCols = 256;

constexpr size_t ws_smem() {
    return 1024 + size_t(kWsStages) * (kWsRows + kWsCols) * kTcKBytes;
}

template <bool kDeg>
__global__ void __launch_bounds__(kWsThreads, 1)
xnor_gemm_tc_ws_kernel(const uint64_t *__restrict__ A, const float *__restrict__ alpha, int64_t N,
                       const float *__restrict__ beta, int F, int K, int words,
                       float *__restrict__ Z, int64_t ldz, int32_t *__restrict__ dots,
                       const int64_t *__restrict__ rowptr, uint16_t *__restrict__ dots16,
                       int64_t ldd16, float *__restrict__ rowscale, bool f16,
                       const uint8_t *__restrict__ bexp) {
    constexpr int NT = kWsCols;
    constexpr int kStageA = kWsRows * kTcKBytes;        // two 128-row halves
    constexpr int kStageB = NT * kTcKBytes;
    constexpr int kStage = kStageA + kStageB;
    constexpr int kRowsPerPass = kWsExpWarps * 32 / 8;    // thread t owns chunk t & 7
    constexpr int kAChunks = kWsRows / kRowsPerPass;      // rows per expander thread
    constexpr int kCopyWarp = kWsExpWarps, kMmaWarp = kWsExpWarps + 1;
    extern __shared__ unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t afull[kWsStages];
    __shared__ __align__(8) uint64_t bfull[kWsStages];
    __shared__ __align__(8) uint64_t empty[kWsStages];
    __shared__ uint32_t tmem_base;
    __shared__ int err;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t m0 = int64_t(blockIdx.x) * kWsRows;
    const int n0 = blockIdx.y * NT;
    const uint32_t raw = smem_addr(smem_raw);
    const uint32_t tile0 = (raw + 1023u) & ~1023u;          // 1024-byte aligned stages
    unsigned char *tiles = smem_raw + (tile0 - raw);
    volatile int *errv = &err;

    if (warp == kMmaWarp) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                         smem_addr(&tmem_base)),
                     "r"(2 * NT));
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;");
    }
    if (tid == 0) {
        for (int s = 0; s < kWsStages; ++s) {
            mbar_init(smem_addr(&afull[s]), kWsExpWarps);
            mbar_init(smem_addr(&bfull[s]), 1);
            mbar_init(smem_addr(&empty[s]), 1);
        }
        err = 0;
        mbar_fence_init();
    }
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const uint32_t tmem = tmem_base;
    grid_dependency_wait();     // the packed operands come from earlier kernels
    const int KB = (K + kTcKBytes - 1) / kTcKBytes;

    if (warp < kWsExpWarps) {
        // Thread t expands chunk c = t & 7 (16 signs) of rows (t >> 3) + P q,
        // P = kRowsPerPass; the words of k-block kb + 2 are loaded while kb is
        // expanded (two register sets, the loop unrolled by two).
        const int c = tid & 7, r0 = tid >> 3;
        uint64_t wa0[kAChunks], wa1[kAChunks];
        auto load_words = [&](int kb, uint64_t(&wa)[kAChunks]) {
            const int k0 = kb * kTcKBytes + c * 16;
#pragma unroll
            for (int q = 0; q < kAChunks; ++q) {
                const int64_t row = m0 + r0 + kRowsPerPass * q;
                wa[q] = (row < N && k0 < K) ? __ldg(A + row * words + (k0 >> 6)) : 0ull;
            }
        };
        // Expands k-block kb from wa into its stage; false when a wait ran out
        // or another role failed.
        auto step = [&](int kb, uint64_t(&wa)[kAChunks]) -> bool {
            const int s = kb % kWsStages;
            if (kb >= kWsStages) {
                const bool done =
                    mbar_wait(smem_addr(&empty[s]), uint32_t((kb - kWsStages) / kWsStages) & 1u);
                if (!__all_sync(kFullMask, done)) {
                    *errv = 1;
                    return false;
                }
            }
            if (__any_sync(kFullMask, *errv != 0)) return false;
            unsigned char *sa = tiles + s * kStage;
            const int k0 = kb * kTcKBytes + c * 16;
            const int sh = k0 & 63;
            const int valid = min(max(K - k0, 0), 16);
#pragma unroll
            for (int q = 0; q < kAChunks; ++q) {
                const int r = r0 + kRowsPerPass * q;
                uint4 v = make_uint4(0u, 0u, 0u, 0u);
                if (m0 + r < N && valid > 0) {
                    const uint32_t bits = uint32_t(wa[q] >> sh);
                    v = make_uint4(signs4_to_e4m3(bits & 15u), signs4_to_e4m3((bits >> 4) & 15u),
                                   signs4_to_e4m3((bits >> 8) & 15u),
                                   signs4_to_e4m3((bits >> 12) & 15u));
                    if (valid < 16) {       // zeros past K
                        uint32_t *e = reinterpret_cast<uint32_t *>(&v);
#pragma unroll
                        for (int p = 0; p < 4; ++p) {
                            const int keep = valid - 4 * p;
                            if (keep <= 0) e[p] = 0u;
                            else if (keep < 4) e[p] &= (1u << (8 * keep)) - 1u;
                        }
                    }
                }
                *reinterpret_cast<uint4 *>(sa + sw128_offset(r, c)) = v;
            }
            if (kb + 2 < KB) load_words(kb + 2, wa);
            asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
            __syncwarp();
            if (lane == 0) mbar_arrive(smem_addr(&afull[s]));
            return true;
        };
        load_words(0, wa0);
        if (KB > 1) load_words(1, wa1);
        for (int kb = 0; kb < KB; kb += 2) {
            if (!step(kb, wa0)) break;
            if (kb + 1 < KB && !step(kb + 1, wa1)) break;
        }
    } else if (warp == kCopyWarp) {
        if (lane == 0) {
            const uint8_t *btiles = bexp + size_t(blockIdx.y) * KB * kStageB;
            int issued = -1;
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % kWsStages;
                if (kb >= kWsStages &&
                    !mbar_wait(smem_addr(&empty[s]), uint32_t((kb - kWsStages) / kWsStages) & 1u)) {
                    *errv = 1;
                    break;
                }
                if (*errv != 0) break;
                const uint32_t fb = smem_addr(&bfull[s]);
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb),
                             "r"(uint32_t(kStageB))
                             : "memory");
                asm volatile(
                    "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], "
                    "%2, [%3];" ::"r"(smem_addr(tiles + s * kStage + kStageA)),
                    "l"(btiles + size_t(kb) * kStageB), "r"(uint32_t(kStageB)), "r"(fb)
                    : "memory");
                issued = kb;
            }
            // Copies still in flight (at most one a stage) land before the
            // shared memory is given up.
            for (int kbp = max(0, issued - kWsStages + 1); kbp <= issued; ++kbp)
                mbar_wait(smem_addr(&bfull[kbp % kWsStages]), uint32_t(kbp / kWsStages) & 1u);
        }
    } else {                                            // kMmaWarp
        if (lane == 0) {
            constexpr uint32_t idesc = e4m3_idesc(NT);
            int last = -1;
            for (int kb = 0; kb < KB; ++kb) {
                const int s = kb % kWsStages;
                const uint32_t ph = uint32_t(kb / kWsStages) & 1u;
                if (!mbar_wait(smem_addr(&afull[s]), ph) || !mbar_wait(smem_addr(&bfull[s]), ph)) {
                    *errv = 1;
                    break;
                }
                if (*errv != 0) break;
                asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
                const uint32_t a0 = smem_addr(tiles + s * kStage);
                const uint32_t b0 = a0 + uint32_t(kStageA);
#pragma unroll
                for (int k = 0; k < kTcKBytes / 32; ++k)
#pragma unroll
                    for (int h = 0; h < 2; ++h)         // rows 128 h .. 128 h + 127
                        mma_e4m3(tmem + uint32_t(h * NT),
                                 sw128_desc(a0 + uint32_t(h * kUmmaM * kTcKBytes) + 32u * k),
                                 sw128_desc(b0 + 32u * k), idesc, (kb > 0 || k > 0) ? 1u : 0u);
                asm volatile(
                    "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 "
                    "[%0];" ::"r"(smem_addr(&empty[s]))
                    : "memory");
                last = kb;
            }
            // Every MMA issued is done once the last commit has arrived.
            const bool done = last < 0 || mbar_wait(smem_addr(&empty[last % kWsStages]),
                                                    uint32_t(last / kWsStages) & 1u);
            if (!done || last != KB - 1) *errv = 1;
        }
    }
    __syncthreads();
    asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
    const bool ok = *errv == 0;
    if (!ok && tid == 0) atomicAdd(&g_tc_timeouts, 1u);
    if (ok && warp < kWsExpWarps)
        tc_epilogue<NT, 2, kWsExpWarps, kDeg>(tmem, warp, lane, m0, n0, N, alpha, rowptr, beta, F, Z,
                                              ldz, dots,
                                 dots16, ldd16, rowscale, f16);
    asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
    __syncthreads();
    if (warp == kMmaWarp)
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem),
                     "r"(2 * NT));
}

// B's signs as the product's FP8 tiles: tile (n-tile y, k-block kb) is NT
// rows (columns n0 + r of W, zero rows past F) x 128 signs (zero past K) in
// the 128B-swizzled layout of a stage, NT * 128 bytes, tiles in (y, kb) order.
template <int NT>
__global__ void __launch_bounds__(kTcThreads)
expand_b_kernel(const uint64_t *__restrict__ B, int F, int K, int words, int KB,
                uint8_t *__restrict__ out) {
    grid_dependency_wait();     // the packed columns come from the previous kernel
    const int tile = blockIdx.x;
    const int y = tile / KB, kb = tile % KB;
    uint8_t *dst = out + size_t(tile) * NT * kTcKBytes;
    for (int q = threadIdx.x; q < NT * 8; q += kTcThreads) {
        const int r = q >> 3, c = q & 7;
        const int col = y * NT + r;
        const int k0 = kb * kTcKBytes + c * 16;
        uint4 v = make_uint4(0u, 0u, 0u, 0u);
        if (col < F && k0 < K) {
            const uint32_t bits = uint32_t(__ldg(B + int64_t(col) * words + (k0 >> 6)) >> (k0 & 63));
            v = make_uint4(signs4_to_e4m3(bits & 15u), signs4_to_e4m3((bits >> 4) & 15u),
                           signs4_to_e4m3((bits >> 8) & 15u), signs4_to_e4m3((bits >> 12) & 15u));
            const int valid = K - k0;
            if (valid < 16) {
                uint32_t *e = reinterpret_cast<uint32_t *>(&v);
#pragma unroll
                for (int p = 0; p < 4; ++p) {
                    const int keep = valid - 4 * p;
                    if (keep <= 0) e[p] = 0u;
                    else if (keep < 4) e[p] &= (1u << (8 * keep)) - 1u;
                }
            }
        }
        *reinterpret_cast<uint4 *>(dst + sw128_offset(r, c)) = v;
    }
}

int tc_nt(int F) { return F <= 64 ? 64 : F <= 128 ? 128 : 256; }

template <int NT, bool kBexp = false>
size_t tc_smem() {
    return 1024 + size_t(kTcStages) * (kUmmaM * kTcKBytes + NT * kTcKBytes);
}

template <int NT, bool kDeg, bool kBexp>
void launch_nt2(const GemmArgs &g, cudaStream_t s, bool pdl) {
    const size_t smem = tc_smem<NT, kBexp>();
    auto kernel = xnor_gemm_tc_kernel<NT, kDeg, kBexp>;
    cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    const dim3 grid(unsigned((g.N + kUmmaM - 1) / kUmmaM), unsigned((g.F + NT - 1) / NT));
    if (kBexp) {
        const int KB = (g.K + kTcKBytes - 1) / kTcKBytes;
        launch_kernel(expand_b_kernel<NT>, dim3(grid.y * unsigned(KB)), dim3(kTcThreads), 0, s,
                      pdl, dim3(1, 1, 1), g.B, g.F, g.K, g.words, KB, g.b_e4m3);
    }
    launch_kernel(kernel, grid, dim3(kTcThreads), smem, s, pdl || kBexp, dim3(1, 1, 1), g.A,
                  g.alpha, g.N, g.B, g.beta, g.F, g.K, g.words, g.Z, g.ldz, g.dots, g.rowptr,
                  g.dots16, g.ldd16, g.rowscale, g.dots_f16, static_cast<const uint8_t *>(g.b_e4m3));
}

template <bool kDeg>
void launch_ws(const GemmArgs &g, cudaStream_t s, bool pdl) {
    const size_t smem = ws_smem();
    auto kernel = xnor_gemm_tc_ws_kernel<kDeg>;
    cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    const dim3 grid(unsigned((g.N + kWsRows - 1) / kWsRows), unsigned((g.F + kWsCols - 1) / kWsCols));
    const int KB = (g.K + kTcKBytes - 1) / kTcKBytes;
    launch_kernel(expand_b_kernel<kWsCols>, dim3(grid.y * unsigned(KB)), dim3(kTcThreads), 0, s,
                  pdl, dim3(1, 1, 1), g.B, g.F, g.K, g.words, KB, g.b_e4m3);
    launch_kernel(kernel, grid, dim3(kWsThreads), smem, s, true, dim3(1, 1, 1), g.A, g.alpha, g.N,
                  g.beta, g.F, g.K, g.words, g.Z, g.ldz, g.dots, g.rowptr, g.dots16, g.ldd16,
                  g.rowscale, g.dots_f16, static_cast<const uint8_t *>(g.b_e4m3));
}

template <int NT, bool kDeg>
void launch_nt(const GemmArgs &g, cudaStream_t s, bool pdl) {
    const bool bexp = g.b_e4m3 != nullptr && xnor_gemm_tc_bexp_bytes(g.K, g.F) > 0;
    if (NT == 256 && bexp) launch_ws<kDeg>(g, s, pdl);   // warp-specialised, 256-row CTAs
    else if (bexp) launch_nt2<NT, kDeg, true>(g, s, pdl);
    else launch_nt2<NT, kDeg, false>(g, s, pdl);
}

template <bool kDeg>
void launch_deg(const GemmArgs &g, cudaStream_t s, bool pdl) {
    if (g.F <= 64) launch_nt<64, kDeg>(g, s, pdl);
    else if (g.F <= 128) launch_nt<128, kDeg>(g, s, pdl);
    else launch_nt<256, kDeg>(g, s, pdl);
}

}  // namespace

size_t xnor_gemm_tc_bexp_bytes(int K, int F) {
    // Expanding W once pays where its share of the per-k-block expansion is
    // large (256-column tiles) and the k-blocks are many; measured on 2^20
    // rows: K = 8192, F = 256: 3637 -> 2773 us; K = 512, F = 64: 168 -> 232 us.
    if (K < 128 || F < 32 || !((F > 128 && K >= 1024) || K >= 4096)) return 0;
    const int NT = tc_nt(F);
    return size_t((F + NT - 1) / NT) * size_t((K + kTcKBytes - 1) / kTcKBytes) * size_t(NT) *
           kTcKBytes;
}

bool xnor_gemm_tc_supported(int64_t N, int K, int F, const DeviceInfo &dev) {
    // Enough 128-row tiles to give every SM one, and shared memory for two stages.
    return K >= 128 && F >= 32 && (N + kUmmaM - 1) / kUmmaM >= dev.sm_count &&
           size_t(dev.max_smem_optin) >= ws_smem();
}

void launch_xnor_gemm_tc(const GemmArgs &g, const DeviceInfo &, cudaStream_t stream, bool pdl) {
    if (g.N == 0) return;
    if (g.rowptr != nullptr) launch_deg<true>(g, stream, pdl);
    else launch_deg<false>(g, stream, pdl);
}

}  // namespace bigcn

extern "C" int32_t bigcn_device_timeouts(void) {
    unsigned int n = 0;
    const unsigned int zero = 0;
    if (cudaDeviceSynchronize() != cudaSuccess ||
        cudaMemcpyFromSymbol(&n, bigcn::g_tc_timeouts, sizeof(n)) != cudaSuccess ||
        cudaMemcpyToSymbol(bigcn::g_tc_timeouts, &zero, sizeof(zero)) != cudaSuccess) {
        cudaGetLastError();
        return -1;
    }
    const uint32_t mix = bigcn::take_mix_timeouts();
    if (mix == ~0u) return -1;
    return int32_t(n + mix);
}
