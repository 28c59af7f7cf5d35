// Gather-rate probe: the ceiling of the aggregation step (Eq. 1 / Eq. 13) on
// sm_103a. The aggregation reads one row of the layer's product per CSR entry,
// at random, from a buffer that mostly sits in L2; this probe times exactly
// that access pattern without the arithmetic:
//   - LDG gathers: each warp walks its own slice of a random index array,
//     32 indices per coalesced load, broadcast by shuffles; L lanes read one
//     row in VB-byte vectors (16 or 32 bytes), U rows in flight per lane group,
//     and the loaded words are summed so that nothing is dead code;
//   - cp.async gathers: the same rows copied 16 bytes per lane into a
//     per-warp shared-memory buffer (two stages), then read back and summed;
//   - cp.async gathers into staged rows of a given pitch, plain or with the
//     16-byte chunk c of staged row r at slot c ^ (r & 7) (the layout the
//     tensor-core aggregation reads with ldmatrix), 24 warps per SM;
//   - the warp-level f16 tensor-core MMA (m16n8k16, fp32 accumulate), the
//     instruction a tensor-core form of the aggregation would issue.
// Every index lies in [0, rows) and every row lies inside the buffer, so all
// accesses stay in bounds. Throughput = bytes (or flops) / CUDA-event time,
// best of five runs. The working sets span L2-resident (<= 110 MB) and
// HBM-resident (2 GB) buffers.
#include <cstdint>
#include <cstdio>
#include <cstdlib>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#define CK(x)                                                                          \
    do {                                                                               \
        cudaError_t e_ = (x);                                                          \
        if (e_ != cudaSuccess) {                                                       \
            printf("CUDA %s at line %d\n", cudaGetErrorString(e_), __LINE__);          \
            exit(1);                                                                   \
        }                                                                              \
    } while (0)

constexpr int kThreads = 256;

// idx[i] = a hash of i reduced into [0, rows).
__global__ void fill_idx(int *idx, int64_t n, int64_t rows, uint64_t seed) {
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n;
         i += int64_t(gridDim.x) * blockDim.x) {
        uint64_t z = uint64_t(i) + seed * 0x9E3779B97F4A7C15ull;
        z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
        z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
        z ^= z >> 31;
        idx[i] = int(z % uint64_t(rows));
    }
}

__global__ void fill_buf(float *b, int64_t n) {
    for (int64_t i = blockIdx.x * int64_t(blockDim.x) + threadIdx.x; i < n;
         i += int64_t(gridDim.x) * blockDim.x)
        b[i] = float(i & 1023) * 1e-3f;
}

template <int VB> struct Ld;
template <> struct Ld<16> {
    static __device__ __forceinline__ float get(const uint8_t *p) {
        const float4 v = __ldg(reinterpret_cast<const float4 *>(p));
        return (v.x + v.y) + (v.z + v.w);
    }
};
template <> struct Ld<32> {
    static __device__ __forceinline__ float get(const uint8_t *p) {
        float a0, a1, a2, a3, a4, a5, a6, a7;
        asm volatile("ld.global.nc.v8.f32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                     : "=f"(a0), "=f"(a1), "=f"(a2), "=f"(a3), "=f"(a4), "=f"(a5), "=f"(a6),
                       "=f"(a7)
                     : "l"(p));
        return ((a0 + a1) + (a2 + a3)) + ((a4 + a5) + (a6 + a7));
    }
};

// Rows of ROWB bytes (ROWB / VB lanes each, a power of two <= 32), pitch bytes apart.
template <int VB, int ROWB, int U>
__global__ void __launch_bounds__(kThreads)
gather_ldg(const uint8_t *__restrict__ buf, int64_t pitch, const int *__restrict__ idx,
           int64_t per_warp, float *out) {
    constexpr int L = ROWB / VB;
    constexpr int P = 32 / L;
    const int lane = threadIdx.x & 31;
    const int g = lane / L, sl = lane % L;
    const int64_t warp = (int64_t(blockIdx.x) * kThreads + threadIdx.x) >> 5;
    const int *my = idx + warp * per_warp;
    float acc = 0.0f;
    for (int64_t base = 0; base < per_warp; base += 32) {
        const int j = __ldg(my + base + lane);
#pragma unroll
        for (int t = 0; t < 32; t += P * U) {
            float v[U];
#pragma unroll
            for (int u = 0; u < U; ++u) {
                const int jj = __shfl_sync(0xffffffffu, j, t + u * P + g);
                v[u] = Ld<VB>::get(buf + int64_t(jj) * pitch + sl * VB);
            }
#pragma unroll
            for (int u = 0; u < U; ++u) acc += v[u];
        }
    }
    out[blockIdx.x * kThreads + threadIdx.x] = acc;
}

__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(dst), "l"(src));
}

// cp.async gathers of 256-byte rows: a warp copies 32 rows per stage
// (2 rows per instruction), two stages in flight, then sums what landed.
constexpr int kRowB = 256;
constexpr int kStageBytes = 32 * kRowB;
__global__ void __launch_bounds__(kThreads)
gather_cpasync(const uint8_t *__restrict__ buf, int64_t pitch, const int *__restrict__ idx,
               int64_t per_warp, float *out) {
    extern __shared__ __align__(16) uint8_t smem[];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint8_t *mine = smem + wid * 2 * kStageBytes;
    const uint32_t base_s = uint32_t(__cvta_generic_to_shared(mine));
    const int64_t warp = (int64_t(blockIdx.x) * kThreads + threadIdx.x) >> 5;
    const int *my = idx + warp * per_warp;
    const int g = lane >> 4, sl = lane & 15;
    float acc = 0.0f;
    const int64_t steps = per_warp / 32;
    auto issue = [&](int64_t st) {
        const int j = __ldg(my + st * 32 + lane);
        const uint32_t dst = base_s + uint32_t(st & 1) * kStageBytes;
#pragma unroll
        for (int r = 0; r < 32; r += 2) {
            const int jj = __shfl_sync(0xffffffffu, j, r + g);
            cp_async16(dst + uint32_t((r + g) * kRowB + sl * 16), buf + int64_t(jj) * pitch + sl * 16);
        }
        asm volatile("cp.async.commit_group;");
    };
    issue(0);
    for (int64_t st = 0; st < steps; ++st) {
        if (st + 1 < steps) {
            issue(st + 1);
            asm volatile("cp.async.wait_group 1;");
        } else {
            asm volatile("cp.async.wait_group 0;");
        }
        __syncwarp();
        const float4 *s = reinterpret_cast<const float4 *>(mine + (st & 1) * kStageBytes);
#pragma unroll 4
        for (int q = lane; q < kStageBytes / 16; q += 32) {
            const float4 v = s[q];
            acc += (v.x + v.y) + (v.z + v.w);
        }
        __syncwarp();
    }
    out[blockIdx.x * kThreads + threadIdx.x] = acc;
}


// cp.async gathers of ROWB-byte rows into staged rows PITCH bytes apart: a
// warp stages R rows per step in S steps' worth of buffers; chunk q = lane +
// 32 k of a step -> row q / (ROWB / 16), chunk q % (ROWB / 16), stored at slot
// chunk (SWZ = 0) or chunk ^ (row & 7) (SWZ = 1).
template <int R, int S, int ROWB, int PITCH, int SWZ>
__global__ void __launch_bounds__(kThreads)
gather_staged(const uint8_t *__restrict__ buf, const int *__restrict__ idx, int64_t per_warp,
              float *out) {
    extern __shared__ __align__(16) uint8_t smem[];
    constexpr int CH = ROWB / 16;
    constexpr int kStage = R * PITCH;
    constexpr int KCH = R * CH / 32;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    uint8_t *mine = smem + wid * S * kStage;
    const uint32_t base_s = uint32_t(__cvta_generic_to_shared(mine));
    const int64_t warp = (int64_t(blockIdx.x) * kThreads + threadIdx.x) >> 5;
    const int *my = idx + warp * per_warp;
    float acc = 0.0f;
    const int64_t steps = per_warp / R;
    auto issue = [&](int64_t st) {
        const int j = lane < R ? __ldg(my + st * R + lane) : 0;
        const uint32_t dst = base_s + uint32_t(st % S) * kStage;
#pragma unroll
        for (int k = 0; k < KCH; ++k) {
            const int q = lane + 32 * k, r = q / CH, c = q % CH;
            const int jj = __shfl_sync(0xffffffffu, j, r);
            const int slot = SWZ ? (c ^ (r & 7)) : c;
            cp_async16(dst + uint32_t(r * PITCH + slot * 16), buf + int64_t(jj) * ROWB + c * 16);
        }
        asm volatile("cp.async.commit_group;");
    };
    for (int s = 0; s < S - 1; ++s)
        if (s < steps) issue(s);
        else asm volatile("cp.async.commit_group;");
    for (int64_t st = 0; st < steps; ++st) {
        if (st + S - 1 < steps) issue(st + S - 1);
        else asm volatile("cp.async.commit_group;");
        asm volatile("cp.async.wait_group %0;" ::"n"(S - 1));
        __syncwarp();
        const float4 *s = reinterpret_cast<const float4 *>(mine + (st % S) * kStage);
#pragma unroll
        for (int q = lane; q < kStage / 16; q += 32) {
            const float4 v = s[q];
            acc += (v.x + v.y) + (v.z + v.w);
        }
        __syncwarp();
    }
    asm volatile("cp.async.wait_group 0;");
    out[blockIdx.x * kThreads + threadIdx.x] = acc;
}

// Warp-level f16 MMA m16n8k16 with fp32 accumulators: 8 independent chains.
__global__ void __launch_bounds__(kThreads) mma_f16(const uint32_t *in, float *out, int iters) {
    const int lane = threadIdx.x & 31;
    uint32_t a[4], b[2];
    for (int i = 0; i < 4; ++i) a[i] = in[(lane * 7 + i) & 255];
    for (int i = 0; i < 2; ++i) b[i] = in[(lane * 5 + i + 64) & 255];
    float d[8][4] = {};
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int q = 0; q < 8; ++q)
            asm volatile(
                "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, "
                "{%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
                : "+f"(d[q][0]), "+f"(d[q][1]), "+f"(d[q][2]), "+f"(d[q][3])
                : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
    }
    float s = 0.0f;
    for (int q = 0; q < 8; ++q) s += d[q][0] + d[q][1] + d[q][2] + d[q][3];
    out[blockIdx.x * kThreads + threadIdx.x] = s;
}

struct Ctx {
    int sms;
    uint8_t *buf;
    int *idx;
    float *out;
    cudaEvent_t e0, e1;
};

template <class F>
float best_ms(Ctx &c, F launch) {
    launch();
    CK(cudaGetLastError());
    CK(cudaDeviceSynchronize());
    float best = 1e30f;
    for (int r = 0; r < 5; ++r) {
        CK(cudaEventRecord(c.e0));
        launch();
        CK(cudaEventRecord(c.e1));
        CK(cudaEventSynchronize(c.e1));
        float ms;
        CK(cudaEventElapsedTime(&ms, c.e0, c.e1));
        if (ms < best) best = ms;
    }
    return best;
}

template <int VB, int ROWB, int U>
void run_ldg(Ctx &c, int64_t ws_bytes, int64_t nidx) {
    const int64_t pitch = ROWB;
    const int64_t rows = ws_bytes / pitch;
    int occ = 0;
    CK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, gather_ldg<VB, ROWB, U>, kThreads, 0));
    const int blocks = c.sms * occ;
    const int64_t warps = int64_t(blocks) * (kThreads / 32);
    const int64_t per_warp = (nidx / warps) / 32 * 32;
    fill_idx<<<1024, 256>>>(c.idx, warps * per_warp, rows, 17);
    const float ms = best_ms(c, [&] {
        gather_ldg<VB, ROWB, U><<<blocks, kThreads>>>(c.buf, pitch, c.idx, per_warp, c.out);
    });
    const double gathered = double(warps * per_warp) * ROWB;
    const double with_idx = gathered + double(warps * per_warp) * 4;
    printf("ldg   row %4d B  vec %2d B  U %d  set %7.1f MB  blocks/SM %d: %8.3f ms  gathered %7.0f GB/s"
           "  (+index %7.0f GB/s)  %.2f G rows/s\n",
           ROWB, VB, U, ws_bytes / 1e6, occ, ms, gathered / ms / 1e6, with_idx / ms / 1e6,
           double(warps * per_warp) / ms / 1e6);
}

void run_cpasync(Ctx &c, int64_t ws_bytes, int64_t nidx) {
    const int64_t rows = ws_bytes / kRowB;
    const int smem = (kThreads / 32) * 2 * kStageBytes;
    CK(cudaFuncSetAttribute(gather_cpasync, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    int occ = 0;
    CK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, gather_cpasync, kThreads, smem));
    const int blocks = c.sms * occ;
    const int64_t warps = int64_t(blocks) * (kThreads / 32);
    const int64_t per_warp = (nidx / warps) / 32 * 32;
    fill_idx<<<1024, 256>>>(c.idx, warps * per_warp, rows, 23);
    const float ms = best_ms(c, [&] {
        gather_cpasync<<<blocks, kThreads, smem>>>(c.buf, kRowB, c.idx, per_warp, c.out);
    });
    const double gathered = double(warps * per_warp) * kRowB;
    printf("cp.async row %4d B  set %7.1f MB  blocks/SM %d: %8.3f ms  gathered %7.0f GB/s\n", kRowB,
           ws_bytes / 1e6, occ, ms, gathered / ms / 1e6);
}

template <int R, int S, int ROWB, int PITCH, int SWZ>
void run_staged(Ctx &c, int64_t ws_bytes, int64_t nidx) {
    const int64_t rows = ws_bytes / ROWB;
    const int smem = (kThreads / 32) * S * R * PITCH;
    auto k = gather_staged<R, S, ROWB, PITCH, SWZ>;
    CK(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    int occ = 0;
    CK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k, kThreads, smem));
    const int blocks = c.sms * occ;
    const int64_t warps = int64_t(blocks) * (kThreads / 32);
    const int64_t per_warp = (nidx / warps) / 32 * 32;
    fill_idx<<<1024, 256>>>(c.idx, warps * per_warp, rows, 31);
    const float ms = best_ms(c, [&] { k<<<blocks, kThreads, smem>>>(c.buf, c.idx, per_warp, c.out); });
    const double gathered = double(warps * per_warp) * ROWB;
    printf("cp.async row %4d B  staged pitch %3d B  swizzle %d  set %7.1f MB  blocks/SM %d: %8.3f ms"
           "  gathered %7.0f GB/s\n",
           ROWB, PITCH, SWZ, ws_bytes / 1e6, occ, ms, gathered / ms / 1e6);
}

int main() {
    Ctx c;
    CK(cudaDeviceGetAttribute(&c.sms, cudaDevAttrMultiProcessorCount, 0));
    int clk = 0;
    CK(cudaDeviceGetAttribute(&clk, cudaDevAttrClockRate, 0));
    const int64_t buf_bytes = int64_t(2) << 30;
    const int64_t nidx = int64_t(1) << 25;
    CK(cudaMalloc(&c.buf, buf_bytes + 4096));
    CK(cudaMalloc(&c.idx, nidx * sizeof(int)));
    CK(cudaMalloc(&c.out, int64_t(c.sms) * 64 * kThreads * sizeof(float)));
    CK(cudaEventCreate(&c.e0));
    CK(cudaEventCreate(&c.e1));
    fill_buf<<<4096, 256>>>(reinterpret_cast<float *>(c.buf), (buf_bytes + 4096) / 4);
    CK(cudaDeviceSynchronize());
    printf("SMs %d, clock attribute %d MHz, %lld random rows per run\n", c.sms, clk / 1000,
           (long long)nidx);

    const int64_t sets[] = {int64_t(16) << 20, int64_t(60) << 20, int64_t(110) << 20,
                            int64_t(2) << 30};
    for (int64_t ws : sets) {
        run_ldg<16, 16, 8>(c, ws, nidx);
        run_ldg<16, 64, 8>(c, ws, nidx);
        run_ldg<16, 128, 8>(c, ws, nidx);
        run_ldg<16, 256, 4>(c, ws, nidx);
        run_ldg<16, 256, 8>(c, ws, nidx);
        run_ldg<32, 256, 4>(c, ws, nidx);
        run_ldg<32, 256, 8>(c, ws, nidx);
        run_ldg<16, 512, 4>(c, ws, nidx);
        run_cpasync(c, ws, nidx);
    }
    // Staged layouts (two steps of 16 or 32 rows per warp, as many blocks per SM as fit).
    const int64_t ws63 = int64_t(60) << 20, ws25 = int64_t(24) << 20;
    run_staged<16, 2, 256, 256, 0>(c, ws63, nidx);
    run_staged<16, 2, 256, 272, 0>(c, ws63, nidx);
    run_staged<16, 2, 256, 256, 1>(c, ws63, nidx);
    run_staged<32, 2, 96, 112, 0>(c, ws25, nidx);
    run_staged<32, 2, 96, 128, 1>(c, ws25, nidx);

    uint32_t *in;
    CK(cudaMalloc(&in, 256 * sizeof(uint32_t)));
    CK(cudaMemset(in, 0x3c, 256 * sizeof(uint32_t)));
    int occ = 0;
    CK(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, mma_f16, kThreads, 0));
    const int iters = 4096, blocks = c.sms * occ;
    const float ms = best_ms(c, [&] { mma_f16<<<blocks, kThreads>>>(in, c.out, iters); });
    const double flops = double(blocks) * (kThreads / 32) * iters * 8 * (2.0 * 16 * 8 * 16);
    printf("mma.sync m16n8k16 f16 -> f32: %8.3f ms  %7.1f TFLOP/s  (%.0f flop/clk/SM at %d MHz)\n",
           ms, flops / ms / 1e9, flops / (ms * 1e-3) / c.sms / (clk * 1e3), clk / 1000);
    CK(cudaFree(in));
    CK(cudaFree(c.buf));
    CK(cudaFree(c.idx));
    CK(cudaFree(c.out));
    return 0;
}
