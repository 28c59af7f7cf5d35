// Instruction-rate probe for the XNOR-popcount product on sm_103a: the
// CUDA-core POPC rate against warp-level mma.sync m16n8k256 on 1-bit
// operands (xor.popc and and.popc). It first checks the b1 fragment layout
// against a host popcount on one 16 x 8 x 256 tile, then times each form with
// every SM running 32 warps of independent instruction chains.
#include <cstdio>
#include <cstdint>
#include <cstdlib>
#include <vector>
#include <cuda_runtime.h>

#define CK(x) do { cudaError_t e = (x); if (e != cudaSuccess) { printf("CUDA %s at %d\n", cudaGetErrorString(e), __LINE__); exit(1);} } while (0)

__device__ __forceinline__ void mma_xor(int *d, const uint32_t *a, const uint32_t *b) {
    asm volatile("mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.xor.popc "
                 "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
                 : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}
__device__ __forceinline__ void mma_and(int *d, const uint32_t *a, const uint32_t *b) {
    asm volatile("mma.sync.aligned.m16n8k256.row.col.s32.b1.b1.s32.and.popc "
                 "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};\n"
                 : "+r"(d[0]), "+r"(d[1]), "+r"(d[2]), "+r"(d[3])
                 : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b[0]), "r"(b[1]));
}

// One warp: A 16 rows x 256 bits (8 x u32 per row), B 8 cols x 256 bits.
__global__ void check_layout(const uint32_t *A, const uint32_t *B, int *D, int use_and) {
    int lane = threadIdx.x, g = lane >> 2, t = lane & 3;
    uint32_t a[4] = {A[g * 8 + t], A[(g + 8) * 8 + t], A[g * 8 + 4 + t], A[(g + 8) * 8 + 4 + t]};
    uint32_t b[2] = {B[g * 8 + t], B[g * 8 + 4 + t]};
    int d[4] = {0, 0, 0, 0};
    if (use_and) mma_and(d, a, b); else mma_xor(d, a, b);
    D[g * 8 + 2 * t] = d[0]; D[g * 8 + 2 * t + 1] = d[1];
    D[(g + 8) * 8 + 2 * t] = d[2]; D[(g + 8) * 8 + 2 * t + 1] = d[3];
}

__global__ void bench_mma(const uint32_t *in, int *out, int iters, int use_and) {
    int lane = threadIdx.x & 31;
    uint32_t a[4], b[2];
    for (int i = 0; i < 4; ++i) a[i] = in[(lane * 7 + i) & 255];
    for (int i = 0; i < 2; ++i) b[i] = in[(lane * 5 + i + 64) & 255];
    int d[8][4] = {};
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int q = 0; q < 8; ++q) {
            if (use_and) mma_and(d[q], a, b); else mma_xor(d[q], a, b);
        }
    }
    int s = 0;
    for (int q = 0; q < 8; ++q) s += d[q][0] + d[q][1] + d[q][2] + d[q][3];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

__global__ void bench_popc(const uint32_t *in, int *out, int iters) {
    uint32_t x[8];
    for (int i = 0; i < 8; ++i) x[i] = in[(threadIdx.x + i * 33) & 255];
    int acc[8] = {};
    for (int it = 0; it < iters; ++it) {
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[q] += __popc(x[q] ^ (uint32_t)it);
    }
    int s = 0;
    for (int q = 0; q < 8; ++q) s += acc[q];
    out[blockIdx.x * blockDim.x + threadIdx.x] = s;
}

int main() {
    int sms = 0; CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0));
    int clk = 0; CK(cudaDeviceGetAttribute(&clk, cudaDevAttrClockRate, 0));
    printf("SMs %d, clock attr %d kHz\n", sms, clk);
    // layout check
    std::vector<uint32_t> hA(16 * 8), hB(8 * 8);
    srand(1);
    for (auto &v : hA) v = (uint32_t(rand()) << 16) ^ uint32_t(rand());
    for (auto &v : hB) v = (uint32_t(rand()) << 16) ^ uint32_t(rand());
    uint32_t *dA, *dB; int *dD;
    CK(cudaMalloc(&dA, hA.size() * 4)); CK(cudaMalloc(&dB, hB.size() * 4)); CK(cudaMalloc(&dD, 128 * 4));
    CK(cudaMemcpy(dA, hA.data(), hA.size() * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(dB, hB.data(), hB.size() * 4, cudaMemcpyHostToDevice));
    for (int use_and = 0; use_and < 2; ++use_and) {
        check_layout<<<1, 32>>>(dA, dB, dD, use_and);
        CK(cudaGetLastError()); CK(cudaDeviceSynchronize());
        std::vector<int> hD(128);
        CK(cudaMemcpy(hD.data(), dD, 512, cudaMemcpyDeviceToHost));
        int bad = 0;
        for (int i = 0; i < 16; ++i) for (int j = 0; j < 8; ++j) {
            int ref = 0;
            for (int w = 0; w < 8; ++w) ref += __builtin_popcount(use_and ? (hA[i * 8 + w] & hB[j * 8 + w]) : (hA[i * 8 + w] ^ hB[j * 8 + w]));
            if (ref != hD[i * 8 + j]) ++bad;
        }
        printf("layout check %s: %d mismatches of 128\n", use_and ? "and.popc" : "xor.popc", bad);
    }
    // throughput
    uint32_t *din; int *dout;
    CK(cudaMalloc(&din, 256 * 4)); CK(cudaMemcpy(din, hA.data(), 128 * 4, cudaMemcpyHostToDevice));
    CK(cudaMemcpy(din + 128, hA.data(), 128 * 4, cudaMemcpyHostToDevice));
    int blocks = sms * 4, threads = 256;
    CK(cudaMalloc(&dout, blocks * threads * 4));
    cudaEvent_t e0, e1; cudaEventCreate(&e0); cudaEventCreate(&e1);
    for (int use_and = 0; use_and < 2; ++use_and) {
        int iters = 2048;
        bench_mma<<<blocks, threads>>>(din, dout, 16, use_and);
        CK(cudaDeviceSynchronize());
        cudaEventRecord(e0);
        bench_mma<<<blocks, threads>>>(din, dout, iters, use_and);
        cudaEventRecord(e1); CK(cudaEventSynchronize(e1));
        float ms; cudaEventElapsedTime(&ms, e0, e1);
        double mmas = double(blocks) * (threads / 32) * iters * 8;
        double bitmac = mmas * 16 * 8 * 256;
        printf("mma b1 %s: %.3f ms, %.1f T bit-MAC/s, %.0f bit-MAC/clk/SM at attr clock\n",
               use_and ? "and" : "xor", ms, bitmac / ms / 1e9, bitmac / (ms * 1e-3) / sms / (clk * 1e3));
    }
    {
        int iters = 8192;
        bench_popc<<<blocks, threads>>>(din, dout, 16);
        CK(cudaDeviceSynchronize());
        cudaEventRecord(e0);
        bench_popc<<<blocks, threads>>>(din, dout, iters);
        cudaEventRecord(e1); CK(cudaEventSynchronize(e1));
        float ms; cudaEventElapsedTime(&ms, e0, e1);
        double pops = double(blocks) * threads * iters * 8;
        printf("popc32: %.3f ms, %.2f T popc/s = %.1f T bit-ops/s, %.1f popc/clk/SM at attr clock\n",
               ms, pops / ms / 1e9, 32 * pops / ms / 1e9, pops / (ms * 1e-3) / sms / (clk * 1e3));
    }
    return 0;
}
