// tcgen05 building blocks shared by the tensor-core kernels: +-1 signs as
// FP8 E4M3 bytes, the 128B-swizzled K-major shared-memory operand layout and
// its descriptor, the E4M3 x E4M3 -> F32 instruction descriptor (M = 128),
// one MMA, and the tensor-memory load of the epilogue.
#pragma once

#include <cstdint>

namespace bigcn {

constexpr int kUmmaM = 128;

// Four signs (bits 0..3 of n) as four FP8 E4M3 bytes, +1 for a set bit:
// n * (1 + 2^7 + 2^14 + 2^21) moves bit i of n to bit 8i (the other partial
// products never land on a multiple of 8 below 32), and flipping the sign bit
// of -1.0 (0xB8) there gives +1.0 (0x38).
__device__ __forceinline__ uint32_t signs4_to_e4m3(uint32_t n) {
    const uint32_t spread = (n * 0x00204081u) & 0x01010101u;
    return 0xB8B8B8B8u ^ (spread << 7);
}

// Byte offset of 16-byte chunk c of row r in a 128B-swizzled K-major tile.
__device__ __forceinline__ uint32_t sw128_offset(int r, int c) {
    return uint32_t((r >> 3) * 1024 + (r & 7) * 128 + ((c ^ (r & 7)) << 4));
}

// Shared-memory matrix descriptor: K-major, 128B swizzle, 8-row groups 1024 B
// apart (stride byte offset), descriptor version 1.
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr) {
    uint64_t d = uint64_t((saddr >> 4) & 0x3FFFu);
    d |= uint64_t(1) << 16;                     // leading byte offset (unused here)
    d |= uint64_t(1024 >> 4) << 32;             // stride byte offset
    d |= uint64_t(1) << 46;                     // version
    d |= uint64_t(2) << 61;                     // swizzle: 128B
    return d;
}

// Instruction descriptor: E4M3 x E4M3 -> F32, both K-major, M = 128, N = n.
__host__ __device__ constexpr uint32_t e4m3_idesc(int n) {
    return (1u << 4) | (uint32_t(n >> 3) << 17) | (uint32_t(kUmmaM >> 4) << 24);
}

__device__ __forceinline__ void mma_e4m3(uint32_t d_tmem, uint64_t a, uint64_t b, uint32_t idesc,
                                         uint32_t accumulate) {
    asm volatile(
        "{\n.reg .pred p;\n"
        "setp.ne.b32 p, %4, 0;\n"
        "tcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n}" ::"r"(d_tmem),
        "l"(a), "l"(b), "r"(idesc), "r"(accumulate));
}

__device__ __forceinline__ void tmem_ld16(uint32_t taddr, uint32_t (&r)[16]) {
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 "
        "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]),
          "=r"(r[6]), "=r"(r[7]), "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]),
          "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

}  // namespace bigcn
