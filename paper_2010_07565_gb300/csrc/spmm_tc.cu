// Step 5 of the Bi-GCN layer (Eq. 13 with the operator of Eq. 1) on the
// tensor cores, for a product kept factored as exact integer dots:
//
//   H_if = c_f * (1/sqrt(dhat_i)) * sum_{j in N(i) u {i}} s_j * dot_jf
//
// with s_j = alpha_j / sqrt(dhat_j) the row scale and c_f = beta_f the column
// scale of Eqs. 11-12. The dots are stored as fp16 (exact: |dot| <= K <= 2048)
// in rows of 16 * FT features (padding features hold zero dots).
//
// Why tensor cores: the aggregation reads one row of dots per CSR entry. Done
// on CUDA cores, every gathered dot costs a decode and an FMA, and the kernel
// is bound by instruction issue well below what L2 delivers to random row
// gathers. Here the sum over a run of 16 CSR entries is one
// mma.sync.m16n8k16 per 16 features: A = the 16 gathered rows (features x
// entries, read from shared memory with ldmatrix.trans), B = the entries'
// weights s_j, D = fp32 accumulators. The MMA consumes the fp16 dots as they
// are, so no decode instruction remains.
//
// B carries the weights as two fp16 parts, hi = fp16(s' ) and lo = fp16(s' -
// hi) with s' = s_j * 2^(14 - E) (an exact power-of-two scaling that puts the
// row's largest weight just below 2^15), so the product keeps 22 bits of each
// weight; hi and lo land in separate accumulator columns and are added in
// fp32 at the end. E is the largest exponent among the weights seen so far for
// that output row: when a later entry raises it, the row's accumulators are
// multiplied by the exact power of two that keeps them consistent.
//
// A warp takes a window of up to 4 consecutive output rows: their lists
// (self entry first, then the CSR neighbours) are walked as one stream of
// positions, 16 at a time, and output row r of the window owns B columns
// 2r (hi) and 2r + 1 (lo). Lane (g, t) of the MMA's fragment layout then
// holds row t's sums for features 16 T + g and 16 T + g + 8 of every tile T.
// Gathered rows are staged by cp.async (16 bytes per copy; positions past the
// end of the stream and out-of-range column indices copy zeros and carry zero
// weight) in a per-warp ring of two (or three) blocks, XOR-swizzled so that
// ldmatrix reads are free of bank conflicts without padding the rows: the
// copies of the next block(s) are in flight while block n is multiplied, and
// the column indices, copied two blocks further ahead, and the row scales go
// through shared memory too, so the loop never waits on a register loaded
// from global memory.
//
// Rows with more than `heavy_degree` neighbours are each walked by all 8 warps
// of one block, whose fp32 partial rows are added in warp order
// (deterministic); light windows go one per warp, or, when there are many,
// in turn to the warps of one wave of persistent blocks that first walk the
// heavy rows.
#include <cuda_fp16.h>

#include "launch.cuh"

namespace bigcn {
namespace {

constexpr int kTcThreads = 256;
constexpr int kTcWarps = kTcThreads / 32;
constexpr int kTcRows = 4;          // output rows per light window

// Entries per block: 32 for narrow rows in one-row windows (every lane owns
// an entry, and the per-block work -- index copies, waits, scales, B
// fragments -- covers twice the entries; two MMA k-steps per block; layer 2 on
// the Reddit-shaped graph: 2.04 -> 1.93 ms), else 16 (wide rows would leave one
// block per SM; in four-row windows 32 was measured slower: 835 -> 1215 us on
// 2^20 nodes of mean degree 16).
constexpr int tc_entries_per_block(int FT, int ROWS) { return ROWS == 1 && FT <= 4 ? 32 : 16; }

template <int FT, int NSTAGES, int EBLOCK>
struct TcGeom {
    static constexpr int FP = 16 * FT;             // features per staged row
    static constexpr int CH = 2 * FT;              // 16-byte copies per row
    // Bytes per staged row: the row's 32 FT bytes rounded up to a multiple of
    // 128, its 16-byte chunk c stored at slot c ^ (r & 7) of staged row r. The
    // eight rows an ldmatrix reads then fall in eight different bank groups,
    // and the two halves of every 32-byte sector of a gathered row stay in one
    // aligned 32-byte slot pair (a padded pitch of 32 FT + 16 bytes split a
    // sector over two shared-memory lines on every other row: 256-byte rows
    // gathered at 13.7 TB/s instead of 20.6 TB/s, 96-byte rows at 8.8 instead
    // of 13.0 TB/s, 24 warps per SM).
    static constexpr int PITCH = (FP * 2 + 127) / 128 * 128;
    static constexpr int EB = EBLOCK;              // entries per block (16 or 32)
    static constexpr int KCH = EB * CH / 32;       // 16-byte row copies per lane and block
    static constexpr int STAGE = EB * PITCH;       // one block of EB entries
    static constexpr int NS = NSTAGES;             // row ring depth (blocks)
    static constexpr int D = NS - 1;               // blocks of rows copied ahead
    static constexpr int DI = 2;                   // groups between a block's index copy and its row copy
    static constexpr int NI = DI + 1;              // index slots
    // one warp's ring: NS row stages, NS x EB row scales, NI x EB column
    // indices (a multiple of 128 bytes, so that every stage starts on a
    // 128-byte line)
    static constexpr int WARP = (NS * STAGE + NS * EB * 4 + NI * EB * 4 + 127) / 128 * 128;
};

__device__ __forceinline__ uint32_t smem_addr(const void *p) {
    return uint32_t(__cvta_generic_to_shared(p));
}

// 16-byte global -> shared copy; copies zeros when `live` is false.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, bool live) {
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src),
                 "r"(live ? 16 : 0)
                 : "memory");
}
__device__ __forceinline__ void cp_async_commit() {
    asm volatile("cp.async.commit_group;" ::: "memory");
}
template <int N>
__device__ __forceinline__ void cp_async_wait() {
    asm volatile("cp.async.wait_group %0;" ::"n"(N) : "memory");
}

__device__ __forceinline__ void ldsm_x4_trans(uint32_t addr, uint32_t (&r)[4]) {
    asm volatile("ldmatrix.sync.aligned.m8n8.x4.trans.shared.b16 {%0,%1,%2,%3}, [%4];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3])
                 : "r"(addr)
                 : "memory");
}

__device__ __forceinline__ void mma_16816(float (&d)[4], const uint32_t (&a)[4], uint32_t b0,
                                          uint32_t b1) {
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, "
        "{%8,%9}, {%0,%1,%2,%3};"
        : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
        : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// 2^e as a float for e in [-126, 127].
__device__ __forceinline__ float exp2i(int e) { return __int_as_float((e + 127) << 23); }

// Unbiased exponent of a non-negative float's bits (-127 for zero and subnormals).
__device__ __forceinline__ int exponent_of(uint32_t bits) { return int(bits >> 23) - 127; }

constexpr int kNoScale = -126;      // exponent of a row that has seen no weight yet

struct TcParams {
    const int64_t *rowptr;
    const int32_t *colidx;
    int64_t N;
    int64_t nnz;
    const uint16_t *D;       // N x ldd fp16 dots
    int64_t ldd;             // halves; a multiple of 8, >= 16 * FT
    const float *rowscale;   // s_j
    int64_t heavy_degree;    // rows with more neighbours are walked by whole blocks
    bool off32;              // N * ldd * 2 < 2^32: row byte offsets fit 32 bits
    int f_base;              // first feature of this launch (column slab y: f_base + 16 FT y)
    int heavy_blocks;        // blocks [0, heavy_blocks) walk the heavy rows
    int light_first;         // blocks [light_first, grid) walk the light windows
};

// A window: up to ROWS output rows, each contributing the list entries
// [q0, q0 + len) of its list (entry 0 = the self-loop, entry q > 0 = CSR
// neighbour q - 1), laid out one after the other as positions. Position p of
// row r is the row's self-loop when p == selfp[r], else CSR entry cbase[r] + p.
template <int ROWS>
struct Window {
    int64_t row[ROWS];       // -1: inactive (no positions)
    int64_t cbase[ROWS];
    int selfp[ROWS];
    int off[ROWS + 1];       // first position of each row; off[ROWS] = stream length
};

// a[r] for a row r known only at run time, as a chain of selects (indexing the
// array dynamically would place the window in local memory).
template <int ROWS, class T>
__device__ __forceinline__ T pick(const T *a, int r) {
    T v = a[0];
#pragma unroll
    for (int k = 1; k < ROWS; ++k)
        if (r == k) v = a[k];
    return v;
}

template <int ROWS>
__device__ __forceinline__ int tag_of(const Window<ROWS> &w, int p) {
    int r = 0;
#pragma unroll
    for (int k = 1; k < ROWS; ++k) r += int(p >= w.off[k]);
    return r;
}

// Column index of the entry at position p, or -1 (past the end, or out of range).
template <int ROWS>
__device__ __forceinline__ int fetch_col(const TcParams &P, const Window<ROWS> &w, int p) {
    if (p >= w.off[ROWS]) return -1;
    const int r = tag_of(w, p);
    const int64_t j = p == pick<ROWS>(w.selfp, r) ? pick<ROWS>(w.row, r)
                                                   : int64_t(__ldg(P.colidx + pick<ROWS>(w.cbase, r) + p));
    return (j >= 0 && j < P.N) ? int(j) : -1;
}

// Per-lane sums of a window after its walk: row t = lane & 3, features
// 16 T + g and 16 T + g + 8 (g = lane >> 2), scaled back to fp32 values.
template <int FT>
struct TcRowSums {
    float v[FT][2];
};

// Walks a window's position stream and leaves its sums in `out`. The warp's
// ring `ring` (shared, TcGeom<FT, NS, EB>::WARP bytes) is free on entry and on exit.
//
// Pipeline (blocks of EB positions; lane e = lane mod EB owns position e of a
// block; with EB = 16 lanes 16-31 repeat lanes 0-15). Group m of cp.async
// copies holds block m + D's rows and row scales and block m + D + DI's column
// indices. Iteration n first waits for group n - DI (block n + D's indices),
// issues group n -- so that its rows are in flight while the warp waits for
// block n -- then waits for group n - D (block n's rows) and multiplies. No
// register of the loop waits on a global load. Block b uses row stage b mod NS
// and index slot b mod NI.
template <int FT, int ROWS, int NS, int EBLOCK>
__device__ __forceinline__ void walk_window(const TcParams &P, const Window<ROWS> &w,
                                           uint8_t *ring, TcRowSums<FT> &out) {
    using G = TcGeom<FT, NS, EBLOCK>;
    const int lane = threadIdx.x & 31;
    const int g = lane >> 2, t = lane & 3;
    constexpr int EB = G::EB;
    const int e16 = lane & (EB - 1);        // this lane's entry of a block
    const int total = w.off[ROWS];
    const int nblk = (total + EB - 1) / EB;
    const uint32_t rows_s = smem_addr(ring);
    float *wslot = reinterpret_cast<float *>(ring + G::NS * G::STAGE);   // NS x EB scales
    int *cslot = reinterpret_cast<int *>(wslot + G::NS * EB);            // NI x EB indices
    const uint32_t wslot_s = smem_addr(wslot), cslot_s = smem_addr(cslot);
    const uint32_t n32 = uint32_t(P.N);     // N <= INT32_MAX
    // Copy plan of one block's rows: chunk q = lane + 32 k -> row q / CH, piece
    // q % CH, stored at slot piece ^ (row & 7) of the staged row. For CH a power
    // of two a lane's rows are r0 + k S (S = 32 / CH) and its slots repeat with
    // period 8 / S, so only that many destinations are kept.
    constexpr bool kPow2 = (G::CH & (G::CH - 1)) == 0;
    constexpr int kStep = kPow2 ? 32 / G::CH : 0;
    constexpr int kPer = kPow2 ? (kStep >= 8 ? 1 : 8 / kStep) : G::KCH;
    constexpr int kArr = kPow2 ? 1 : G::KCH;
    int crow[kArr], cpo[kArr];
    uint32_t cdst[kPer];
    if constexpr (kPow2) {
        const int r0 = lane / G::CH, piece = lane % G::CH;
        crow[0] = r0;
        cpo[0] = piece * 16;
#pragma unroll
        for (int m = 0; m < kPer; ++m)
            cdst[m] = uint32_t(r0 * G::PITCH + ((piece ^ ((r0 + m * kStep) & 7)) * 16));
    } else {
#pragma unroll
        for (int k = 0; k < G::KCH; ++k) {
            const int piece = (lane + 32 * k) % G::CH;
            crow[k] = (lane + 32 * k) / G::CH;
            cpo[k] = piece * 16;
            cdst[k] = uint32_t(crow[k] * G::PITCH + ((piece ^ (crow[k] & 7)) * 16));
        }
    }
    auto plan_row = [&](int k) { return kPow2 ? crow[0] + k * kStep : crow[k]; };
    auto plan_src = [&](int k) { return kPow2 ? cpo[0] : cpo[k]; };
    auto plan_dst = [&](int k) {
        return kPow2 ? cdst[k % kPer] + uint32_t(k * kStep * G::PITCH) : cdst[k];
    };
    const char *Dbytes = reinterpret_cast<const char *>(P.D) +
                         2 * (int64_t(P.f_base) + int64_t(blockIdx.y) * G::FP);
    const uint32_t row_bytes = uint32_t(P.ldd) * 2u;
    // ldmatrix addresses of this lane: matrices (entries 0-7 | 8-15) x
    // (features 0-7 | 8-15) of a tile; lane l supplies entry e = (l & 7) +
    // 8 (l >> 4), chunk c = 2 T + b with b = (l >> 3) & 1, stored at slot
    // c ^ (e & 7) = 2 (T ^ y) + (b ^ x0) with x0 = l & 1, y = (l >> 1) & 3.
    // Stages start on 128-byte lines and the row pitch is a multiple of 128,
    // so the address is ((stage + tl) ^ 32 (T & 3)) + 128 (T >> 2) with
    // tl = e PITCH + 16 (b ^ x0) + 32 y.
    constexpr int kTq = FT < 4 ? FT : 4;
    const uint32_t tl = uint32_t(((lane & 7) + 8 * (lane >> 4)) * G::PITCH +
                                 16 * (((lane >> 3) & 1) ^ (lane & 1)) + 32 * ((lane >> 1) & 3));

    // Block b's column indices -> index slot `st` (zeros for self / dead entries).
    auto copy_cols = [&](int b, int st) {
        const int p = b * EB + e16;
        const int tg = tag_of(w, p);
        const bool live = p < total && p != pick<ROWS>(w.selfp, tg);
        const int32_t *src = P.colidx + (live ? pick<ROWS>(w.cbase, tg) + p : 0);
        if (lane < EB)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(
                             cslot_s + uint32_t((st * EB + e16) * 4)),
                         "l"(src), "r"(live ? 4 : 0)
                         : "memory");
    };
    // Column of block b's entry of this lane, from its landed index slot `st`.
    auto column = [&](int b, int st) -> int {
        const int p = b * EB + e16;
        if (p >= total) return -1;
        const int tg = tag_of(w, p);
        const int j = p == pick<ROWS>(w.selfp, tg) ? int(pick<ROWS>(w.row, tg))
                                                    : cslot[st * EB + e16];
        return uint32_t(j) < n32 ? j : -1;
    };
    // A block's rows and row scales (column j per lane; -1: dead) -> stage `st`.
    // Dead entries copy zeros and read nothing (pointing them all at one real
    // row instead made that row's L2 line a hot spot: 2.7 -> 4.5 ms on the
    // Reddit-shaped graph).
    auto copy_rows = [&](int st, int j) {
        const uint32_t base = rows_s + uint32_t(st * G::STAGE);
        if (P.off32) {          // each lane's row byte offset, shuffled once per copy
            const uint32_t ro = j >= 0 ? uint32_t(j) * row_bytes : 0xffffffffu;
#pragma unroll
            for (int k = 0; k < G::KCH; ++k) {
                const uint32_t r = __shfl_sync(kFullMask, ro, plan_row(k));
                const bool live = r != 0xffffffffu;
                cp_async16(base + plan_dst(k), Dbytes + (live ? r : 0u) + plan_src(k), live);
            }
        } else {
#pragma unroll
            for (int k = 0; k < G::KCH; ++k) {
                const int jj = __shfl_sync(kFullMask, j, plan_row(k));
                cp_async16(base + plan_dst(k),
                           Dbytes + int64_t(jj >= 0 ? jj : 0) * row_bytes + plan_src(k), jj >= 0);
            }
        }
        if (lane < EB)
            asm volatile("cp.async.ca.shared.global [%0], [%1], 4, %2;" ::"r"(
                             wslot_s + uint32_t((st * EB + e16) * 4)),
                         "l"(P.rowscale + (j >= 0 ? j : 0)), "r"(j >= 0 ? 4 : 0)
                         : "memory");
    };

    float acc[FT][4];
#pragma unroll
    for (int T = 0; T < FT; ++T)
#pragma unroll
        for (int c = 0; c < 4; ++c) acc[T][c] = 0.0f;
    int E[ROWS];
#pragma unroll
    for (int r = 0; r < ROWS; ++r) E[r] = kNoScale;

    // Prologue: groups -DI .. -1 (the index copies of blocks D .. D + DI - 1;
    // from group -D on also the rows of blocks 0 .. D - 1, whose indices are
    // read directly).
#pragma unroll
    for (int m = -G::DI; m < 0; ++m) {
        if (m + G::D >= 0) copy_rows(m + G::D, fetch_col(P, w, EB * (m + G::D) + e16));
        copy_cols(m + G::D + G::DI, (m + G::D + G::DI) % G::NI);
        cp_async_commit();
    }

    int st = 0;                             // row stage of block n (n mod NS)
    int si = G::D % G::NI;                  // index slot of block n + D
    for (int n = 0; n < nblk; ++n) {
        const int stD = st == 0 ? G::NS - 1 : st - 1;       // row stage of block n + D (= n - 1)
        const int siI = si == 0 ? G::NI - 1 : si - 1;       // index slot of block n + D + DI
        cp_async_wait<G::DI - 1>();     // group n - DI: block n + D's indices
        __syncwarp();
        const int jD = column(n + G::D, si);
        __syncwarp();           // every lane has read index slot si before it is reused
        copy_rows(stD, jD);
        copy_cols(n + G::D + G::DI, siI);
        cp_async_commit();
        cp_async_wait<G::D>();          // group n - D: block n's rows and scales
        __syncwarp();

        // This block's weights and the scale exponent of each row they belong to.
        const float w0 = wslot[st * EB + e16];      // 0 for dead entries
        uint32_t b0[EB / 16], b1[EB / 16];
        if constexpr (ROWS == 1) {
            const int e = exponent_of(__reduce_max_sync(kFullMask, __float_as_uint(w0)));
            if (e > E[0]) {     // keep the sums on the row's current scale
                const float f = exp2i(max(E[0] - e, -126));
#pragma unroll
                for (int T = 0; T < FT; ++T)
#pragma unroll
                    for (int c = 0; c < 4; ++c) acc[T][c] *= f;
                E[0] = e;
            }
            const float ws = w0 * exp2i(min(14 - E[0], 127));
            const __half hi = __float2half_rn(ws);
            const __half lo = __float2half_rn(ws - __half2float(hi));
            const uint32_t pw = uint32_t(__half_as_ushort(hi)) | (uint32_t(__half_as_ushort(lo)) << 16);
            // B fragment: column 0 = hi, column 1 = lo, columns 2-7 zero; entries
            // 2t, 2t+1 (b0) and 2t+8, 2t+9 (b1).
            const uint32_t sel = g == 0 ? 0x5410u : 0x7632u;
#pragma unroll
            for (int kk = 0; kk < EB / 16; ++kk) {
                const uint32_t v0 = __shfl_sync(kFullMask, pw, 16 * kk + 2 * t);
                const uint32_t v1 = __shfl_sync(kFullMask, pw, 16 * kk + 2 * t + 1);
                const uint32_t v2 = __shfl_sync(kFullMask, pw, 16 * kk + 2 * t + 8);
                const uint32_t v3 = __shfl_sync(kFullMask, pw, 16 * kk + 2 * t + 9);
                b0[kk] = g < 2 ? __byte_perm(v0, v1, sel) : 0u;
                b1[kk] = g < 2 ? __byte_perm(v2, v3, sel) : 0u;
            }
        } else {
            const int pos = n * EB + e16;
            const int tg = pos < total ? tag_of(w, pos) : ROWS;
            const int tlo = tag_of(w, n * EB);
            const int thi = tag_of(w, min(n * EB + EB - 1, total - 1));
            bool grew = false;
            int Enew[ROWS];
#pragma unroll
            for (int r = 0; r < ROWS; ++r) {
                Enew[r] = E[r];
                if (r >= tlo && r <= thi) {
                    const int e = exponent_of(
                        __reduce_max_sync(kFullMask, tg == r ? __float_as_uint(w0) : 0u));
                    if (e > Enew[r]) {
                        Enew[r] = e;
                        grew = true;
                    }
                }
            }
            if (grew) {         // keep every row's sums on its current scale
                const float f = exp2i(max(pick<ROWS>(E, t) - pick<ROWS>(Enew, t), -126));
#pragma unroll
                for (int T = 0; T < FT; ++T)
#pragma unroll
                    for (int c = 0; c < 4; ++c) acc[T][c] *= f;
#pragma unroll
                for (int r = 0; r < ROWS; ++r) E[r] = Enew[r];
            }
            uint32_t pw = 0u;
            if (tg < ROWS) {
                const float ws = w0 * exp2i(min(14 - pick<ROWS>(E, tg), 127));
                const __half hi = __float2half_rn(ws);
                const __half lo = __float2half_rn(ws - __half2float(hi));
                pw = uint32_t(__half_as_ushort(hi)) | (uint32_t(__half_as_ushort(lo)) << 16);
            }
            // B fragment: column g = 2 r + part, entries 2t, 2t+1, 2t+8, 2t+9.
            const int sel_row = g >> 1;
            const uint32_t sel = (g & 1) ? 0x7632u : 0x5410u;
            auto pair = [&](int e) -> uint32_t {   // entries e, e + 1 of column g
                const uint32_t va = __shfl_sync(kFullMask, pw, e);
                const uint32_t vb = __shfl_sync(kFullMask, pw, e + 1);
                const int ta = __shfl_sync(kFullMask, tg, e);
                const int tb = __shfl_sync(kFullMask, tg, e + 1);
                const uint32_t h = __byte_perm(va, vb, sel);
                return (ta == sel_row ? (h & 0xffffu) : 0u) | (tb == sel_row ? (h & 0xffff0000u) : 0u);
            };
#pragma unroll
            for (int kk = 0; kk < EB / 16; ++kk) {
                b0[kk] = pair(16 * kk + 2 * t);
                b1[kk] = pair(16 * kk + 2 * t + 8);
            }
        }

        const uint32_t sl = rows_s + uint32_t(st * G::STAGE) + tl;
        uint32_t tq[kTq];
#pragma unroll
        for (int m = 0; m < kTq; ++m) tq[m] = sl ^ uint32_t(32 * m);
#pragma unroll
        for (int kk = 0; kk < EB / 16; ++kk)
#pragma unroll
            for (int T = 0; T < FT; ++T) {
                uint32_t a[4];
                ldsm_x4_trans(tq[T & 3] + uint32_t(kk * 16 * G::PITCH + 128 * (T >> 2)), a);
                mma_16816(acc[T], a, b0[kk], b1[kk]);
            }
        __syncwarp();           // stage st is refilled in iteration n + 1
        st = st == G::NS - 1 ? 0 : st + 1;
        si = si == G::NI - 1 ? 0 : si + 1;
    }
    cp_async_wait<0>();         // the ring is idle before the next window
    __syncwarp();

    const int Et = pick<ROWS>(E, t);
    const float back = exp2i(max(min(Et - 14, 127), -126));
#pragma unroll
    for (int T = 0; T < FT; ++T) {
        out.v[T][0] = (acc[T][0] + acc[T][1]) * back;
        out.v[T][1] = (acc[T][2] + acc[T][3]) * back;
    }
}

// The output rows of a walk as the epilogues see them: lane (g, t) holds the
// sums of row rows[t] (-1: none) with the normalisation dinv[t].
struct TcRows {
    int64_t row[4];
    float dinv[4];
    __device__ __forceinline__ int64_t of(int t) const {
        int64_t i = row[0];
#pragma unroll
        for (int r = 1; r < 4; ++r)
            if (t == r) i = row[r];
        return i;
    }
    __device__ __forceinline__ float dinv_of(int t) const {
        float d = dinv[0];
#pragma unroll
        for (int r = 1; r < 4; ++r)
            if (t == r) d = dinv[r];
        return d;
    }
};

// Epilogue of the plain aggregation: H_if = dinv_i * (c_f * sum_f) for f < F
// (features f0 .. f0 + 16 FT - 1 of the block's column slab), with an
// optional argmax of each row (lowest index on ties; one slab only).
template <int FT>
struct TcStore {
    float *H;
    int64_t ldh;
    int F;
    const float *colscale;   // nullable: 1
    int32_t *pred;           // nullable (one column slab only)
    int f_base;              // first feature of the launch's slab 0
    static constexpr size_t kSmemFloats = 0;
    __device__ __forceinline__ void prologue(float *) {}
    __device__ __forceinline__ void operator()(const TcRows &rows, const TcRowSums<FT> &s) const {
        const int lane = threadIdx.x & 31;
        const int g = lane >> 2, t = lane & 3;
        const int64_t i = rows.of(t);
        const float di = rows.dinv_of(t);
        const int f0 = f_base + int(blockIdx.y) * 16 * FT;
        float bestv = 0.0f;
        int best = -1;
        if (i >= 0) {
#pragma unroll
            for (int T = 0; T < FT; ++T)
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int f = f0 + 16 * T + g + 8 * h;
                    if (f < F) {
                        const float c = colscale != nullptr ? __ldg(colscale + f) : 1.0f;
                        const float o = di * (c * s.v[T][h]);
                        H[i * ldh + f] = o;
                        if (best < 0 || o > bestv) {
                            bestv = o;
                            best = f;
                        }
                    }
                }
        }
        if (pred != nullptr) {          // over the 8 lanes of the row (lane bits 2..4)
#pragma unroll
            for (int o = 4; o < 32; o <<= 1) {
                const float ov = __shfl_xor_sync(kFullMask, bestv, o);
                const int oi = __shfl_xor_sync(kFullMask, best, o);
                if (oi >= 0 && (best < 0 || ov > bestv || (ov == bestv && oi < best))) {
                    bestv = ov;
                    best = oi;
                }
            }
            if (i >= 0 && g == 0) pred[i] = best;
        }
    }
};

// Epilogue of layer 1 fused with layer 2's binarization and product: H1_i =
// dinv_i * beta1 . sums (optionally stored), its signs packed LSB-first,
// alpha2_i = mean |H1_i| (Eqs. 7-8), and the XNOR-popcount dots against W2's
// packed columns (Eqs. 11-12), stored as fp16 rows of ldd2 halves (zeros past
// Fo) with the row scale s2_i = alpha2_i * dinv_i -- layer 2's factored product.
template <int FT>
struct TcPackGemm {
    float *H1;               // nullable N x Fh (row stride ldh1)
    int64_t ldh1;
    int Fh;
    const float *beta1;      // Fh
    const uint64_t *wbits2;  // Fo x words2
    int Fo;
    int words2;              // 1 or 2
    uint16_t *D2;            // N x ldd2 fp16 dots
    int64_t ldd2;
    float *s2;               // N
    const float *sBeta1 = nullptr;     // shared copies, set by prologue()
    const uint64_t *sW2 = nullptr;

    static constexpr size_t kSmemFloats = 128 + 2 * kMaxFusedOut * 2;
    __device__ __forceinline__ void prologue(float *smem) {
        float *b1 = smem;
        uint64_t *w2 = reinterpret_cast<uint64_t *>(smem + 128);
        for (int q = threadIdx.x; q < Fh; q += kTcThreads) b1[q] = __ldg(beta1 + q);
        for (int q = threadIdx.x; q < Fo * words2; q += kTcThreads) w2[q] = __ldg(wbits2 + q);
        sBeta1 = b1;
        sW2 = w2;
    }
    __device__ __forceinline__ void operator()(const TcRows &rows, const TcRowSums<FT> &s) const {
        const int lane = threadIdx.x & 31;
        const int g = lane >> 2, t = lane & 3;
        const int64_t i = rows.of(t);
        const float di = rows.dinv_of(t);
        uint64_t w0 = 0, w1 = 0;
        float l1 = 0.0f;
#pragma unroll
        for (int T = 0; T < FT; ++T)
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int f = 16 * T + g + 8 * h;
                if (f < Fh) {
                    const float v = di * (sBeta1[f] * s.v[T][h]);
                    if (H1 != nullptr && i >= 0) H1[i * ldh1 + f] = v;
                    l1 += fabsf(v);
                    if (v >= 0.0f) {
                        if (f < 64) w0 |= 1ull << f;
                        else w1 |= 1ull << (f - 64);
                    }
                }
            }
#pragma unroll
        for (int o = 4; o < 32; o <<= 1) {     // the row's 8 lanes
            w0 |= __shfl_xor_sync(kFullMask, w0, o);
            w1 |= __shfl_xor_sync(kFullMask, w1, o);
            l1 += __shfl_xor_sync(kFullMask, l1, o);
        }
        if (i < 0) return;
        if (g == 0) s2[i] = (l1 / float(Fh)) * di;
        for (int o = g; o < ldd2; o += 8) {
            uint16_t d = 0;
            if (o < Fo) {
                int mism = __popcll(w0 ^ sW2[o * words2]);
                if (words2 > 1) mism += __popcll(w1 ^ sW2[o * words2 + 1]);
                d = __half_as_ushort(__int2half_rn(Fh - 2 * mism));
            }
            D2[i * ldd2 + o] = d;
        }
    }
};

// One light window: rows first .. first + ROWS - 1, leaving out heavy ones.
template <int FT, int ROWS, int NS, int EBLOCK, class Epi>
__device__ __forceinline__ void light_window(const TcParams &P, const Epi &epi, uint8_t *ring,
                                             int64_t first) {
    Window<ROWS> w;
    TcRows out;
    int pos = 0;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        out.row[r] = -1;
        out.dinv[r] = 0.0f;
    }
#pragma unroll
    for (int r = 0; r < ROWS; ++r) {
        const int64_t i = first + r;
        w.off[r] = pos;
        w.row[r] = -1;
        w.cbase[r] = 0;
        w.selfp[r] = -1;
        if (i < P.N) {
            const int64_t rb = __ldg(P.rowptr + i), re = __ldg(P.rowptr + i + 1);
            const int64_t b = min(max(rb, int64_t(0)), P.nnz);
            const int64_t e = min(max(re, b), P.nnz);
            const int64_t deg = e - b;
            out.row[r] = i;
            out.dinv[r] = inv_sqrt_degree(deg);
            if (deg <= P.heavy_degree) {
                w.row[r] = i;
                w.selfp[r] = pos;
                w.cbase[r] = b - pos - 1;
                pos += int(deg + 1);
            } else {
                out.row[r] = -1;    // a heavy block's row
            }
        }
    }
    w.off[ROWS] = pos;
    TcRowSums<FT> s;
    walk_window<FT, ROWS, NS, EBLOCK>(P, w, ring, s);
    epi(out, s);
}

// Heavy rows (blocks take chunks of 32 rows in turn): every warp of the block
// walks an eighth of the row's list (a one-row window), and warp 0 adds the
// eight partial rows in warp order. A warp's partial row goes to the start of
// its own ring, which is idle between walks.
template <int FT, int NS, int EBLOCK, class Epi>
__device__ __forceinline__ void heavy_rows(const TcParams &P, const Epi &epi, uint8_t *rings) {
    using G = TcGeom<FT, NS, EBLOCK>;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int g = lane >> 2, t = lane & 3;
    uint8_t *ring = rings + warp * G::WARP;
    auto part = [&](int q) { return reinterpret_cast<float *>(rings + q * G::WARP); };
    for (int64_t base = int64_t(blockIdx.x) * 32; base < P.N;
         base += int64_t(P.heavy_blocks) * 32) {
        const int64_t r = base + lane;
        bool heavy = false;
        int64_t rb = 0, deg = 0;
        if (r < P.N) {
            const int64_t a = __ldg(P.rowptr + r), e0 = __ldg(P.rowptr + r + 1);
            rb = min(max(a, int64_t(0)), P.nnz);
            deg = min(max(e0, rb), P.nnz) - rb;
            heavy = deg > P.heavy_degree;
        }
        unsigned mm = __ballot_sync(kFullMask, heavy);
        while (mm != 0u) {
            const int bit = __ffs(mm) - 1;
            mm &= mm - 1u;
            const int64_t i = base + bit;
            const int64_t cb = __shfl_sync(kFullMask, rb, bit);
            const int64_t dg = __shfl_sync(kFullMask, deg, bit);
            const int64_t span = dg + 1;
            const int64_t q0 = span * warp / kTcWarps, q1 = span * (warp + 1) / kTcWarps;
            Window<1> w;
            w.row[0] = i;
            w.selfp[0] = int(-q0);          // position of entry 0 (outside unless q0 == 0)
            w.cbase[0] = cb + q0 - 1;
            w.off[0] = 0;
            w.off[1] = int(q1 - q0);
            TcRowSums<FT> s;
            walk_window<FT, 1, NS, EBLOCK>(P, w, ring, s);
            if (t == 0) {
#pragma unroll
                for (int T = 0; T < FT; ++T) {
                    part(warp)[16 * T + g] = s.v[T][0];
                    part(warp)[16 * T + g + 8] = s.v[T][1];
                }
            }
            __syncthreads();
            if (warp == 0) {
#pragma unroll
                for (int T = 0; T < FT; ++T)
#pragma unroll
                    for (int h = 0; h < 2; ++h) {
                        float a = 0.0f;
                        for (int q = 0; q < kTcWarps; ++q) a += part(q)[16 * T + g + 8 * h];
                        s.v[T][h] = a;
                    }
                TcRows out;
                out.row[0] = i;
                out.dinv[0] = inv_sqrt_degree(dg);
#pragma unroll
                for (int k = 1; k < 4; ++k) {
                    out.row[k] = -1;
                    out.dinv[k] = 0.0f;
                }
                epi(out, s);
            }
            __syncthreads();    // the rings are walked again by the next heavy row
        }
    }
}

// Blocks per SM the kernel is compiled for: three with two-stage rings (at
// most 80 registers a thread), two with three stages.
constexpr int tc_min_blocks(int NS) { return NS == 2 ? 3 : 2; }

template <int FT, int ROWS, int NS, class Epi>
__global__ void __launch_bounds__(kTcThreads, tc_min_blocks(NS))
spmm_tc_kernel(TcParams P, Epi epi) {
    constexpr int EB = tc_entries_per_block(FT, ROWS);
    using G = TcGeom<FT, NS, EB>;
    extern __shared__ __align__(128) uint8_t smem[];
    // The rings start on a 128-byte line (the ldmatrix addressing relies on it).
    uint8_t *rings = smem + ((128u - (smem_addr(smem) & 127u)) & 127u);
    float *extra = reinterpret_cast<float *>(rings + kTcWarps * G::WARP);
    grid_dependency_wait();     // the dots and row scales come from the previous kernel
    epi.prologue(extra);
    __syncthreads();
    const int warp = threadIdx.x >> 5;
    uint8_t *ring = rings + warp * G::WARP;
    // Blocks [0, heavy_blocks) walk the heavy rows; blocks from light_first on
    // then walk light windows, warp by warp in turn. Many windows: one wave of
    // persistent blocks does both (a block per window would hold its SM until
    // its longest row ended, most of its warps idle). Few windows: a warp per
    // window, with separate leading blocks for the heavy rows.
    if (int(blockIdx.x) < P.heavy_blocks) heavy_rows<FT, NS, EB>(P, epi, rings);
    if (int(blockIdx.x) < P.light_first) return;
    const int64_t windows = (P.N + ROWS - 1) / ROWS;
    for (int64_t wi = int64_t(int(blockIdx.x) - P.light_first) * kTcWarps + warp; wi < windows;
         wi += int64_t(int(gridDim.x) - P.light_first) * kTcWarps)
        light_window<FT, ROWS, NS, EB>(P, epi, ring, wi * ROWS);
}

template <int FT, int NS, int EB>
size_t tc_smem(size_t extra_floats) {
    using G = TcGeom<FT, NS, EB>;
    static_assert(G::FP * 4 <= G::WARP, "a warp's partial row must fit its ring");
    static_assert(G::WARP % 16 == 0, "rings must keep 16-byte alignment");
    return 128 + size_t(kTcWarps) * G::WARP + extra_floats * 4;
}

// Rows per light window: one when rows are long (a window's blocks then all
// belong to one row), four for short rows (so that a block of 16 entries
// spans several rows instead of mostly padding).
int tc_rows(int64_t N, int64_t nnz) { return N > 0 && nnz >= 24 * N ? 1 : kTcRows; }

// Heavy-row threshold: rows above max(64, 4 x the mean degree) take a whole block.
int64_t tc_heavy_degree(int64_t N, int64_t nnz) {
    const int64_t mean = N > 0 ? nnz / N : 0;
    return 4 * mean > 64 ? 4 * mean : 64;
}

template <int FT, int ROWS, int NS, class Epi>
void launch_rows(const TcParams &P0, const Epi &epi, int slabs, const DeviceInfo &dev,
                 cudaStream_t s, bool pdl) {
    TcParams P = P0;
    P.heavy_degree = tc_heavy_degree(P.N, P.nnz);
    const size_t smem = tc_smem<FT, NS, tc_entries_per_block(FT, ROWS)>(Epi::kSmemFloats);
    auto kernel = spmm_tc_kernel<FT, ROWS, NS, Epi>;
    cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, int(smem));
    // One wave of resident blocks, or fewer when the windows do not need them.
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, kTcThreads, smem) !=
            cudaSuccess ||
        per_sm < 1) {
        cudaGetLastError();
        per_sm = 1;
    }
    const int64_t windows = (P.N + ROWS - 1) / ROWS;
    const int64_t need = (windows + kTcWarps - 1) / kTcWarps;
    const int64_t resident = int64_t(per_sm) * dev.sm_count;
    const int64_t chunks = (P.N + 31) / 32;
    int64_t blocks;
    if (need > 4 * resident) {          // persistent: every block does both
        blocks = resident;
        P.heavy_blocks = int(resident);
        P.light_first = 0;
    } else {                            // leading heavy blocks, then a warp per window
        const int64_t hb = chunks < 2 * int64_t(dev.sm_count) ? chunks : 2 * int64_t(dev.sm_count);
        P.heavy_blocks = int(hb);
        P.light_first = int(hb);
        blocks = hb + need;
    }
    const dim3 grid(static_cast<unsigned>(blocks), static_cast<unsigned>(slabs));
    launch_kernel(kernel, grid, dim3(kTcThreads), smem, s, pdl, dim3(1, 1, 1), P, epi);
}

template <int FT, class Epi>
void launch_ft(const TcParams &P, const Epi &epi, const DeviceInfo &dev, cudaStream_t s,
               bool pdl, int slabs = 1) {
    // Two-stage rings and three blocks (24 warps) per SM: on the Reddit-shaped
    // graph 3109 -> 3000 us (layer 1) and 1927 -> 1869 us (layer 2) against
    // three stages at two blocks per SM; four-row windows 846 -> 782 us (2^20
    // nodes of mean degree 16, 64 features). Four-row windows of more than 64
    // features keep three stages: at 80 registers they would spill.
    constexpr int kNs4 = FT <= 4 ? 2 : 3;
    if (tc_rows(P.N, P.nnz) == 1) launch_rows<FT, 1, 2>(P, epi, slabs, dev, s, pdl);
    else launch_rows<FT, kTcRows, kNs4>(P, epi, slabs, dev, s, pdl);
}

}  // namespace

bool spmm_tc_supported(int F) { return F >= 1; }

// Column slabs of 128 features (FT = 8) in one launch, then the remaining
// F mod 128 features in a second launch with as many 16-feature tiles as they
// need (or one launch of ceil(F / 16) tiles when F <= 128).
void launch_spmm_tc(const SpmmTcArgs &a, const DeviceInfo &dev, cudaStream_t s, bool pdl) {
    if (a.N == 0) return;
    TcParams P{a.rowptr, a.colidx, a.N, a.nnz, a.D, a.ldd, a.rowscale, 0,
               a.N * a.ldd * 2 < (int64_t(1) << 32), 0, 0, 0};
    const int full = a.F > 128 ? a.F / 128 : 0;
    if (full > 0) {
        launch_ft<8>(P, TcStore<8>{a.H, a.ldh, a.F, a.colscale, nullptr, 0}, dev, s, pdl, full);
        pdl = true;         // the remainder launch follows on the same stream
    }
    const int rest = a.F - 128 * full;
    if (rest == 0) return;
    P.f_base = 128 * full;
    int32_t *pred = full == 0 ? a.pred : nullptr;
    switch ((rest + 15) / 16) {
#define BIGCN_TC_CASE(ft)                                                                     \
    case ft:                                                                                  \
        launch_ft<ft>(P, TcStore<ft>{a.H, a.ldh, a.F, a.colscale, pred, P.f_base}, dev, s, pdl); \
        break;
        BIGCN_TC_CASE(1)
        BIGCN_TC_CASE(2)
        BIGCN_TC_CASE(3)
        BIGCN_TC_CASE(4)
        BIGCN_TC_CASE(5)
        BIGCN_TC_CASE(6)
        BIGCN_TC_CASE(7)
        BIGCN_TC_CASE(8)
#undef BIGCN_TC_CASE
        default: break;
    }
}

bool spmm_tc_pack_gemm_supported(int Fh, int Fo) {
    return Fh >= 1 && Fh <= 128 && Fo >= 1 && Fo <= kMaxFusedOut;
}

void launch_spmm_tc_pack_gemm(const SpmmTcPackGemmArgs &a, const DeviceInfo &dev,
                              cudaStream_t s, bool pdl) {
    if (a.N == 0) return;
    TcParams P{a.rowptr, a.colidx, a.N, a.nnz, a.D1, a.ldd1, a.s1, 0,
               a.N * a.ldd1 * 2 < (int64_t(1) << 32), 0, 0, 0};
    const int words2 = (a.Fh + 63) / 64;
    switch ((a.Fh + 15) / 16) {
#define BIGCN_TCPG_CASE(ft)                                                                 \
    case ft: {                                                                              \
        TcPackGemm<ft> e{a.H1, a.ldh1, a.Fh, a.beta1, a.wbits2, a.Fo, words2, a.D2, a.ldd2, \
                         a.s2};                                                             \
        launch_ft<ft>(P, e, dev, s, pdl);                                                   \
        break;                                                                              \
    }
        BIGCN_TCPG_CASE(1)
        BIGCN_TCPG_CASE(2)
        BIGCN_TCPG_CASE(3)
        BIGCN_TCPG_CASE(4)
        BIGCN_TCPG_CASE(5)
        BIGCN_TCPG_CASE(6)
        BIGCN_TCPG_CASE(7)
        BIGCN_TCPG_CASE(8)
#undef BIGCN_TCPG_CASE
        default: break;
    }
}

}  // namespace bigcn
