// Internal launchers of the four Bi-GCN kernels. Each entry point of
// include/bigcn.h validates its arguments and calls one of these; the fused
// layer calls them in sequence on one stream. Arguments are assumed valid.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "bigcn_internal.cuh"

namespace bigcn {

// Steps 1+2: centre, sign-pack rows, per-node scale (Sec. 6.2, Eqs. 7-8).
// `pdl`: launch with programmatic serialization (see grid_dependency_wait);
// `x_upstream`: X is written by an earlier kernel of the chain (the kernel
// then waits before reading it; otherwise it waits only before it exits).
void launch_pack_rows(const float *X, int64_t N, int K, int64_t ldx, const float *scale,
                      const float *shift, uint64_t *bits, int words, float *alpha,
                      const DeviceInfo &dev, cudaStream_t stream, bool pdl = false,
                      bool x_upstream = true);

// Step 3: sign-pack weight columns, per-column scale (Eqs. 3-4).
void launch_pack_weights(const float *Wt, int K, int F, int64_t ldw, uint64_t *bits,
                         int words, float *beta, cudaStream_t stream);

// One weight matrix to pack: W (K x F, row stride ldw) -> bits (F x words), beta.
struct WeightPack {
    const float *W;
    int K;
    int F;
    int64_t ldw;
    uint64_t *bits;
    int words;
    float *beta;
    int tiles;               // set by the launcher
};

// Step 3 for two matrices in one launch (b.W == nullptr: a only).
// The kernel lets its dependent launch at once (it is the first of a chain).
void launch_pack_weights2(const WeightPack &a, const WeightPack &b, cudaStream_t stream);

struct GemmArgs {
    const uint64_t *A;       // N x words packed node rows
    const float *alpha;      // N per-node scales
    int64_t N;
    const uint64_t *B;       // F x words packed weight columns
    const float *beta;       // F per-column scales
    int F;
    int K;
    int words;
    float *Z;                // N x F (row stride ldz)
    int64_t ldz;
    int32_t *dots;           // nullable N x F raw dots (row stride F)
    const int64_t *rowptr;   // nullable: scale row i by 1/sqrt(1 + deg_i)
    // Compressed output (nullable; replaces Z): dots + 32768 as uint16 (row
    // stride ldd16, a multiple of 4 >= F, padding columns hold 32768, i.e. 0),
    // and each row's scale alpha_i (times 1/sqrt(1 + deg_i) with rowptr) in
    // rowscale; Z[i,j] is then rowscale_i * beta_j * dot[i,j]. Needs K <= 32767.
    uint16_t *dots16 = nullptr;
    int64_t ldd16 = 0;
    float *rowscale = nullptr;
    // With dots_f16 the compressed dots are fp16 bits instead (exact for
    // K <= 2048), padding columns zero: the input of launch_spmm_tc.
    bool dots_f16 = false;
    // Nullable device scratch of xnor_gemm_tc_bexp_bytes(K, F) bytes (16-byte
    // aligned): the tensor-core product then expands B's signs to FP8 once
    // into it, and each CTA copies its tiles instead of expanding them.
    uint8_t *b_e4m3 = nullptr;
};

// Bytes of the pre-expanded B of the tensor-core product (0 when it would
// not be used for these widths).
size_t xnor_gemm_tc_bexp_bytes(int K, int F);

// Step 4 on the tensor cores (xnor_gemm_tc.cu): +-1 signs as FP8 E4M3,
// tcgen05.mma with fp32 accumulators in tensor memory. Used by
// launch_xnor_gemm when K >= 128, F >= 32 and N gives every SM a 128-row tile.
bool xnor_gemm_tc_supported(int64_t N, int K, int F, const DeviceInfo &dev);
struct GemmArgs;
void launch_xnor_gemm_tc(const GemmArgs &args, const DeviceInfo &dev, cudaStream_t stream,
                         bool pdl);

// Step 4: the XNOR-popcount product and its scaling (Eqs. 11-12).
void launch_xnor_gemm(const GemmArgs &args, const DeviceInfo &dev, cudaStream_t stream,
                      bool pdl = false);

// Aggregators of step 5: Eq. 1's D^-1/2 (A + I) D^-1/2, the mean over
// N(i) u {i} (inductive GCN), GraphSAGE's self + mean over N(i), and Eq. 1's
// operator on a weighted A (Sec. 3: entries a_ij, D^_ii = 1 + sum_j a_ij).
enum : int { kAggGcn = 0, kAggMean = 1, kAggSage = 2, kAggWeighted = 3 };

struct SpmmArgs {
    const int64_t *rowptr;   // N + 1
    const int32_t *colidx;   // nnz
    int64_t N;
    int64_t nnz;
    const float *Z;          // N x F (row stride ldz)
    int64_t ldz;
    int F;
    float *H;                // N x F (row stride ldh)
    int64_t ldh;
    bool prescaled;          // Z rows already carry their 1/sqrt(dhat_j)
    bool z_pad4;             // Z's columns F .. round_up(F, 4) are readable and finite
    // Compressed input (nullable; replaces Z): rows of dots + 32768 as uint16
    // (row stride ldz, a multiple of 4; padding columns hold 32768), with
    // Z[j,f] = rowscale_j * colscale_f * dot[j,f] and rowscale_j already
    // including 1/sqrt(dhat_j).
    const uint16_t *D16 = nullptr;
    const float *rowscale = nullptr;
    const float *colscale = nullptr;
    // Nullable: receives each output row's argmax (lowest index on ties),
    // in the aggregation's epilogue when a row fits one column slab, else
    // by a separate kernel.
    int32_t *pred = nullptr;
    // Aggregator: kAggGcn (Eq. 1, the default), kAggMean (the mean over
    // N(i) u {i}: pass prescaled rows carrying no degree factor, or dots with
    // rowscale = alpha) or kAggSage (Zs[i] + the mean over N(i) of Z[j]: Z /
    // D16 point at the neighbour half of each row, Zs at the self half with
    // the same stride, colscale_s its column scales for dots).
    int agg = kAggGcn;
    const void *Zs = nullptr;
    const float *colscale_s = nullptr;
    // Rows of Z when they differ from the N output rows (a shard's own rows
    // followed by its halo rows): column indices must lie below it. 0: N.
    // Needs pre-scaled rows or dots with a row scale (no neighbour degree is read).
    int64_t ncols = 0;
    // kAggWeighted: the weight a_ij of each CSR entry (nnz) and every node's
    // 1/sqrt(dhat) (N, from launch_weighted_dinv). fp32 rows (prescaled
    // false) are weighted by a_ij dinv_j, dots by a_ij rowscale_j (rowscale
    // carrying dinv_j); the sum is multiplied by dinv_i.
    const float *values = nullptr;
    const float *dinv = nullptr;
};

// Step 5: H = D^-1/2 (A + I) D^-1/2 Z (Eqs. 1, 13); launches one kernel, or
// two when an argmax is asked for rows wider than one column slab.
void launch_spmm_norm(const SpmmArgs &args, const DeviceInfo &dev, cudaStream_t stream,
                      bool pdl = false);
// The weighted degrees of A + I (weighted.cu): dinv_i = 1/sqrt(1 + sum of
// row i's values) and, when alpha is given, s_i = alpha_i dinv_i.
void launch_weighted_dinv(const int64_t *rowptr, const float *values, int64_t N, int64_t nnz,
                          const float *alpha, float *dinv, float *s, cudaStream_t stream);

struct FrontArgs {
    const float *X;          // N x K (row stride ldx)
    int64_t N;
    int K;
    int64_t ldx;
    const float *scale;      // nullable (identity centring)
    const float *shift;
    const uint64_t *wbits;   // F x words packed weight columns
    const float *beta;       // F
    int F;
    int words;
    const int64_t *rowptr;   // nullable: rows are scaled by 1/sqrt(1 + deg)
    float *Z;                // N x F (row stride ldz)
    int64_t ldz;
    // Compressed output (nullable; replaces Z), as in GemmArgs: dots + 32768
    // as uint16 (row stride ldd16, a multiple of 4 >= F, padding = 32768) and
    // the row scale alpha_i / sqrt(1 + deg_i). Needs K <= 32767.
    uint16_t *D16 = nullptr;
    int64_t ldd16 = 0;
    float *rowscale = nullptr;
    bool dots_f16 = false;   // as in GemmArgs
};

// Whether the fused pack + XNOR-GEMM kernel fits (F <= 128, packed tiles in
// shared memory).
bool front_supported(int64_t N, int K, int F, const DeviceInfo &dev);

// Whether the split form of that kernel applies (few rows, each shared by
// several warps): then it is faster than packing and multiplying apart.
bool front_split_supported(int64_t N, int K, int F, const DeviceInfo &dev);

// Steps 1, 2 and 4 of one layer in one kernel (see front.cu).
void launch_front(const FrontArgs &args, const DeviceInfo &dev, cudaStream_t stream,
                  bool pdl = false);

// Largest layer-2 output width the fused aggregation handles.
constexpr int kMaxFusedOut = 64;

struct SpmmPackGemmArgs {
    const int64_t *rowptr;
    const int32_t *colidx;
    int64_t N;
    int64_t nnz;
    // Layer 1's Z', either fp32 rows pre-scaled by 1/sqrt(dhat) (Z1, row
    // stride Fh) or compressed (D1 non-null: uint16 dots + 32768, row stride
    // ldz1 >= Fh rounded up to 4 with zero dots as padding, with the row
    // scale s1 and the column scale beta1).
    const float *Z1;
    const uint16_t *D1;
    int64_t ldz1;
    const float *s1;
    const float *beta1;
    int Fh;
    float *H1;               // nullable N x Fh output (row stride ldh)
    int64_t ldh;
    const uint64_t *wbits2;  // Fo x ceil(Fh/64) packed columns of W2
    const float *beta2;      // Fo
    int Fo;
    float *Z2;               // N x Fo, rows pre-scaled by 1/sqrt(dhat) (row stride ldz2;
    int64_t ldz2;            // columns Fo .. ldz2 are written as zeros)
};

// Whether (Fh, Fo) fit the fused kernel: Fh % 4 == 0, Fh <= 128, Fo <= 64.
bool spmm_pack_gemm_supported(int Fh, int Fo);

// Layer-1 step 5 fused with layer-2 steps 2 and 4 (see spmm.cu).
void launch_spmm_pack_gemm(const SpmmPackGemmArgs &args, const DeviceInfo &dev,
                           cudaStream_t stream, bool pdl = false);

// Step 5 on the tensor cores (spmm_tc.cu) over a product kept factored as
// fp16 integer dots (exact for |dot| <= 2048): H_if = colscale_f *
// (1/sqrt(dhat_i)) * sum_{j in N(i) u {i}} rowscale_j * D[j, f], with
// rowscale_j carrying 1/sqrt(dhat_j). D's rows hold ldd halves (a multiple of
// 8, at least F rounded up to 16); features F .. round_up(F, 16) must hold
// zero dots. F <= 128.
struct SpmmTcArgs {
    const int64_t *rowptr;
    const int32_t *colidx;
    int64_t N;
    int64_t nnz;
    const uint16_t *D;       // fp16 bits
    int64_t ldd;
    const float *rowscale;   // N
    int F;
    float *H;                // N x F (row stride ldh)
    int64_t ldh;
    const float *colscale;   // nullable: 1
    int32_t *pred;           // nullable: each row's argmax (lowest index on ties)
};
bool spmm_tc_supported(int F);
void launch_spmm_tc(const SpmmTcArgs &args, const DeviceInfo &dev, cudaStream_t stream,
                    bool pdl = false);

// Layer 1's tensor-core aggregation fused with layer 2's binarization and
// XNOR product (spmm_tc.cu): from layer 1's fp16 dots D1 (row scale s1,
// column scale beta1) to layer 2's fp16 dots D2 (rows of ldd2 halves, a
// multiple of 8 >= Fo rounded up to 16, zeros past Fo) and row scale s2
// (alpha2_i / sqrt(dhat_i)); H1 (nullable) receives layer 1's output.
struct SpmmTcPackGemmArgs {
    const int64_t *rowptr;
    const int32_t *colidx;
    int64_t N;
    int64_t nnz;
    const uint16_t *D1;
    int64_t ldd1;
    const float *s1;
    int Fh;
    const float *beta1;
    float *H1;
    int64_t ldh1;
    const uint64_t *wbits2;  // Fo x ceil(Fh / 64)
    int Fo;
    uint16_t *D2;
    int64_t ldd2;
    float *s2;
};
bool spmm_tc_pack_gemm_supported(int Fh, int Fo);
void launch_spmm_tc_pack_gemm(const SpmmTcPackGemmArgs &args, const DeviceInfo &dev,
                              cudaStream_t stream, bool pdl = false);

// Ablation products of step 4 (ablation.cu): one operand real, the other
// binarized, on the tensor cores with the real operand as three bf16 parts.
struct RealBinaryArgs {      // weights binarized: Z = Y W~
    const float *X;          // N x K (row stride ldx), centred by scale/shift
    int64_t ldx;
    const float *scale;      // nullable (identity)
    const float *shift;      // nullable with scale non-null: y = x * scale (rounded once)
    const uint64_t *b_bits;  // F x words
    const float *beta;       // F; nullable: column scales of 1
    int64_t N;
    int K;
    int F;
    int words;
    float *Z;                // N x F (row stride ldz)
    int64_t ldz;
    const int64_t *rowptr;   // nullable: scale row i by 1/sqrt(1 + deg_i)
    bool clip = false;       // store z where |z| < 1, else 0 (Eq. bp-H)
};
void launch_real_binary_gemm(const RealBinaryArgs &args, const DeviceInfo &dev,
                             cudaStream_t stream, bool pdl = false);

struct BinaryRealArgs {      // features binarized: Z = H~ W
    const uint64_t *a_bits;  // N x words
    const float *alpha;      // N
    const uint16_t *wparts;  // 3 x F x (words * 64) bf16 parts of W (launch_split_weights)
    int64_t N;
    int K;
    int F;
    int words;
    float *Z;                // N x F (row stride ldz)
    int64_t ldz;
    const int64_t *rowptr;   // nullable: scale row i by 1/sqrt(1 + deg_i)
};
void launch_binary_real_gemm(const BinaryRealArgs &args, const DeviceInfo &dev,
                             cudaStream_t stream, bool pdl = false);

// Transposed signs x real (ablation.cu): partial[s] = sum over the nodes of
// chunk s of alpha_i sign(y_ik) G_ij (K x F each; dL/dW~ = H~^T G is their
// sum in order). Returns the number of chunks written (<= max_split).
struct SignTRealArgs {
    const uint64_t *bits;    // N x words packed node signs (K features)
    int words;
    const float *alpha;      // N
    const float *G;          // N x F (row stride ldg)
    int64_t ldg;
    int64_t N;
    int K;
    int F;
    float *partial;          // max_split x K x F
};
int launch_sign_t_real_gemm(const SignTRealArgs &args, int max_split, const DeviceInfo &dev,
                            cudaStream_t stream);

// Bytes of the bf16 parts of a K x F weight matrix, and the kernel that
// writes them (parts[p][j][k], zero for k >= K up to bigcn_words(K) * 64).
size_t weight_parts_bytes(int K, int F);
void launch_split_weights(const float *Wt, int K, int F, int64_t ldw, uint16_t *wparts,
                          cudaStream_t stream);

// Sub-row bucketing (bucket.cu): buckets of 64 bw signs, scales N x nb / F x nb.
void launch_pack_rows_bucketed(const float *X, int64_t N, int K, int64_t ldx, const float *scale,
                               const float *shift, int bw, uint64_t *bits, int words,
                               float *alpha, const DeviceInfo &dev, cudaStream_t stream);
void launch_pack_weights_bucketed(const float *Wt, int K, int F, int64_t ldw, int bw,
                                  uint64_t *bits, int words, float *beta, cudaStream_t stream);
struct BucketGemmArgs {
    const uint64_t *A;       // N x words
    const float *alpha;      // N x nb
    int64_t N;
    const uint64_t *B;       // F x words
    const float *beta;       // F x nb
    int F;
    int K;
    int words;               // ceil(K / 64)
    int bw;                  // words per bucket
    float *Z;                // N x F (row stride ldz)
    int64_t ldz;
    const int64_t *rowptr;   // nullable: scale row i by 1/sqrt(1 + deg_i)
};
void launch_xnor_gemm_bucketed(const BucketGemmArgs &args, const DeviceInfo &dev,
                               cudaStream_t stream);

// Waits of the ablation products that ran out since the last call (and
// resets the count); ~0u on a CUDA error.
uint32_t take_mix_timeouts();

}  // namespace bigcn
