// Internal launchers of the four Bi-GCN kernels. Each entry point of
// include/bigcn.h validates its arguments and calls one of these; the fused
// layer calls them in sequence on one stream. Arguments are assumed valid.
#pragma once

#include <cuda_runtime.h>

#include <cstdint>

#include "bigcn_internal.cuh"

namespace bigcn {

// Steps 1+2: centre, sign-pack rows, per-node scale (Sec. 6.2, Eqs. 7-8).
void launch_pack_rows(const float *X, int64_t N, int K, int64_t ldx, const float *scale,
                      const float *shift, uint64_t *bits, int words, float *alpha,
                      const DeviceInfo &dev, cudaStream_t stream);

// Step 3: sign-pack weight columns, per-column scale (Eqs. 3-4).
void launch_pack_weights(const float *Wt, int K, int F, int64_t ldw, uint64_t *bits,
                         int words, float *beta, cudaStream_t stream);

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
};

// Step 4: the XNOR-popcount product and its scaling (Eqs. 11-12).
void launch_xnor_gemm(const GemmArgs &args, const DeviceInfo &dev, cudaStream_t stream);

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
};

// Step 5: H = D^-1/2 (A + I) D^-1/2 Z (Eqs. 1, 13).
void launch_spmm_norm(const SpmmArgs &args, const DeviceInfo &dev, cudaStream_t stream);

}  // namespace bigcn
