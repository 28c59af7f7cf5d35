// Binarized layers of inductive GNNs (Sec. 6.3, Table 3: Bi-inductiveGCN and
// Bi-GraphSAGE). Binarizing "every feature-extraction step" of GraphSAGE's
// models leaves their structure: the product of Eqs. 10-12 on each node's own
// features, then an aggregation of the d_out-wide products -- the count under
// which Table 3's cycle operations and model sizes reproduce (two products
// per GraphSAGE layer, one aggregation of d_out-wide rows).
//
//   mean (inductive GCN):  H_i = (1 / dhat_i) sum over j in N(i) u {i} of zeta_j
//   sage (GraphSAGE-mean): H_i = zeta_i + (1 / |N(i)|) sum over j in N(i) of zeta'_j
//
// where zeta' is the product with the neighbour weights (GraphSAGE's
// W [h_i || mean_j h_j] = W_self h_i + W_neigh mean_j h_j, with the mean
// taken after the product, as Bi-GCN aggregates after its product).
//
// Both run on the Bi-GCN kernels: pack rows (centre, sign, alpha), pack
// weights, the XNOR product without a degree factor (for few long rows the
// split front kernel packs and multiplies in one pass) (its row scale is alpha_j
// alone) and the aggregation in its mean / GraphSAGE mode. GraphSAGE's two
// products are one product over the packed columns of W_self and W_neigh
// (packed by one launch into the two halves of one array), each half padded
// to a multiple of 8 columns with beta = 0 (so the padding's products are
// exactly 0), so that both halves of a product row start on a 16-byte
// boundary for the gathers.
#include "launch.cuh"

using namespace bigcn;

namespace {

constexpr size_t kIAlign = 256;
size_t iround(size_t x) { return (x + kIAlign - 1) / kIAlign * kIAlign; }
constexpr int32_t kMaxDots16K = 32767;

// Workspace: A bits, alpha, B bits, beta, Z (factored or fp32), row scale.
// Fz = product columns (F, or 2 Fp for GraphSAGE).
struct InductiveWorkspace {
    size_t a_bits, alpha, b_bits, beta, z, rowscale, total;
    int64_t Fp, Fz, ldz;
    bool compressed;
};

bool inductive_workspace(int32_t agg, int64_t N, int32_t K, int32_t F, InductiveWorkspace *w) {
    if (N < 0 || K < 1 || F < 1) return false;
    if (agg != BIGCN_AGG_MEAN && agg != BIGCN_AGG_SAGE) return false;
    const bool sage = agg == BIGCN_AGG_SAGE;
    w->Fp = (int64_t(F) + 7) / 8 * 8;
    w->Fz = sage ? 2 * w->Fp : F;
    w->compressed = K <= kMaxDots16K;
    w->ldz = w->compressed ? (w->Fz + 7) / 8 * 8 : w->Fz;
    const int64_t words = bigcn_words(K);
    if (N > kMaxElems / (words > w->ldz ? words : w->ldz)) return false;
    if (int64_t(K) > kMaxElems / w->Fz) return false;
    size_t off = 0;
    w->a_bits = off; off = iround(off + size_t(N) * size_t(words) * 8);
    w->alpha = off;  off = iround(off + size_t(N) * 4);
    w->b_bits = off; off = iround(off + size_t(w->Fz) * size_t(words) * 8);
    w->beta = off;   off = iround(off + size_t(w->Fz) * 4);
    w->z = off;      off = iround(off + size_t(N) * size_t(w->ldz) * (w->compressed ? 2 : 4));
    w->rowscale = off;
    if (w->compressed) off = iround(off + size_t(N) * 4);
    w->total = off;
    return true;
}

}  // namespace

extern "C" size_t bigcn_inductive_layer_workspace_bytes(int32_t aggregator, int64_t N, int32_t K,
                                                        int32_t F) {
    if (aggregator == BIGCN_AGG_GCN) return bigcn_layer_workspace_bytes(N, K, F);
    InductiveWorkspace w;
    return inductive_workspace(aggregator, N, K, F, &w) ? w.total : 0;
}

extern "C" bigcn_status bigcn_inductive_layer_forward(
    int32_t aggregator, const float *X, int64_t N, int32_t K, int64_t ldx, const float *scale,
    const float *shift, const float *Wt, int32_t F, int64_t ldw, const float *W_neigh,
    int64_t ldwn, const int64_t *rowptr, const int32_t *colidx, int64_t nnz, void *workspace,
    size_t ws_bytes, float *H, int64_t ldh, void *stream) {
    if (aggregator == BIGCN_AGG_GCN)
        return bigcn_layer_forward(X, N, K, ldx, scale, shift, Wt, F, ldw, rowptr, colidx, nnz,
                                   workspace, ws_bytes, H, ldh, stream);
    InductiveWorkspace w;
    const bool sage = aggregator == BIGCN_AGG_SAGE;
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || ldx < K || ldw < F || ldh < F ||
        nnz < 0 || (sage && ldwn < F))
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (!inductive_workspace(aggregator, N, K, F, &w)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / ldh)) return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw || (sage && int64_t(K) > kMaxElems / ldwn))
        return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!X || !Wt || (sage && !W_neigh) || !rowptr || !H || !workspace || (nnz > 0 && !colidx))
        return BIGCN_ERR_INVALID_ARG;
    if (ws_bytes < w.total) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(Wt, 4) || (sage && !aligned_to(W_neigh, 4)) ||
        !aligned_to(rowptr, 8) || (colidx && !aligned_to(colidx, 4)) || !aligned_to(H, 4) ||
        !aligned_to(workspace, kIAlign) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t hb = span_bytes(N, F, ldh, 4);
    const void *inputs[] = {X, Wt, sage ? W_neigh : nullptr, rowptr, colidx, scale, shift};
    const size_t in_bytes[] = {span_bytes(N, K, ldx, 4), span_bytes(K, F, ldw, 4),
                               sage ? span_bytes(K, F, ldwn, 4) : 0, size_t(N + 1) * 8,
                               size_t(nnz) * 4, size_t(K) * 4, size_t(K) * 4};
    for (int q = 0; q < 7; ++q) {
        if (overlaps(workspace, w.total, inputs[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
        if (overlaps(H, hb, inputs[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
    }
    if (overlaps(H, hb, workspace, w.total)) return BIGCN_ERR_INVALID_ARG;

    DeviceInfo dev;
    const bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    char *ws = static_cast<char *>(workspace);
    uint64_t *a_bits = reinterpret_cast<uint64_t *>(ws + w.a_bits);
    float *alpha = reinterpret_cast<float *>(ws + w.alpha);
    uint64_t *b_bits = reinterpret_cast<uint64_t *>(ws + w.b_bits);
    float *beta = reinterpret_cast<float *>(ws + w.beta);
    const int words = bigcn_words(K);
    const int Fz = int(w.Fz);
    cudaStream_t s = as_stream(stream);

    // Packed weight columns: Wt's, or Wt's in columns [0, F) and W_neigh's in
    // [Fp, Fp + F), the padding columns with beta = 0 (their bits are never
    // scaled by anything else).
    if (sage && F != w.Fp && cudaMemsetAsync(beta, 0, size_t(Fz) * 4, s) != cudaSuccess)
        return BIGCN_ERR_CUDA;
    const bool fused = front_split_supported(N, K, Fz, dev);
    if (!fused) launch_pack_rows(X, N, K, ldx, scale, shift, a_bits, words, alpha, dev, s);
    const WeightPack wa{Wt, K, F, ldw, b_bits, words, beta, 0};
    const WeightPack wb = sage ? WeightPack{W_neigh, K, F, ldwn, b_bits + w.Fp * words, words,
                                            beta + w.Fp, 0}
                               : WeightPack{nullptr, 1, 0, 0, nullptr, 0, nullptr, 0};
    launch_pack_weights2(wa, wb, s);
    // The product without a degree factor: Z_ij = alpha_i beta_j dot_ij, kept
    // factored (uint16 dots, row scale alpha_i) when K allows.
    GemmArgs g{a_bits, alpha, N, b_bits, beta, Fz, K, words, nullptr, Fz, nullptr, nullptr};
    SpmmArgs a{rowptr, colidx, N, nnz, nullptr, w.ldz, F, H, ldh, true, true};
    a.agg = sage ? kAggSage : kAggMean;
    const int64_t half = sage ? w.Fp : 0;
    if (w.compressed) {
        uint16_t *D16 = reinterpret_cast<uint16_t *>(ws + w.z);
        float *rowscale = reinterpret_cast<float *>(ws + w.rowscale);
        g.dots16 = D16;
        g.ldd16 = w.ldz;
        g.rowscale = rowscale;
        a.D16 = D16 + half;
        a.rowscale = rowscale;
        a.colscale = beta + half;
        a.Zs = D16;
        a.colscale_s = beta;
    } else {
        float *Z = reinterpret_cast<float *>(ws + w.z);
        g.Z = Z;
        g.ldz = w.ldz;
        a.Z = Z + half;
        a.Zs = Z;
        // fp32 rows: the gathers read up to F rounded to 4, inside the padded half.
        a.z_pad4 = sage || F % 4 == 0;
    }
    if (fused) {         // few long rows: centring, packing and product in one kernel
        FrontArgs fr{X, N, K, ldx, scale, shift, b_bits, beta, Fz, words, nullptr, g.Z, g.ldz,
                     g.dots16, g.ldd16, g.rowscale};
        launch_front(fr, dev, s);
    } else {
        launch_xnor_gemm(g, dev, s);
    }
    launch_spmm_norm(a, dev, s);
    return launch_status();
}
