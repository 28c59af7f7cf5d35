// The two-layer Bi-GCN forward of Sec. 6.2 (Wang et al., CVPR 2021) as one
// call: layer 1 centred (Sec. 6.2), layer 2 on H1 raw (Sec. 4.1.2), each
// layer Eq. 13 with zeta of Eqs. 11-12. Kernel sequence on one stream:
//
//   0 pack W1 and W2 (one launch)                          Eqs. 3-4
//   1 centre + pack rows of X + XNOR GEMM, rows scaled     Sec. 6.2, Eqs. 7-8,
//     by 1/sqrt(dhat) (packed rows stay in shared memory)  Eqs. 11-12
//   2 aggregation of layer 1 fused with layer 2's row      Eq. 13, then
//     packing and XNOR GEMM (H1 stays in registers)        Eqs. 7-8, 11-12
//   3 aggregation of layer 2 -> logits                     Eq. 13
//
// Step 1 runs as two kernels (pack rows, then GEMM) when the packed weight
// tile does not fit in shared memory (hidden width above 128 or very long
// rows), and step 2 as three (aggregation, packing, GEMM) when the widths do
// not fit the fused kernel (hidden width not a multiple of 4 or above 128, or
// more than 64 outputs). Every step runs on the GPU either way.
//
// When K <= 2048 (layer 1's dots exact in fp16), Fh <= 128 and Fo <= 64, the
// products stay factored as fp16 dots with a row scale and both
// aggregations run on the tensor cores (spmm_tc.cu): step 2 writes layer 2's
// dots D2 and row scale s2 instead of fp32 Z2', and step 3 multiplies by beta2.
//
// Every kernel after the first is launched with programmatic serialization:
// it may start while its predecessor drains, and waits (griddepcontrol) only
// before it reads what an earlier kernel wrote -- the fused front streams and
// packs X while the weights are still being packed.
#include "launch.cuh"

namespace bigcn {
namespace {

constexpr size_t kAlign = 256;
size_t round_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Largest K (or Fh) whose dots the compressed uint16 form holds.
constexpr int32_t kMaxDots16K = 32767;
// Largest K whose dots fp16 holds exactly: the tensor-core aggregation's input.
constexpr int32_t kMaxDotsF16K = 2048;

// The tensor-core path: layer 1's dots as fp16, both aggregations on
// spmm_tc.cu, layer 2's product kept factored as fp16 dots as well.
bool forward2_tc(int32_t K, int32_t Fh, int32_t Fo) {
    return K <= kMaxDotsF16K && spmm_tc_pack_gemm_supported(Fh, Fo);
}

// Workspace carve-up. Layer 1's Z' is fp32 (N x Fh) or, when K <= 32767,
// compressed: uint16 dots (N x Fh8, Fh8 = Fh rounded up to 8) and a row
// scale. Layer 2's Z' is fp32, pre-scaled, with rows padded to a multiple of
// 4 (its rows are narrow: the extra row-scale read would cost more than the
// bytes a compressed row saves).
struct Forward2Workspace {
    size_t bits1, alpha1, wbits1, beta1, z1, s1, wbits2, beta2, z2, h1, bits2, alpha2, d2, s2,
        total;
    bool c16, tc;
};

bool forward2_workspace(int64_t N, int32_t K, int32_t Fh, int32_t Fo, Forward2Workspace *w) {
    if (N < 0 || K < 1 || Fh < 1 || Fo < 1) return false;
    const int64_t w1 = bigcn_words(K), w2 = bigcn_words(Fh);
    const int64_t Fh8 = (int64_t(Fh) + 7) / 8 * 8, Fo4 = (int64_t(Fo) + 3) / 4 * 4;
    int64_t widest = w1;
    if (Fh8 > widest) widest = Fh8;
    if (Fo4 > widest) widest = Fo4;
    if (N > kMaxElems / widest) return false;
    w->c16 = K <= kMaxDots16K;
    w->tc = forward2_tc(K, Fh, Fo);
    const int64_t Fh16 = (int64_t(Fh) + 15) / 16 * 16, Fo16 = (int64_t(Fo) + 15) / 16 * 16;
    size_t off = 0;
    auto take = [&](size_t bytes) { size_t at = off; off = round_up(off + bytes); return at; };
    w->bits1 = take(size_t(N) * w1 * 8);
    w->alpha1 = take(size_t(N) * 4);
    w->wbits1 = take(size_t(Fh) * w1 * 8);
    w->beta1 = take(size_t(Fh) * 4);
    w->z1 = take(w->tc ? size_t(N) * Fh16 * 2 : w->c16 ? size_t(N) * Fh8 * 2 : size_t(N) * Fh * 4);
    w->s1 = take(size_t(N) * 4);
    w->wbits2 = take(size_t(Fo) * w2 * 8);
    w->beta2 = take(size_t(Fo) * 4);
    w->z2 = take(size_t(N) * Fo4 * 4);
    w->h1 = take(size_t(N) * Fh * 4);
    w->bits2 = take(size_t(N) * w2 * 8);
    w->alpha2 = take(size_t(N) * 4);
    w->d2 = take(w->tc ? size_t(N) * Fo16 * 2 : 0);
    w->s2 = take(w->tc ? size_t(N) * 4 : 0);
    w->total = off;
    return true;
}

}  // namespace
}  // namespace bigcn

using namespace bigcn;

extern "C" size_t bigcn_forward_2layer_workspace_bytes(int64_t N, int32_t K, int32_t Fh,
                                                       int32_t Fo) {
    Forward2Workspace w;
    return forward2_workspace(N, K, Fh, Fo, &w) ? w.total : 0;
}

extern "C" int32_t bigcn_forward_2layer_aggregation(int32_t K, int32_t Fh, int32_t Fo) {
    if (K < 1 || Fh < 1 || Fo < 1) return -1;
    return forward2_tc(K, Fh, Fo) ? 1 : 0;
}

extern "C" int32_t bigcn_forward_2layer_launches(int64_t N, int32_t K, int32_t Fh, int32_t Fo) {
    if (N < 0 || K < 1 || Fh < 1 || Fo < 1) return -1;
    DeviceInfo dev;
    if (current_device(&dev) != BIGCN_OK) return -1;
    return 1 + (front_supported(N, K, Fh, dev) ? 1 : 2) +
           (forward2_tc(K, Fh, Fo) || spmm_pack_gemm_supported(Fh, Fo) ? 1 : 3) + 1;
}

extern "C" bigcn_status bigcn_forward_2layer(
    const float *X, int64_t N, int32_t K, int64_t ldx, const float *scale, const float *shift,
    const float *W1, int32_t Fh, int64_t ldw1, const float *W2, int32_t Fo, int64_t ldw2,
    const int64_t *rowptr, const int32_t *colidx, int64_t nnz, void *workspace, size_t ws_bytes,
    float *H1, int64_t ldh1, float *out, int64_t ldo, int32_t *pred, void *const *events,
    int32_t n_events, void *stream) {
    Forward2Workspace w;
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || Fh < 1 || Fo < 1 || ldx < K || ldw1 < Fh ||
        ldw2 < Fo || ldo < Fo || (H1 && ldh1 < Fh) || nnz < 0 || n_events < 0)
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (!forward2_workspace(N, K, Fh, Fo, &w)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / ldo || (H1 && N > kMaxElems / ldh1)))
        return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw1 || int64_t(Fh) > kMaxElems / ldw2)
        return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!X || !W1 || !W2 || !rowptr || !out || !workspace || (nnz > 0 && !colidx) ||
        (n_events > 0 && !events))
        return BIGCN_ERR_INVALID_ARG;
    if (ws_bytes < w.total) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(W1, 4) || !aligned_to(W2, 4) || !aligned_to(rowptr, 8) ||
        (colidx && !aligned_to(colidx, 4)) || !aligned_to(out, 4) || (H1 && !aligned_to(H1, 4)) ||
        (pred && !aligned_to(pred, 4)) ||
        !aligned_to(workspace, kAlign) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const void *in[] = {X, W1, W2, rowptr, colidx, scale, shift};
    const size_t in_bytes[] = {span_bytes(N, K, ldx, 4), span_bytes(K, Fh, ldw1, 4),
                               span_bytes(Fh, Fo, ldw2, 4), size_t(N + 1) * 8, size_t(nnz) * 4,
                               size_t(K) * 4, size_t(K) * 4};
    const void *outs[] = {workspace, out, H1, pred};
    const size_t out_bytes[] = {w.total, span_bytes(N, Fo, ldo, 4),
                                H1 ? span_bytes(N, Fh, ldh1, 4) : 0, pred ? size_t(N) * 4 : 0};
    for (int o = 0; o < 4; ++o) {
        for (int q = 0; q < 7; ++q)
            if (overlaps(outs[o], out_bytes[o], in[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
        for (int p = o + 1; p < 4; ++p)
            if (overlaps(outs[o], out_bytes[o], outs[p], out_bytes[p])) return BIGCN_ERR_INVALID_ARG;
    }

    DeviceInfo dev;
    bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;

    char *ws = static_cast<char *>(workspace);
    auto at = [&](size_t off) { return static_cast<void *>(ws + off); };
    uint64_t *bits1 = static_cast<uint64_t *>(at(w.bits1));
    float *alpha1 = static_cast<float *>(at(w.alpha1));
    uint64_t *wbits1 = static_cast<uint64_t *>(at(w.wbits1));
    float *beta1 = static_cast<float *>(at(w.beta1));
    void *Z1 = at(w.z1);
    float *s1 = static_cast<float *>(at(w.s1));
    uint64_t *wbits2 = static_cast<uint64_t *>(at(w.wbits2));
    float *beta2 = static_cast<float *>(at(w.beta2));
    float *Z2 = static_cast<float *>(at(w.z2));
    const int words1 = bigcn_words(K), words2 = bigcn_words(Fh);
    const int64_t Fh8 = (Fh + 7) / 8 * 8, Fo4 = (Fo + 3) / 4 * 4;
    const int64_t Fh16 = (Fh + 15) / 16 * 16, Fo16 = (Fo + 15) / 16 * 16;
    const int64_t ldd1 = w.tc ? Fh16 : Fh8;     // layer 1's compressed row stride
    const bool fused = spmm_pack_gemm_supported(Fh, Fo);
    uint16_t *D1 = w.c16 ? static_cast<uint16_t *>(Z1) : nullptr;
    float *Z1f = w.c16 ? nullptr : static_cast<float *>(Z1);
    cudaStream_t s = as_stream(stream);
    EventMarks marks(events, n_events, s);
    if (!marks.ok()) return BIGCN_ERR_CUDA;
    auto mark = [&]() { marks.mark(); };

    mark();
    WeightPack p1{W1, K, Fh, ldw1, wbits1, words1, beta1, 0};
    WeightPack p2{W2, Fh, Fo, ldw2, wbits2, words2, beta2, 0};
    launch_pack_weights2(p1, p2, s);
    mark();
    if (front_supported(N, K, Fh, dev)) {
        FrontArgs fr{X, N, K, ldx, scale, shift, wbits1, beta1, Fh, words1, rowptr, Z1f, Fh};
        if (w.c16) {
            fr.D16 = D1;
            fr.ldd16 = ldd1;
            fr.rowscale = s1;
            fr.dots_f16 = w.tc;
        }
        launch_front(fr, dev, s, true);
        mark();
    } else {
        launch_pack_rows(X, N, K, ldx, scale, shift, bits1, words1, alpha1, dev, s, true, false);
        mark();
        GemmArgs g1{bits1, alpha1, N, wbits1, beta1, Fh, K, words1, Z1f, Fh, nullptr, rowptr};
        if (w.c16) {
            g1.dots16 = D1;
            g1.ldd16 = ldd1;
            g1.rowscale = s1;
            g1.dots_f16 = w.tc;
        }
        launch_xnor_gemm(g1, dev, s, true);
        mark();
    }
    if (w.tc) {
        // Both aggregations on the tensor cores: layer 1's fused with layer 2's
        // binarization and product (fp16 dots D2 and row scale s2), then layer 2's.
        uint16_t *D2 = static_cast<uint16_t *>(at(w.d2));
        float *s2 = static_cast<float *>(at(w.s2));
        SpmmTcPackGemmArgs f{rowptr, colidx, N, nnz, D1, ldd1, s1, Fh, beta1, H1, ldh1,
                             wbits2, Fo, D2, Fo16, s2};
        launch_spmm_tc_pack_gemm(f, dev, s, true);
        mark();
        SpmmTcArgs a2{rowptr, colidx, N, nnz, D2, Fo16, s2, Fo, out, ldo, beta2, pred};
        launch_spmm_tc(a2, dev, s, true);
        mark();
        const bigcn_status ls = launch_status();
        return marks.failed() ? BIGCN_ERR_CUDA : ls;
    }
    if (fused) {
        SpmmPackGemmArgs f{rowptr, colidx, N, nnz, Z1f, D1, Fh8, s1, beta1, Fh, H1, ldh1,
                           wbits2, beta2, Fo, Z2, Fo4};
        launch_spmm_pack_gemm(f, dev, s, true);
        mark();
    } else {
        float *H1w = H1 ? H1 : static_cast<float *>(at(w.h1));
        const int64_t ldh = H1 ? ldh1 : Fh;
        uint64_t *bits2 = static_cast<uint64_t *>(at(w.bits2));
        float *alpha2 = static_cast<float *>(at(w.alpha2));
        SpmmArgs a1{rowptr, colidx, N, nnz, Z1f, w.c16 ? Fh8 : Fh, Fh, H1w, ldh, true, false};
        if (w.c16) {
            a1.D16 = D1;
            a1.rowscale = s1;
            a1.colscale = beta1;
        }
        launch_spmm_norm(a1, dev, s, true);
        mark();
        launch_pack_rows(H1w, N, Fh, ldh, nullptr, nullptr, bits2, words2, alpha2, dev, s, true,
                         true);
        mark();
        GemmArgs g2{bits2, alpha2, N, wbits2, beta2, Fo, Fh, words2, Z2, Fo4, nullptr, rowptr};
        launch_xnor_gemm(g2, dev, s, true);
        mark();
    }
    // The fused kernel writes Z2's padding columns as zeros: whole 4-wide
    // vectors may be gathered.
    SpmmArgs a2{rowptr, colidx, N, nnz, Z2, Fo4, Fo, out, ldo, true, fused};
    a2.pred = pred;
    launch_spmm_norm(a2, dev, s, true);
    mark();
    const bigcn_status ls = launch_status();
    return marks.failed() ? BIGCN_ERR_CUDA : ls;
}
