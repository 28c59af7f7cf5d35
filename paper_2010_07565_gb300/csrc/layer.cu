// The fused Bi-GCN layer (Wang et al., CVPR 2021, Eq. 13 with zeta from
// Eqs. 11-12) and the interface's small helpers: status strings, the packed
// row width, the per-device property cache and the workspace layout.
//
// bigcn_layer_forward enqueues, on one stream:
//   pack_rows (centre + sign + alpha) -> pack_weights (sign + beta)
//   -> xnor_gemm whose epilogue also multiplies row j by 1/sqrt(dhat_j)
//   -> spmm over the pre-scaled rows, which multiplies by 1/sqrt(dhat_i);
// for few long rows (fewer than a wave of warps) the split front kernel does
// pack_rows' and xnor_gemm's work in one pass after pack_weights.
// Folding the source-side degree factor into the product's epilogue saves the
// aggregation one random read of the CSR row pointers per edge. When the dots
// fit 16 bits (K <= 32767) the product leaves Z factored: the integer dots
// and the row scale s_j = alpha_j / sqrt(dhat_j), and the aggregation applies
// s_j per neighbour and beta_f per column, so each gathered row is half the
// bytes. With K <= 2048 the dots are fp16 (exact) and the aggregation runs on
// the tensor cores (spmm_tc.cu); else they are biased uint16 and it runs on
// the CUDA cores (spmm.cu).
#include <mutex>

#include "launch.cuh"

namespace bigcn {

namespace {
constexpr int kMaxDevices = 64;
DeviceInfo g_info[kMaxDevices];
bigcn_status g_info_status[kMaxDevices];
std::once_flag g_info_once[kMaxDevices];

void query_device(int dev) {
    DeviceInfo &d = g_info[dev];
    d.device = dev;
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&d.sm_count, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&d.max_smem_optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) !=
            cudaSuccess) {
        cudaGetLastError();
        g_info_status[dev] = BIGCN_ERR_CUDA;
        return;
    }
    g_info_status[dev] = (major == 10 && minor == 3) ? BIGCN_OK : BIGCN_ERR_UNSUPPORTED;
}

constexpr size_t kAlign = 256;
size_t round_up(size_t x) { return (x + kAlign - 1) / kAlign * kAlign; }

// Workspace carve-up of the fused layer; every piece 256-byte aligned.
// Largest K whose dots (|dot| <= K) the compressed uint16 form holds.
constexpr int32_t kMaxDots16K = 32767;

// Workspace carve-up of the fused layer; every piece 256-byte aligned. Z is
// either fp32 (N x F) or compressed: uint16 dots (N x round_up(F, 8), so that
// the aggregation can load eight dots at a time) and a row scale (N); then the
// FP8 tiles of the weight signs for the tensor-core product (about F x K bytes
// when K >= 128 and F >= 32).
struct LayerWorkspace {
    size_t a_bits, alpha, b_bits, beta, z, rowscale, bexp, bexp_bytes, total;
    bool compressed;
    bool f16;                // dots as fp16 (K <= 2048): the tensor-core aggregation
    int64_t ldd;             // halves per compressed row
};

// Largest K whose dots fp16 holds exactly.
constexpr int32_t kMaxDotsF16K = 2048;

bool layer_workspace(int64_t N, int32_t K, int32_t F, LayerWorkspace *w) {
    if (N < 0 || K < 1 || F < 1) return false;
    const int64_t words = bigcn_words(K);
    const int64_t F8 = (int64_t(F) + 7) / 8 * 8;
    if (N > kMaxElems / (words > F8 ? words : F8)) return false;
    w->compressed = K <= kMaxDots16K;
    // fp16 dots and the tensor-core aggregation for rows of up to 128 features
    // (wider rows would walk their index lists once per 128-feature slab; the
    // CUDA-core aggregation was measured faster at 256: 2047 vs 2567 us on
    // 2^20 nodes of mean degree 16).
    w->f16 = K <= kMaxDotsF16K && F <= 128;
    w->ldd = w->f16 ? (int64_t(F) + 15) / 16 * 16 : F8;
    size_t off = 0;
    w->a_bits = off; off = round_up(off + size_t(N) * size_t(words) * 8);
    w->alpha = off;  off = round_up(off + size_t(N) * 4);
    w->b_bits = off; off = round_up(off + size_t(F) * size_t(words) * 8);
    w->beta = off;   off = round_up(off + size_t(F) * 4);
    w->z = off;
    if (w->compressed) {
        off = round_up(off + size_t(N) * size_t(w->ldd) * 2);
        w->rowscale = off; off = round_up(off + size_t(N) * 4);
    } else {
        off = round_up(off + size_t(N) * size_t(F) * 4);
        w->rowscale = off;
    }
    // The tensor-core product's weight signs expanded to FP8 tiles once.
    w->bexp = off;
    w->bexp_bytes = xnor_gemm_tc_bexp_bytes(K, F);
    off = round_up(off + w->bexp_bytes);
    w->total = off;
    return true;
}
}  // namespace

bigcn_status current_device(DeviceInfo *info) {
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) {
        cudaGetLastError();
        return BIGCN_ERR_CUDA;
    }
    if (dev < 0 || dev >= kMaxDevices) return BIGCN_ERR_UNSUPPORTED;
    std::call_once(g_info_once[dev], query_device, dev);
    if (g_info_status[dev] != BIGCN_OK) return g_info_status[dev];
    *info = g_info[dev];
    return BIGCN_OK;
}

bigcn_status launch_status() {
    return cudaGetLastError() == cudaSuccess ? BIGCN_OK : BIGCN_ERR_CUDA;
}

}  // namespace bigcn

using namespace bigcn;

extern "C" const char *bigcn_status_string(int status) {
    switch (status) {
        case BIGCN_OK: return "BIGCN_OK";
        case BIGCN_ERR_INVALID_ARG: return "BIGCN_ERR_INVALID_ARG";
        case BIGCN_ERR_MISALIGNED: return "BIGCN_ERR_MISALIGNED";
        case BIGCN_ERR_CUDA: return "BIGCN_ERR_CUDA";
        case BIGCN_ERR_UNSUPPORTED: return "BIGCN_ERR_UNSUPPORTED";
        case BIGCN_ERR_SCRATCH_LIMIT: return "BIGCN_ERR_SCRATCH_LIMIT";
        default: return "BIGCN_ERR_UNKNOWN";
    }
}

extern "C" int32_t bigcn_words(int32_t K) { return K <= 0 ? 0 : int32_t((int64_t(K) + 63) / 64); }

extern "C" size_t bigcn_layer_workspace_bytes(int64_t N, int32_t K, int32_t F) {
    LayerWorkspace w;
    return layer_workspace(N, K, F, &w) ? w.total : 0;
}

extern "C" bigcn_status bigcn_layer_forward_timed(const float *X, int64_t N, int32_t K,
                                                  int64_t ldx, const float *scale,
                                                  const float *shift, const float *Wt, int32_t F,
                                                  int64_t ldw, const int64_t *rowptr,
                                                  const int32_t *colidx, int64_t nnz,
                                                  void *workspace, size_t ws_bytes, float *H,
                                                  int64_t ldh, void *const *events,
                                                  int32_t n_events, void *stream) {
    if (n_events < 0 || (n_events > 0 && !events)) return BIGCN_ERR_INVALID_ARG;
    LayerWorkspace w;
    if (N < 0 || N > int64_t(INT32_MAX) || K < 1 || F < 1 || ldx < K || ldw < F || ldh < F ||
        nnz < 0)
        return BIGCN_ERR_INVALID_ARG;
    if ((scale == nullptr) != (shift == nullptr)) return BIGCN_ERR_INVALID_ARG;
    if (!layer_workspace(N, K, F, &w)) return BIGCN_ERR_INVALID_ARG;
    if (N > 0 && (N > kMaxElems / ldx || N > kMaxElems / ldh)) return BIGCN_ERR_INVALID_ARG;
    if (int64_t(K) > kMaxElems / ldw) return BIGCN_ERR_INVALID_ARG;
    if (N == 0) return BIGCN_OK;
    if (!X || !Wt || !rowptr || !H || !workspace || (nnz > 0 && !colidx))
        return BIGCN_ERR_INVALID_ARG;
    if (ws_bytes < w.total) return BIGCN_ERR_INVALID_ARG;
    if (!aligned_to(X, 4) || !aligned_to(Wt, 4) || !aligned_to(rowptr, 8) ||
        (colidx && !aligned_to(colidx, 4)) || !aligned_to(H, 4) || !aligned_to(workspace, kAlign) ||
        (scale && (!aligned_to(scale, 4) || !aligned_to(shift, 4))))
        return BIGCN_ERR_MISALIGNED;
    const size_t xb = span_bytes(N, K, ldx, 4), hb = span_bytes(N, F, ldh, 4);
    const size_t wb = span_bytes(K, F, ldw, 4);
    const void *inputs[] = {X, Wt, rowptr, colidx, scale, shift};
    const size_t in_bytes[] = {xb, wb, size_t(N + 1) * 8, size_t(nnz) * 4, size_t(K) * 4,
                               size_t(K) * 4};
    for (int q = 0; q < 6; ++q) {
        if (overlaps(workspace, w.total, inputs[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
        if (overlaps(H, hb, inputs[q], in_bytes[q])) return BIGCN_ERR_INVALID_ARG;
    }
    if (overlaps(H, hb, workspace, w.total)) return BIGCN_ERR_INVALID_ARG;

    DeviceInfo dev;
    bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;

    char *ws = static_cast<char *>(workspace);
    uint64_t *a_bits = reinterpret_cast<uint64_t *>(ws + w.a_bits);
    float *alpha = reinterpret_cast<float *>(ws + w.alpha);
    uint64_t *b_bits = reinterpret_cast<uint64_t *>(ws + w.b_bits);
    float *beta = reinterpret_cast<float *>(ws + w.beta);
    float *Zs = reinterpret_cast<float *>(ws + w.z);
    const int words = bigcn_words(K);
    cudaStream_t s = as_stream(stream);
    EventMarks marks(events, n_events, s);
    if (!marks.ok()) return BIGCN_ERR_CUDA;

    // Few long rows: centring, packing and the product in one kernel (the
    // split front), after the weights are packed.
    const bool fused = front_split_supported(N, K, F, dev);
    marks.mark();
    if (!fused) launch_pack_rows(X, N, K, ldx, scale, shift, a_bits, words, alpha, dev, s);
    marks.mark();
    launch_pack_weights(Wt, K, F, ldw, b_bits, words, beta, s);
    marks.mark();
    GemmArgs g{a_bits, alpha, N, b_bits, beta, F, K, words, Zs, F, nullptr, rowptr};
    if (w.bexp_bytes > 0) g.b_e4m3 = reinterpret_cast<uint8_t *>(ws + w.bexp);
    SpmmArgs a{rowptr, colidx, N, nnz, Zs, F, F, H, ldh, true, false};
    if (w.compressed) {
        uint16_t *D16 = reinterpret_cast<uint16_t *>(ws + w.z);
        float *rowscale = reinterpret_cast<float *>(ws + w.rowscale);
        g.Z = nullptr;
        g.dots16 = D16;
        g.ldd16 = w.ldd;
        g.rowscale = rowscale;
        g.dots_f16 = w.f16;
        a.Z = nullptr;
        a.ldz = w.ldd;
        a.D16 = D16;
        a.rowscale = rowscale;
        a.colscale = beta;
    }
    if (fused) {
        FrontArgs fr{X, N, K, ldx, scale, shift, b_bits, beta, F, words, rowptr, g.Z, g.ldz,
                     g.dots16, g.ldd16, g.rowscale, g.dots_f16};
        launch_front(fr, dev, s);
    } else {
        launch_xnor_gemm(g, dev, s);
    }
    marks.mark();
    if (w.f16) {        // fp16 dots: the aggregation on the tensor cores
        SpmmTcArgs t{rowptr, colidx, N, nnz, a.D16, w.ldd, a.rowscale, F, H, ldh, beta, nullptr};
        launch_spmm_tc(t, dev, s);
    } else {
        launch_spmm_norm(a, dev, s);
    }
    marks.mark();
    const bigcn_status ls = launch_status();
    return marks.failed() ? BIGCN_ERR_CUDA : ls;
}

extern "C" bigcn_status bigcn_layer_forward(const float *X, int64_t N, int32_t K, int64_t ldx,
                                            const float *scale, const float *shift,
                                            const float *Wt, int32_t F, int64_t ldw,
                                            const int64_t *rowptr, const int32_t *colidx,
                                            int64_t nnz, void *workspace, size_t ws_bytes,
                                            float *H, int64_t ldh, void *stream) {
    return bigcn_layer_forward_timed(X, N, K, ldx, scale, shift, Wt, F, ldw, rowptr, colidx, nnz,
                                     workspace, ws_bytes, H, ldh, nullptr, 0, stream);
}

// ---------------------------------------------------------------------------
// bigcn_layer_forward_static: the layer for callers that cannot allocate.
//
// Its workspace is this file-scope device array. In host code the name
// g_static_scratch is only a host-side shadow of the symbol, not a device
// address, so the address a kernel may use is looked up once per device with
// cudaGetSymbolAddress (with that device current) and cached.
namespace {
static __device__ __align__(256) unsigned char g_static_scratch[BIGCN_STATIC_SCRATCH_BYTES];

std::once_flag g_scratch_once[kMaxDevices];
void *g_scratch_addr[kMaxDevices];
cudaError_t g_scratch_err[kMaxDevices];

void resolve_static_scratch(int dev) {
    g_scratch_err[dev] = cudaGetSymbolAddress(&g_scratch_addr[dev], g_static_scratch);
    if (g_scratch_err[dev] != cudaSuccess) {
        g_scratch_addr[dev] = nullptr;
        cudaGetLastError();
    }
}
}  // namespace

extern "C" bigcn_status bigcn_layer_forward_static(const float *X, int64_t N, int32_t K,
                                                   int64_t ldx, const float *scale,
                                                   const float *shift, const float *Wt,
                                                   int32_t F, int64_t ldw, const int64_t *rowptr,
                                                   const int32_t *colidx, int64_t nnz, float *H,
                                                   int64_t ldh, void *stream) {
    const size_t need = bigcn_layer_workspace_bytes(N, K, F);
    if (need > BIGCN_STATIC_SCRATCH_BYTES) return BIGCN_ERR_SCRATCH_LIMIT;
    DeviceInfo dev;
    bigcn_status st = current_device(&dev);
    if (st != BIGCN_OK) return st;
    std::call_once(g_scratch_once[dev.device], resolve_static_scratch, dev.device);
    if (g_scratch_err[dev.device] != cudaSuccess) return BIGCN_ERR_CUDA;
    return bigcn_layer_forward(X, N, K, ldx, scale, shift, Wt, F, ldw, rowptr, colidx, nnz,
                               g_scratch_addr[dev.device], BIGCN_STATIC_SCRATCH_BYTES, H, ldh,
                               stream);
}
