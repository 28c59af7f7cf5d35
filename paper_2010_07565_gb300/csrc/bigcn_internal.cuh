// Internal helpers shared by the Bi-GCN CUDA translation units: argument
// checks, the per-device property cache, launch-status mapping and warp-level
// reductions. Not part of the public interface (include/bigcn.h).
#pragma once

#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>

#include "bigcn.h"

namespace bigcn {

constexpr unsigned kFullMask = 0xffffffffu;
constexpr int64_t kMaxElems = int64_t(1) << 62;

struct DeviceInfo {
    int device;
    int sm_count;
    int max_smem_optin;  // bytes of shared memory a block may opt in to
};

// Properties of the current device, queried once per device and cached.
// Returns BIGCN_ERR_UNSUPPORTED unless the device is sm_103.
bigcn_status current_device(DeviceInfo *info);

// Maps the launch result (cudaGetLastError) to a status.
bigcn_status launch_status();

inline bool aligned_to(const void *p, size_t a) {
    return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0;
}

// True when the byte ranges [a, a + na) and [b, b + nb) intersect.
inline bool overlaps(const void *a, size_t na, const void *b, size_t nb) {
    if (a == nullptr || b == nullptr || na == 0 || nb == 0) return false;
    uintptr_t pa = reinterpret_cast<uintptr_t>(a), pb = reinterpret_cast<uintptr_t>(b);
    return pa < pb + nb && pb < pa + na;
}

// Bytes spanned by a rows x cols matrix of elem-byte elements with row stride ld.
inline size_t span_bytes(int64_t rows, int64_t cols, int64_t ld, size_t elem) {
    if (rows <= 0 || cols <= 0) return 0;
    return size_t((rows - 1) * ld + cols) * elem;
}

inline cudaStream_t as_stream(void *s) { return reinterpret_cast<cudaStream_t>(s); }

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(kFullMask, v, o);
    return v;
}

// Programmatic dependent launch. A kernel launched with the programmatic
// stream-serialization attribute may begin while its predecessor in the
// stream is still running; grid_dependency_wait() returns once the
// predecessor grid has completed and its memory writes are visible (at once
// when the launch has no programmatic predecessor). Every kernel calls it
// before it touches anything an earlier kernel writes; work on the call's
// own inputs may come first. allow_dependent_launch() lets the next kernel
// launch before this one finishes.
__device__ __forceinline__ void grid_dependency_wait() {
    asm volatile("griddepcontrol.wait;" ::: "memory");
}
__device__ __forceinline__ void allow_dependent_launch() {
    asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}

// Launches `kernel` with optional programmatic serialization (pdl) and an
// optional cluster shape; the launch error is left for launch_status().
template <typename... KArgs, typename... Args>
void launch_kernel(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                   cudaStream_t stream, bool pdl, dim3 cluster, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    int n = 0;
    if (cluster.x * cluster.y * cluster.z > 1) {
        attr[n].id = cudaLaunchAttributeClusterDimension;
        attr[n].val.clusterDim.x = cluster.x;
        attr[n].val.clusterDim.y = cluster.y;
        attr[n].val.clusterDim.z = cluster.z;
        ++n;
    }
    if (pdl) {
        attr[n].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[n].val.programmaticStreamSerializationAllowed = 1;
        ++n;
    }
    cfg.attrs = attr;
    cfg.numAttrs = n;
    cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

// Records caller-supplied timing events between the kernels of an entry
// point: mark() records the next event of the array (if any is left) on the
// stream. Inside a stream capture an event must be recorded as an external
// node to be timed later; outside a capture a plain record does that.
class EventMarks {
  public:
    EventMarks(void *const *events, int32_t n, cudaStream_t s) : events_(events), n_(n), s_(s) {
        if (n_ > 0 && cudaStreamIsCapturing(s_, &capture_) != cudaSuccess) {
            cudaGetLastError();
            ok_ = false;
        }
    }
    bool ok() const { return ok_; }
    bool failed() const { return failed_; }
    void mark() {
        if (recorded_ < n_) {
            cudaEvent_t ev = static_cast<cudaEvent_t>(events_[recorded_]);
            const cudaError_t r = capture_ == cudaStreamCaptureStatusActive
                                      ? cudaEventRecordWithFlags(ev, s_, cudaEventRecordExternal)
                                      : cudaEventRecord(ev, s_);
            if (r != cudaSuccess) failed_ = true;
        }
        ++recorded_;
    }

  private:
    void *const *events_;
    int32_t n_;
    cudaStream_t s_;
    cudaStreamCaptureStatus capture_ = cudaStreamCaptureStatusNone;
    int32_t recorded_ = 0;
    bool ok_ = true;
    bool failed_ = false;
};

// A dot of Eqs. 11-12 in the compressed forms of a factored product: uint16
// with a bias of 32768 (|dot| <= 32767), or fp16 bits when `f16` (exact for
// |dot| <= 2048); `valid` false gives the zero dot of a padding column.
__device__ __forceinline__ uint16_t encode_dot(int dot, bool valid, bool f16) {
    if (f16) return valid ? __half_as_ushort(__int2half_rn(dot)) : uint16_t(0);
    return uint16_t(valid ? dot + 32768 : 32768);
}

// 1 / sqrt(1 + row length): the D^-1/2 factor of A + I (Sec. 3.1, Eq. 1),
// with IEEE-rounded sqrt and division.
__device__ __forceinline__ float inv_sqrt_degree(int64_t row_len) {
    return 1.0f / sqrtf(1.0f + float(row_len));
}

}  // namespace bigcn
