// Internal helpers shared by the CUDA translation units of libbitlogic.
#pragma once

#include <cstdint>
#include <cuda_runtime.h>

#include "bitlogic.h"

namespace bitlogic {

// Device-side index flag.  `static` gives each translation unit its own
// copy; every unit registers a reader with bitlogic_device_error().
static __device__ unsigned int g_index_error;

__device__ __forceinline__ void flag_index_error() { atomicOr(&g_index_error, 1u); }

// Reads and clears this unit's flag (synchronizes the stream).
static inline int read_and_clear_index_error(cudaStream_t stream) {
    unsigned int v = 0, zero = 0;
    if (cudaMemcpyFromSymbolAsync(&v, g_index_error, sizeof(v), 0,
                                  cudaMemcpyDeviceToHost, stream) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    if (cudaMemcpyToSymbolAsync(g_index_error, &zero, sizeof(zero), 0,
                                cudaMemcpyHostToDevice, stream) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return BITLOGIC_ERR_CUDA;
    return v ? BITLOGIC_ERR_DEVICE : BITLOGIC_OK;
}

inline int launch_status() {
    return cudaGetLastError() == cudaSuccess ? BITLOGIC_OK : BITLOGIC_ERR_CUDA;
}

inline bool aligned16(const void* p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Number of SMs of the current device (queried once per device, then
// cached; 152 if the query fails).  Defined in abi.cu.
int sm_count();

// Wire bit rows (the layer-1 input at one bit per sample): samples per word
// block; a row holds 32 words per block, bit 8 m + r of word L being the
// block's sample 128 r + 4 L + m.
constexpr int kBitBlock = 1024;

// Thresholds travel by value in the kernel parameters: no constant-memory
// state is shared between calls or streams.
struct Thresholds {
    int b;
    uint8_t t[32];
};

// Threshold i of a by-value Thresholds with a compile-time unrolled select
// (a runtime index into kernel parameters would copy them to local memory).
__device__ __forceinline__ uint32_t threshold_at(const Thresholds& th, int i) {
    uint32_t v = 0;
#pragma unroll
    for (int q = 0; q < 32; ++q)
        if (q == i) v = th.t[q];
    return v;
}

inline int make_thresholds(const uint8_t* thr_host, int32_t b, Thresholds* out) {
    if (!thr_host) return BITLOGIC_ERR_NULL;
    if (b < 1 || b > 32) return BITLOGIC_ERR_THRESH;
    out->b = b;
    for (int i = 0; i < 32; ++i) out->t[i] = i < b ? thr_host[i] : 0;
    return BITLOGIC_OK;
}

// Logistic function on the CUDA-core FP32 path: CUDA's expf and an
// IEEE-rounded division (no fast-math).
__device__ __forceinline__ float sigmoidf(float z) { return 1.0f / (1.0f + expf(-z)); }

// Asynchronous 16-byte global -> shared copies (cp.async, bypassing L1),
// grouped per pipeline stage.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    const unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

// Programmatic dependent launch (sm_90 and later).  A kernel launched with
// launch_dependent() may start while the kernel before it on the stream is
// still finishing: it runs grid_dependency_wait() before its first access to
// memory that the earlier work writes or reads, and the wait returns once that
// work has completed with its writes visible.  The earlier kernel lets its
// dependent start early with allow_dependent_launch() (else the dependent
// starts as its blocks exit).  When the previous operation on the stream is
// not a kernel, the launch is an ordinary one and the wait returns at once.
__device__ __forceinline__ void grid_dependency_wait() { asm volatile("griddepcontrol.wait;\n" ::: "memory"); }
__device__ __forceinline__ void allow_dependent_launch() {
    asm volatile("griddepcontrol.launch_dependents;\n" ::: "memory");
}

// First statement of every kernel launched with launch_dependent(): wait for
// the work before it on the stream, then let the next kernel be scheduled.
// Waiting before triggering makes the chain transitive: once a kernel's wait
// returns, everything before its predecessor has completed too.
__device__ __forceinline__ void dependent_kernel_start() {
    grid_dependency_wait();
    allow_dependent_launch();
}

template <typename... KArgs, typename... Args>
inline cudaError_t launch_dependent(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem,
                                    cudaStream_t stream, Args... args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<KArgs>(args)...);
}

}  // namespace bitlogic

#define BITLOGIC_ERROR_READER(name)                                            \
    extern "C" int bitlogic_internal_index_error_##name(cudaStream_t s) {      \
        return bitlogic::read_and_clear_index_error(s);                        \
    }
