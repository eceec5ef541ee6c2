// Distributive (quantile) thermometer fit (paper §3 "Encoders and heads";
// App. A "Initialization": the thresholds are fit once from the empirical
// pixel quantiles of the training split; App. B: over the globally flattened
// pixel distribution).
//
// The quantiles of uint8 pixels follow from their 256-bin histogram, so the
// device work is one pass over the training pixels that counts values; the
// threshold for level i/(b+1) is then read off the cumulative counts on the
// host (256 bins) in exact integer arithmetic.
//
// Histogram: every warp owns 16 copies of a 256-bin shared histogram and
// lane l adds into copy l % 16 with a shared atomic whose result is unused,
// so lanes rarely contend (two lanes per copy) even on a point mass (the zero
// pixels of digit images), and no add waits for another.  Each thread keeps
// 8 independent 16-byte loads in flight.  Blocks publish their counts with
// 64-bit integer atomics: exact and independent of the order.
#include "common.cuh"

namespace bitlogic {
namespace {

constexpr int kHistWarps = 4;
constexpr int kHistCopies = 16;   // lane l adds into copy l % kHistCopies
constexpr int kHistLoads = 8;     // 16-byte loads in flight per thread
constexpr int kHistSmem = kHistWarps * 256 * kHistCopies * 4;

// x16: the 16-byte aligned middle of the input (n16 chunks); head/tail:
// the bytes before and after it (< 16 each), counted by block 0.
__global__ void __launch_bounds__(kHistWarps * 32)
pixel_histogram_kernel(const uint4* __restrict__ x16, long long n16, const uint8_t* __restrict__ head,
                       int n_head, const uint8_t* __restrict__ tail, int n_tail,
                       unsigned long long* __restrict__ hist) {
    extern __shared__ unsigned int sh[];   // [warp][bin][copy]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    for (int i = threadIdx.x; i < kHistWarps * 256 * kHistCopies; i += blockDim.x) sh[i] = 0u;
    __syncthreads();
    unsigned int* h = sh + warp * 256 * kHistCopies + (lane & (kHistCopies - 1));
    auto count = [&](uint32_t w) {
#pragma unroll
        for (int byte = 0; byte < 4; ++byte) atomicAdd(h + ((w >> (8 * byte)) & 0xffu) * kHistCopies, 1u);
    };
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long c0 = (long long)blockIdx.x * blockDim.x + threadIdx.x; c0 < n16;
         c0 += stride * kHistLoads) {
        uint4 v[kHistLoads];
#pragma unroll
        for (int u = 0; u < kHistLoads; ++u) {
            const long long c = c0 + u * stride;
            if (c < n16) v[u] = __ldg(x16 + c);
        }
#pragma unroll
        for (int u = 0; u < kHistLoads; ++u) {
            if (c0 + u * stride < n16) {
                count(v[u].x);
                count(v[u].y);
                count(v[u].z);
                count(v[u].w);
            }
        }
    }
    if (blockIdx.x == 0 && threadIdx.x < 32) {
        if (lane < n_head) atomicAdd(h + (unsigned)head[lane] * kHistCopies, 1u);
        if (lane < n_tail) atomicAdd(h + (unsigned)tail[lane] * kHistCopies, 1u);
    }
    __syncthreads();
    for (int v = threadIdx.x; v < 256; v += blockDim.x) {
        unsigned long long s = 0;
        for (int q = 0; q < kHistWarps; ++q) {
            const unsigned int* row = sh + (q * 256 + v) * kHistCopies;
#pragma unroll
            for (int c = 0; c < kHistCopies; ++c) s += row[c];
        }
        if (s) atomicAdd(hist + v, s);
    }
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

extern "C" int bitlogic_pixel_histogram(const uint8_t* x, int64_t n, uint64_t* hist, cudaStream_t stream) {
    if (n < 0) return BITLOGIC_ERR_SHAPE;
    if (n == 0) return BITLOGIC_OK;
    if (!x || !hist) return BITLOGIC_ERR_NULL;
    const uintptr_t addr = reinterpret_cast<uintptr_t>(x);
    long long n_head = (long long)((16 - (addr & 15)) & 15);
    if (n_head > n) n_head = n;
    const long long n16 = (n - n_head) / 16;
    const long long n_tail = n - n_head - 16 * n16;
    const uint4* x16 = reinterpret_cast<const uint4*>(x + n_head);
    // three blocks per SM (the shared histograms take 64 KB each), fewer
    // for small inputs
    const long long per_block = (long long)kHistWarps * 32 * kHistLoads;
    long long blocks = (n16 + per_block - 1) / per_block;
    const long long cap = (long long)sm_count() * 3;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    if (cudaFuncSetAttribute(pixel_histogram_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, kHistSmem) !=
        cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    pixel_histogram_kernel<<<(unsigned)blocks, kHistWarps * 32, kHistSmem, stream>>>(
        x16, n16, x, (int)n_head, x + n_head + 16 * n16, (int)n_tail,
        reinterpret_cast<unsigned long long*>(hist));
    return launch_status();
}

extern "C" int bitlogic_quantile_thresholds(const uint64_t* hist_host, int32_t b, uint8_t* thr_host) {
    if (!hist_host || !thr_host) return BITLOGIC_ERR_NULL;
    if (b < 1 || b > 32) return BITLOGIC_ERR_THRESH;
    uint64_t n = 0;
    for (int v = 0; v < 256; ++v) {
        if (hist_host[v] > (UINT64_MAX >> 7) - n) return BITLOGIC_ERR_SHAPE;   // keeps (n-1)*32 in range
        n += hist_host[v];
    }
    if (n == 0) return BITLOGIC_ERR_SHAPE;
    // value of the order statistic of rank r (0-based): the smallest v whose
    // cumulative count exceeds r
    auto order_stat = [&](uint64_t r) {
        uint64_t cum = 0;
        for (int v = 0; v < 256; ++v) {
            cum += hist_host[v];
            if (cum > r) return v;
        }
        return 255;
    };
    for (int i = 1; i <= b; ++i) {
        // level i/(b+1): h = (n-1) i/(b+1) = lo + rem/(b+1)
        const uint64_t num = (n - 1) * (uint64_t)i;
        const uint64_t lo = num / (uint64_t)(b + 1), rem = num % (uint64_t)(b + 1);
        const int v_lo = order_stat(lo);
        const int v_hi = lo + 1 < n ? order_stat(lo + 1) : v_lo;
        thr_host[i - 1] = (uint8_t)(v_lo + (int)((rem * (uint64_t)(v_hi - v_lo)) / (uint64_t)(b + 1)));
    }
    return BITLOGIC_OK;
}
