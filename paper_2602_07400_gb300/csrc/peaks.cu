// Issue-throughput probe behind the roofline peaks of the integer paths.
// The hard layer's mux tree runs on two pipes (IMAD on the FMA pipe, LOP3 on
// the logic pipe); the probe measures what they sustain when nothing else
// limits it.  One block of 1024 threads per SM (so every SM holds exactly one
// block); every thread runs kProbeChains chains, and a step computes each
// chain's next value from its own and its neighbours' previous values, so
// the chains' operations are independent within a step and no run of steps
// collapses into fewer operations.  Unrolled so that loop control is ~2% of
// the issue slots.  Each block reports the SM clock cycles it ran
// (clock64), so rates come out per SM and clock, whatever the clock.
// Kinds: LOP3 mux with a loop-invariant operand (x & a) | (~x & b); IMAD;
// FFMA (the FP32 pipe, reference); LOP3 mux of three varying registers (the
// form of the hard tree's upper levels); IMAD and that mux interleaved one
// to one (the hard tree's mix).  Not part of the method.
#include "common.cuh"

namespace bitlogic {
namespace {

constexpr int kProbeChains = 8;
constexpr int kProbeUnroll = 16;
constexpr int kProbeThreads = 1024;   // one block per SM

template <int KIND>
__global__ void __launch_bounds__(kProbeThreads, 1)
issue_probe_kernel(long long iters, uint32_t seed, uint32_t* __restrict__ sink, long long* __restrict__ cycles) {
    const uint32_t tid = blockIdx.x * kProbeThreads + threadIdx.x;
    const uint32_t b = seed ^ (tid * 0x9e3779b9u), c = seed + 0x7f4a7c15u * (tid | 1u);
    const float fb = 1.0f + (float)(seed & 7u) * 1e-7f, fc = (float)(tid & 255u) * 1e-9f;
    uint32_t a[kProbeChains];
    float f[kProbeChains];
#pragma unroll
    for (int i = 0; i < kProbeChains; ++i) {
        a[i] = seed + (uint32_t)i * 0x85ebca6bu + tid;
        f[i] = (float)i * 0.125f + fc;
    }
    __syncthreads();
    const long long t0 = clock64();
    for (long long it = 0; it < iters; ++it) {
#pragma unroll
        for (int u = 0; u < kProbeUnroll; ++u) {
            uint32_t na[kProbeChains];
            float nf[kProbeChains];
#pragma unroll
            for (int i = 0; i < kProbeChains; ++i) {
                const int n = (i + 1) % kProbeChains, m = (i + 3) % kProbeChains;
                if constexpr (KIND == BITLOGIC_PROBE_LOP3) na[i] = (a[n] & a[i]) | (~a[n] & b);
                else if constexpr (KIND == BITLOGIC_PROBE_IMAD) na[i] = a[i] * a[n] + c;
                else if constexpr (KIND == BITLOGIC_PROBE_FFMA) nf[i] = fmaf(f[i], fb, fc);
                else if constexpr (KIND == BITLOGIC_PROBE_MUX3) na[i] = (a[n] & a[i]) | (~a[n] & a[m]);
                else na[i] = (i & 1) ? ((a[n] & a[i]) | (~a[n] & a[m])) : a[i] * a[n] + c;   // MIX
            }
#pragma unroll
            for (int i = 0; i < kProbeChains; ++i) {
                if constexpr (KIND == BITLOGIC_PROBE_FFMA) f[i] = nf[i];
                else a[i] = na[i];
            }
        }
    }
    __syncthreads();
    const long long t1 = clock64();
    uint32_t r = 0;
#pragma unroll
    for (int i = 0; i < kProbeChains; ++i) r ^= a[i] ^ __float_as_uint(f[i]);
    sink[tid] = r;
    if (cycles && threadIdx.x == 0) cycles[blockIdx.x] = t1 - t0;
}

}  // namespace
}  // namespace bitlogic

extern "C" int64_t bitlogic_issue_probe_blocks(void) { return (int64_t)bitlogic::sm_count(); }

extern "C" int64_t bitlogic_issue_probe_threads(void) {
    return (int64_t)bitlogic::sm_count() * bitlogic::kProbeThreads;
}

extern "C" int64_t bitlogic_issue_probe_ops_per_iter(void) {
    return (int64_t)bitlogic::kProbeChains * bitlogic::kProbeUnroll;
}

extern "C" int bitlogic_issue_probe(int32_t kind, int64_t iters, uint32_t seed, uint32_t* sink,
                                    int64_t sink_len, int64_t* cycles, cudaStream_t stream) {
    using namespace bitlogic;
    if (!sink) return BITLOGIC_ERR_NULL;
    // at most 2^20 iterations: about 3 s at the slowest rate measured
    if (iters < 0 || iters > (1ll << 20) || sink_len < bitlogic_issue_probe_threads()) return BITLOGIC_ERR_SHAPE;
    const unsigned grid = (unsigned)sm_count();
    long long* cyc = reinterpret_cast<long long*>(cycles);
    switch (kind) {
        case BITLOGIC_PROBE_LOP3:
            issue_probe_kernel<BITLOGIC_PROBE_LOP3><<<grid, kProbeThreads, 0, stream>>>(iters, seed, sink, cyc);
            break;
        case BITLOGIC_PROBE_IMAD:
            issue_probe_kernel<BITLOGIC_PROBE_IMAD><<<grid, kProbeThreads, 0, stream>>>(iters, seed, sink, cyc);
            break;
        case BITLOGIC_PROBE_FFMA:
            issue_probe_kernel<BITLOGIC_PROBE_FFMA><<<grid, kProbeThreads, 0, stream>>>(iters, seed, sink, cyc);
            break;
        case BITLOGIC_PROBE_MUX3:
            issue_probe_kernel<BITLOGIC_PROBE_MUX3><<<grid, kProbeThreads, 0, stream>>>(iters, seed, sink, cyc);
            break;
        case BITLOGIC_PROBE_MIX:
            issue_probe_kernel<BITLOGIC_PROBE_MIX><<<grid, kProbeThreads, 0, stream>>>(iters, seed, sink, cyc);
            break;
        default:
            return BITLOGIC_ERR_SHAPE;
    }
    return launch_status();
}
