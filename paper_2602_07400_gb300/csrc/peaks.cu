// Issue-throughput probe behind the roofline peaks of the integer paths.
// The hard layer's mux tree runs on two pipes (IMAD on the FMA pipe, LOP3 on
// the logic pipe); the probe measures what each sustains when nothing else
// limits it.  Every thread runs kChains chains; a step computes each
// chain's next value from its own and its neighbour's previous value (the
// hard tree's mux (x & hi) | (~x & lo), or an integer multiply-add), so the
// chains' operations are independent within a step, and no run of steps is
// a function of three values that one logic operation could replace.
// Unrolled so that loop control is ~2% of the issue slots; the caller times
// the launch with events.  FFMA runs the same loop as the reference for the
// FP32 pipe.  Not part of the method.
#include "common.cuh"

namespace bitlogic {
namespace {

constexpr int kProbeChains = 8;
constexpr int kProbeUnroll = 16;
constexpr int kProbeThreads = 256;
constexpr int kProbeBlocksPerSM = 4;

template <int KIND>
__global__ void __launch_bounds__(kProbeThreads)
issue_probe_kernel(long long iters, uint32_t seed, uint32_t* __restrict__ sink) {
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
    for (long long it = 0; it < iters; ++it) {
#pragma unroll
        for (int u = 0; u < kProbeUnroll; ++u) {
            uint32_t na[kProbeChains];
            float nf[kProbeChains];
#pragma unroll
            for (int i = 0; i < kProbeChains; ++i) {
                const int n = (i + 1) % kProbeChains;
                if constexpr (KIND == BITLOGIC_PROBE_LOP3) na[i] = (a[n] & a[i]) | (~a[n] & b);
                else if constexpr (KIND == BITLOGIC_PROBE_IMAD) na[i] = a[i] * a[n] + c;
                else nf[i] = fmaf(f[i], fb, fc);
            }
#pragma unroll
            for (int i = 0; i < kProbeChains; ++i) {
                if constexpr (KIND == BITLOGIC_PROBE_FFMA) f[i] = nf[i];
                else a[i] = na[i];
            }
        }
    }
    uint32_t r = 0;
#pragma unroll
    for (int i = 0; i < kProbeChains; ++i) r ^= a[i] ^ __float_as_uint(f[i]);
    sink[tid] = r;
}

}  // namespace
}  // namespace bitlogic

extern "C" int64_t bitlogic_issue_probe_threads(void) {
    return (int64_t)bitlogic::sm_count() * bitlogic::kProbeBlocksPerSM * bitlogic::kProbeThreads;
}

extern "C" int64_t bitlogic_issue_probe_ops_per_iter(void) {
    return (int64_t)bitlogic::kProbeChains * bitlogic::kProbeUnroll;
}

extern "C" int bitlogic_issue_probe(int32_t kind, int64_t iters, uint32_t seed, uint32_t* sink,
                                    int64_t sink_len, cudaStream_t stream) {
    using namespace bitlogic;
    if (!sink) return BITLOGIC_ERR_NULL;
    // at most 2^20 iterations: about 1.6 s at the slowest rate measured
    if (iters < 0 || iters > (1ll << 20) || sink_len < bitlogic_issue_probe_threads()) return BITLOGIC_ERR_SHAPE;
    const unsigned grid = (unsigned)(sm_count() * kProbeBlocksPerSM);
    switch (kind) {
        case BITLOGIC_PROBE_LOP3:
            issue_probe_kernel<BITLOGIC_PROBE_LOP3><<<grid, kProbeThreads, 0, stream>>>(iters, seed, sink);
            break;
        case BITLOGIC_PROBE_IMAD:
            issue_probe_kernel<BITLOGIC_PROBE_IMAD><<<grid, kProbeThreads, 0, stream>>>(iters, seed, sink);
            break;
        case BITLOGIC_PROBE_FFMA:
            issue_probe_kernel<BITLOGIC_PROBE_FFMA><<<grid, kProbeThreads, 0, stream>>>(iters, seed, sink);
            break;
        default:
            return BITLOGIC_ERR_SHAPE;
    }
    return launch_status();
}
