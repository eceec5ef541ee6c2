// Soft forward of a LUT layer whose input is binary wires (the thermometer
// encoder's output, §3 "Encoders and heads"), as byte rows (each byte 0 or
// 1) or as wire bit rows (one bit per sample, the training step's form).
//
// The relaxed table of §2, y = sum_a t_a prod_i x_i^{a_i} (1 - x_i)^{1 - a_i},
// has one-hot corner weights on binary inputs: the product is 1 for the
// corner a = sum_i x_i 2^i the inputs sit on and 0 for every other corner, so
// y is the table entry t_a itself.  On byte rows the layer is therefore a
// gather of k bytes and one table read per (node, sample); the first layer of
// the training step sees only such inputs.  Table entries follow the node
// form (the sigmoid of the logit, or [theta > 0] for the straight-through
// node), the same entries the fp32 forward interpolates.
//
// Layout: a warp per node over a batch slice; lanes over 4 consecutive
// samples (one 32-bit load per input row gives the 4 samples' bytes of that
// input); the corner indices of the 4 samples are built byte-wise in one
// register (shift and OR, no carry crosses a byte for k <= 7); the node's
// table (2^k <= 64 entries) sits in two registers per lane and each lookup is
// a shuffle from the lane holding the entry.  Rows are gathered with several
// 128-sample groups in flight per lane.  A scalar form (one sample per lane)
// serves ragged batches and unaligned rows.  The bit-row form takes the
// same lanes and samples with one 32-bit word per input row and 1024-sample
// block in place of the byte loads.
#include "common.cuh"

namespace bitlogic {
namespace {

#ifndef BITLOGIC_BYTES_FWD_GROUPS
#define BITLOGIC_BYTES_FWD_GROUPS 8
#endif
#ifndef BITLOGIC_BYTES_FWD_STREAM
#define BITLOGIC_BYTES_FWD_STREAM 1
#endif
constexpr int kBytesFwdWarps = 8;    // warps (nodes) per block
constexpr int kBytesFwdGroups = BITLOGIC_BYTES_FWD_GROUPS;   // 128-sample groups in flight per lane

__device__ __forceinline__ float node_entry(float th, int node) {
    return node == BITLOGIC_NODE_ST ? (th > 0.f ? 1.f : 0.f) : sigmoidf(th);
}

// Entry a (< 2^k) of the node's table, held as entry lane in `lo` and entry
// 32 + lane in `hi`.  Every lane of the warp takes part.
template <int K>
__device__ __forceinline__ float table_at(float lo, float hi, uint32_t a) {
    const float vlo = __shfl_sync(0xffffffffu, lo, (int)(a & 31u));
    if constexpr (K > 32) {
        const float vhi = __shfl_sync(0xffffffffu, hi, (int)(a & 31u));
        return (a & 32u) ? vhi : vlo;
    } else {
        (void)hi;
        return vlo;
    }
}

template <int k, bool VEC>
__global__ void __launch_bounds__(kBytesFwdWarps * 32)
lut_forward_u8_kernel(const uint8_t* __restrict__ X, int w_in, long long B, const int* __restrict__ conn,
                      const float* __restrict__ theta, int w, int node, float* __restrict__ Y, long long chunk) {
    constexpr int K = 1 << k;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kBytesFwdWarps + warp;
    if (j >= w) return;   // warp-uniform
    const uint8_t* xr[k];
    bool bad = false;
#pragma unroll
    for (int i = 0; i < k; ++i) {
        int c = __ldg(conn + (long long)j * k + i);
        if ((unsigned)c >= (unsigned)w_in) {
            bad = true;
            c = 0;
        }
        xr[i] = X + (long long)c * B;
    }
    if (bad && lane == 0) flag_index_error();
    const float lo = lane < K ? node_entry(__ldg(theta + (long long)j * K + lane), node) : 0.f;
    const float hi = K > 32 ? node_entry(__ldg(theta + (long long)j * K + 32 + (lane & 31)), node) : 0.f;
    const long long s0 = (long long)blockIdx.y * chunk;
    const long long s1 = min(B, s0 + chunk);
    float* yr = Y + (long long)j * B;
    if constexpr (VEC) {
        // lane: samples base + 128 u + 4 lane .. + 3 (B % 4 == 0: all four in range)
        for (long long base = s0; base < s1; base += 128 * kBytesFwdGroups) {
            uint32_t v[kBytesFwdGroups];
#pragma unroll
            for (int u = 0; u < kBytesFwdGroups; ++u) {
                const long long s4 = base + 128 * u + 4 * lane;
                v[u] = 0u;
                if (s4 < s1) {
                    v[u] = __ldg(reinterpret_cast<const uint32_t*>(xr[k - 1] + s4)) & 0x01010101u;
#pragma unroll
                    for (int i = k - 2; i >= 0; --i)
                        v[u] = (v[u] << 1) | (__ldg(reinterpret_cast<const uint32_t*>(xr[i] + s4)) & 0x01010101u);
                }
            }
#pragma unroll
            for (int u = 0; u < kBytesFwdGroups; ++u) {
                const long long s4 = base + 128 * u + 4 * lane;
                float4 y;
                y.x = table_at<K>(lo, hi, v[u] & 0xffu);
                y.y = table_at<K>(lo, hi, (v[u] >> 8) & 0xffu);
                y.z = table_at<K>(lo, hi, (v[u] >> 16) & 0xffu);
                y.w = table_at<K>(lo, hi, v[u] >> 24);
                if (s4 < s1) {
#if BITLOGIC_BYTES_FWD_STREAM
                    __stcs(reinterpret_cast<float4*>(yr + s4), y);
#else
                    *reinterpret_cast<float4*>(yr + s4) = y;
#endif
                }
            }
        }
    } else {
        for (long long base = s0; base < s1; base += 32) {
            const long long s = base + lane;
            uint32_t a = 0u;
            if (s < s1) {
#pragma unroll
                for (int i = 0; i < k; ++i) a |= (uint32_t)(__ldg(xr[i] + s) & 1u) << i;
            }
            const float y = table_at<K>(lo, hi, a);
            if (s < s1) yr[s] = y;
        }
    }
}

// The same forward on wire bit rows (one bit per sample; see kBitBlock): per
// 1024-sample block each lane loads one 32-bit word per input row and finds
// stage r's 4 samples' wires as bytes of (word >> r) & 0x01010101, so the
// layer input is an eighth of the byte rows (12 MB at the CIFAR-100 shape,
// resident in L2) and one load serves 32 samples.  Lanes, samples and
// outputs are those of the byte-row form.  VEC: B % 4 == 0 and 16-byte
// aligned Y (float4 stores), else per-sample stores.
template <int k, bool VEC>
__global__ void __launch_bounds__(kBytesFwdWarps * 32)
lut_forward_bits_kernel(const uint32_t* __restrict__ X, int w_in, long long B, long long words,
                        const int* __restrict__ conn, const float* __restrict__ theta, int w, int node,
                        float* __restrict__ Y, long long chunk_blocks) {
    constexpr int K = 1 << k;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kBytesFwdWarps + warp;
    if (j >= w) return;   // warp-uniform
    const uint32_t* xr[k];
    bool bad = false;
#pragma unroll
    for (int i = 0; i < k; ++i) {
        int c = __ldg(conn + (long long)j * k + i);
        if ((unsigned)c >= (unsigned)w_in) {
            bad = true;
            c = 0;
        }
        xr[i] = X + (long long)c * words + lane;
    }
    if (bad && lane == 0) flag_index_error();
    const float lo = lane < K ? node_entry(__ldg(theta + (long long)j * K + lane), node) : 0.f;
    const float hi = K > 32 ? node_entry(__ldg(theta + (long long)j * K + 32 + (lane & 31)), node) : 0.f;
    const long long nblk = words / 32;
    const long long b0 = (long long)blockIdx.y * chunk_blocks;
    const long long b1 = min(nblk, b0 + chunk_blocks);
    float* yr = Y + (long long)j * B;
    for (long long blk = b0; blk < b1; ++blk) {
        uint32_t wv[k];
#pragma unroll
        for (int i = 0; i < k; ++i) wv[i] = __ldg(xr[i] + blk * 32);
#pragma unroll
        for (int r = 0; r < 8; ++r) {
            const long long s4 = blk * kBitBlock + 128 * r + 4 * lane;
            uint32_t v = (wv[k - 1] >> r) & 0x01010101u;
#pragma unroll
            for (int i = k - 2; i >= 0; --i) v = (v << 1) | ((wv[i] >> r) & 0x01010101u);
            float4 y;
            y.x = table_at<K>(lo, hi, v & 0xffu);
            y.y = table_at<K>(lo, hi, (v >> 8) & 0xffu);
            y.z = table_at<K>(lo, hi, (v >> 16) & 0xffu);
            y.w = table_at<K>(lo, hi, v >> 24);
            if constexpr (VEC) {
                if (s4 < B) __stcs(reinterpret_cast<float4*>(yr + s4), y);
            } else {
                if (s4 < B) yr[s4] = y.x;
                if (s4 + 1 < B) yr[s4 + 1] = y.y;
                if (s4 + 2 < B) yr[s4 + 2] = y.z;
                if (s4 + 3 < B) yr[s4 + 3] = y.w;
            }
        }
    }
}

// Samples per warp: the whole batch unless that leaves fewer than about two
// waves of warps (then slices of at least 512 samples, a multiple of 128).
// Slicing the batch so that a slice of the layer input stays in L2 was
// measured slower (CIFAR-100 shape, 94 MB of byte rows: 321 and 380 us in
// two and three slices against 310 us whole), and an evict-last L2 policy
// on the gathers changed nothing (311 us).
long long forward_u8_chunk(int w, long long B) {
    const long long wanted = 2ll * sm_count() * 64;
    long long c = (long long)w * B / wanted;
    c = (c / 128) * 128;
    if (c < 512) c = 512;
    return c < B ? c : B;
}

template <int k>
int launch_forward_u8(const uint8_t* X, int w_in, long long B, const int* conn, const float* theta, int w,
                      int node, float* Y, cudaStream_t st) {
    const bool vec = (B % 4 == 0) && ((reinterpret_cast<uintptr_t>(X) & 3u) == 0) && aligned16(Y);
    long long chunk = forward_u8_chunk(w, B);
    if (vec) chunk = (chunk + 3) / 4 * 4;
    const long long ny = (B + chunk - 1) / chunk;
    if (ny > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((w + kBytesFwdWarps - 1) / kBytesFwdWarps), (unsigned)ny);
    if (vec)
        lut_forward_u8_kernel<k, true><<<grid, kBytesFwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, node, Y,
                                                                            chunk);
    else
        lut_forward_u8_kernel<k, false><<<grid, kBytesFwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, node, Y,
                                                                             chunk);
    return launch_status();
}

template <int k>
int launch_forward_bits(const uint32_t* X, int w_in, long long B, const int* conn, const float* theta, int w,
                        int node, float* Y, cudaStream_t st) {
    const long long nblk = (B + kBitBlock - 1) / kBitBlock;
    long long chunk = (forward_u8_chunk(w, B) + kBitBlock - 1) / kBitBlock;   // in blocks
    if (chunk < 1) chunk = 1;
    const long long ny = (nblk + chunk - 1) / chunk;
    if (ny > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((w + kBytesFwdWarps - 1) / kBytesFwdWarps), (unsigned)ny);
    if (B % 4 == 0 && aligned16(Y))
        lut_forward_bits_kernel<k, true><<<grid, kBytesFwdWarps * 32, 0, st>>>(X, w_in, B, nblk * 32, conn, theta,
                                                                               w, node, Y, chunk);
    else
        lut_forward_bits_kernel<k, false><<<grid, kBytesFwdWarps * 32, 0, st>>>(X, w_in, B, nblk * 32, conn, theta,
                                                                                w, node, Y, chunk);
    return launch_status();
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(lut_bytes)

extern "C" int bitlogic_lut_forward_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                                       const float* theta, int32_t w, int32_t k, int32_t node, float* Y,
                                       cudaStream_t stream) {
    if (!conn || !theta) return BITLOGIC_ERR_NULL;
    if (B > 0 && (!X || !Y)) return BITLOGIC_ERR_NULL;   // an empty batch may come as NULL
    if (w_in <= 0 || w <= 0 || B < 0) return BITLOGIC_ERR_SHAPE;
    if (k < 1 || k > 6 || k > w_in) return BITLOGIC_ERR_FANIN;
    if ((int64_t)w * k > 0x7fffffffLL) return BITLOGIC_ERR_SHAPE;
    if (node != BITLOGIC_NODE_SOFT && node != BITLOGIC_NODE_ST) return BITLOGIC_ERR_NODE;
    if (B == 0) return BITLOGIC_OK;
    switch (k) {
        case 1: return launch_forward_u8<1>(X, w_in, B, conn, theta, w, node, Y, stream);
        case 2: return launch_forward_u8<2>(X, w_in, B, conn, theta, w, node, Y, stream);
        case 3: return launch_forward_u8<3>(X, w_in, B, conn, theta, w, node, Y, stream);
        case 4: return launch_forward_u8<4>(X, w_in, B, conn, theta, w, node, Y, stream);
        case 5: return launch_forward_u8<5>(X, w_in, B, conn, theta, w, node, Y, stream);
        default: return launch_forward_u8<6>(X, w_in, B, conn, theta, w, node, Y, stream);
    }
}

extern "C" int bitlogic_lut_forward_bitrows(const uint32_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                                            const float* theta, int32_t w, int32_t k, int32_t node, float* Y,
                                            cudaStream_t stream) {
    if (!conn || !theta) return BITLOGIC_ERR_NULL;
    if (B > 0 && (!X || !Y)) return BITLOGIC_ERR_NULL;   // an empty batch may come as NULL
    if (w_in <= 0 || w <= 0 || B < 0) return BITLOGIC_ERR_SHAPE;
    if (k < 1 || k > 6 || k > w_in) return BITLOGIC_ERR_FANIN;
    if ((int64_t)w * k > 0x7fffffffLL) return BITLOGIC_ERR_SHAPE;
    if (node != BITLOGIC_NODE_SOFT && node != BITLOGIC_NODE_ST) return BITLOGIC_ERR_NODE;
    if (B == 0) return BITLOGIC_OK;
    if ((reinterpret_cast<uintptr_t>(X) & 3u) != 0) return BITLOGIC_ERR_ALIGN;
    switch (k) {
        case 1: return launch_forward_bits<1>(X, w_in, B, conn, theta, w, node, Y, stream);
        case 2: return launch_forward_bits<2>(X, w_in, B, conn, theta, w, node, Y, stream);
        case 3: return launch_forward_bits<3>(X, w_in, B, conn, theta, w, node, Y, stream);
        case 4: return launch_forward_bits<4>(X, w_in, B, conn, theta, w, node, Y, stream);
        case 5: return launch_forward_bits<5>(X, w_in, B, conn, theta, w, node, Y, stream);
        default: return launch_forward_bits<6>(X, w_in, B, conn, theta, w, node, Y, stream);
    }
}
