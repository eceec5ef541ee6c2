// Thermometer encoder (paper §3 "Encoders and heads": the linear thermometer
// emits b+1 levels on b wires; wire j*b + i of feature j is x_j > T_i, with
// the strict comparison of App. B's "(pixel > 0)").
//
// Two forms:
//   * soft:   fp32 {0,1} rows [d*b][B] feeding the first soft LUT layer;
//   * packed: 32 samples per uint32 along the batch (App. C.1 "Bit-packed
//     inference" packs samples along the batch into machine words), fused
//     with the comparison so the fp32 form is never materialised.
//
// Both stage a tile of raw samples (sample-major uint8) in shared memory and
// write feature-major rows, so global reads and writes are coalesced.
#include "common.cuh"

namespace bitlogic {
namespace {

// ----------------------------------------------------------------- soft --

constexpr int kEncTS = 64;   // samples per tile
constexpr int kEncTF = 32;   // features per tile

__global__ void __launch_bounds__(256)
encode_soft_kernel(const uint8_t* __restrict__ x, long long B, int d, Thresholds th,
                   float* __restrict__ bits) {
    __shared__ uint8_t tile[kEncTF][kEncTS + 4];   // feature-major
    const long long s0 = (long long)blockIdx.y * kEncTS;
    const int f0 = blockIdx.x * kEncTF;
    // load: thread t reads features f0 + (t % 32) of samples s0 + t/32 + 8q
    const int tf = threadIdx.x & 31, ts = threadIdx.x >> 5;
#pragma unroll
    for (int q = 0; q < kEncTS / 8; ++q) {
        const int sl = ts + 8 * q;
        const long long s = s0 + sl;
        uint8_t v = 0;
        if (s < B && f0 + tf < d) v = __ldg(x + s * d + f0 + tf);
        tile[tf][sl] = v;
    }
    __syncthreads();
    // store: rows (f, i) of kEncTS samples; 4 rows per pass of 256 threads
    const int nf = min(kEncTF, d - f0);
    const int rows = nf * th.b;
    const int tsl = threadIdx.x & 63, tr = threadIdx.x >> 6;
    const long long s = s0 + tsl;
    if (s >= B) return;
    for (int r = tr; r < rows; r += 4) {
        const int f = r / th.b, i = r - f * th.b;
        bits[((long long)(f0 + f) * th.b + i) * B + s] = tile[f][tsl] > th.t[i] ? 1.0f : 0.0f;
    }
}

// --------------------------------------------------------------- packed --

constexpr int kPackWords = 32;             // words per tile (1024 samples)
constexpr int kPackTS = kPackWords * 32;   // samples per tile
constexpr int kPackTF = 8;                 // features per tile
constexpr int kPackWarps = 8;

__global__ void __launch_bounds__(kPackWarps * 32)
pack_bits_kernel(const uint8_t* __restrict__ x, long long N, int d, Thresholds th,
                 uint32_t* __restrict__ xp, long long W, bool vec8) {
    __shared__ __align__(16) uint8_t tile[kPackTS][kPackTF];   // sample-major, 8-byte rows
    __shared__ uint32_t stage[kPackTF * 32][kPackWords];       // [wire in tile][word]
    const long long s0 = (long long)blockIdx.y * kPackTS;
    const int f0 = blockIdx.x * kPackTF;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nf = min(kPackTF, d - f0);
    // load 1024 samples x 8 features
    for (int sl = threadIdx.x; sl < kPackTS; sl += kPackWarps * 32) {
        const long long s = s0 + sl;
        uint2 v = make_uint2(0u, 0u);
        if (s < N) {
            const uint8_t* p = x + s * d + f0;
            if (vec8 && nf == kPackTF) {
                v = __ldg(reinterpret_cast<const uint2*>(p));
            } else {
                uint8_t b8[8] = {0, 0, 0, 0, 0, 0, 0, 0};
                for (int f = 0; f < nf; ++f) b8[f] = __ldg(p + f);
                v.x = b8[0] | (b8[1] << 8) | (b8[2] << 16) | ((uint32_t)b8[3] << 24);
                v.y = b8[4] | (b8[5] << 8) | (b8[6] << 16) | ((uint32_t)b8[7] << 24);
            }
        }
        *reinterpret_cast<uint2*>(&tile[sl][0]) = v;
    }
    __syncthreads();
    // each warp builds 4 words: lane = sample bit, one ballot per wire
#pragma unroll
    for (int u = 0; u < kPackWords / kPackWarps; ++u) {
        const int q = warp * (kPackWords / kPackWarps) + u;
        const uint2 v = *reinterpret_cast<const uint2*>(&tile[q * 32 + lane][0]);
        for (int f = 0; f < nf; ++f) {
            const uint32_t byte = ((f < 4 ? v.x : v.y) >> (8 * (f & 3))) & 0xffu;
            for (int i = 0; i < th.b; ++i) {
                const uint32_t word = __ballot_sync(0xffffffffu, byte > th.t[i]);
                if (lane == 0) stage[f * th.b + i][q] = word;
            }
        }
    }
    __syncthreads();
    // coalesced store: one 128-byte row segment per warp step
    const long long q0 = (long long)blockIdx.y * kPackWords;
    const int rows = nf * th.b;
    for (int r = warp; r < rows; r += kPackWarps) {
        const long long q = q0 + lane;
        if (q < W) {
            const int f = r / th.b, i = r - f * th.b;
            xp[((long long)(f0 + f) * th.b + i) * W + q] = stage[r][lane];
        }
    }
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(encode)

extern "C" int bitlogic_encode_thermometer(const uint8_t* x, int64_t B, int32_t d,
                                           const uint8_t* thr_host, int32_t b,
                                           float* bits, cudaStream_t stream) {
    Thresholds th;
    int st = make_thresholds(thr_host, b, &th);
    if (st) return st;
    if (B < 0 || d <= 0) return BITLOGIC_ERR_SHAPE;
    if (B == 0) return BITLOGIC_OK;   // an empty batch may come as NULL
    if (!x || !bits) return BITLOGIC_ERR_NULL;
    const long long gy = (B + kEncTS - 1) / kEncTS;
    if (gy > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((d + kEncTF - 1) / kEncTF), (unsigned)gy);
    encode_soft_kernel<<<grid, 256, 0, stream>>>(x, B, d, th, bits);
    return launch_status();
}

extern "C" int bitlogic_pack_bits(const uint8_t* x, int64_t N, int32_t d,
                                  const uint8_t* thr_host, int32_t b,
                                  uint32_t* xp, cudaStream_t stream) {
    Thresholds th;
    int st = make_thresholds(thr_host, b, &th);
    if (st) return st;
    if (N < 0 || d <= 0) return BITLOGIC_ERR_SHAPE;
    if (N == 0) return BITLOGIC_OK;   // an empty batch may come as NULL
    if (!x || !xp) return BITLOGIC_ERR_NULL;
    const long long W = (N + 31) / 32;
    const long long gy = (N + kPackTS - 1) / kPackTS;
    if (gy > 65535) return BITLOGIC_ERR_SHAPE;
    const bool vec8 = (d % 8 == 0) && ((reinterpret_cast<uintptr_t>(x) & 7u) == 0);
    dim3 grid((unsigned)((d + kPackTF - 1) / kPackTF), (unsigned)gy);
    pack_bits_kernel<<<grid, kPackWarps * 32, 0, stream>>>(x, N, d, th, xp, W, vec8);
    return launch_status();
}
