// Thermometer encoder (paper §3 "Encoders and heads": the linear thermometer
// emits b+1 levels on b wires; wire j*b + i of feature j is x_j > T_i, with
// the strict comparison of App. B's "(pixel > 0)").
//
// Three forms:
//   * soft:     fp32 {0,1} rows [d*b][B] (or bytes 0/1) feeding the first
//     soft LUT layer;
//   * bit rows: the soft layer-1 input at one bit per sample, in the order
//     of the layer-1 kernels' lanes (below);
//   * packed:   32 samples per uint32 along the batch (App. C.1 "Bit-packed
//     inference" packs samples along the batch into machine words), fused
//     with the comparison so the fp32 form is never materialised.
//
// All stage a tile of raw samples (sample-major uint8) in shared memory and
// write feature-major rows, so global reads and writes are coalesced.
#include "common.cuh"

namespace bitlogic {
namespace {

// ----------------------------------------------------------------- soft --

constexpr int kEncTS = 64;   // samples per tile
constexpr int kEncTF = 32;   // features per tile

// Output wires as fp32 (the soft layers' input) or as bytes (byte-row
// consumers such as the routing gathers).
__device__ __forceinline__ void put_bit(float* p, bool v) { *p = v ? 1.0f : 0.0f; }
__device__ __forceinline__ void put_bit(uint8_t* p, bool v) { *p = v ? 1u : 0u; }
// The 4 comparisons of a SWAR test (bit 7 of byte r set: sample r's wire is 1).
__device__ __forceinline__ void put_high_bits4(float* p, uint32_t hb) {
    *reinterpret_cast<float4*>(p) = make_float4((hb & 0x80u) ? 1.0f : 0.0f, (hb & 0x8000u) ? 1.0f : 0.0f,
                                                (hb & 0x800000u) ? 1.0f : 0.0f, (hb & 0x80000000u) ? 1.0f : 0.0f);
}
__device__ __forceinline__ void put_high_bits4(uint8_t* p, uint32_t hb) {
    *reinterpret_cast<uint32_t*>(p) = hb >> 7;
}

// Byte-wise test v > T on 4 bytes at once (no carry crosses a byte):
//   T < 127:  v > T  <=>  v >= 128 or (v & 127) + (127 - T) >= 128
//   T >= 127: v > T  <=>  v >= 128 and (v & 127) + (255 - T) >= 128
// with C = the byte constant times 0x01010101 and `orf` the first form;
// returns the high bits 0x80 of the bytes whose test holds.
struct ThresholdSwar {
    uint32_t C;
    bool orf;
};
__device__ __forceinline__ ThresholdSwar threshold_swar(uint32_t T) {
    // T == 255: nothing exceeds it (C = 0, AND form: the sum never reaches 128)
    return ThresholdSwar{(T < 127u ? 127u - T : 255u - T) * 0x01010101u, T < 127u};
}
__device__ __forceinline__ uint32_t swar_greater(uint32_t q, uint32_t lo7, const ThresholdSwar& t) {
    return (t.orf ? (q | (lo7 + t.C)) : (q & (lo7 + t.C))) & 0x80808080u;
}

template <typename OutT>
__global__ void __launch_bounds__(256)
encode_soft_kernel(const uint8_t* __restrict__ x, long long B, int d, Thresholds th,
                   OutT* __restrict__ bits, uint8_t* __restrict__ bits8) {
    __shared__ uint8_t tile[kEncTF][kEncTS + 4];   // feature-major
    __shared__ uint32_t sT[32];
    if (threadIdx.x < th.b) sT[threadIdx.x] = threshold_at(th, threadIdx.x);
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
        const long long o = ((long long)(f0 + f) * th.b + i) * B + s;
        const bool v = tile[f][tsl] > sT[i];
        put_bit(bits + o, v);
        if (bits8) put_bit(bits8 + o, v);   // the same wires as bytes
    }
}

// Vector form (B % 4 == 0, 16-byte aligned output): tiles of 32 features x
// 128 samples; each thread loads 16 feature bytes of one sample (one 16-byte
// load when d % 16 == 0 and x is aligned), the tile is transposed through
// shared memory, and each thread writes 4 consecutive samples of a wire row
// as one float4 (512 contiguous bytes per warp).
constexpr int kEncVS = 128;   // samples per tile (vector form)

template <typename OutT>
__global__ void __launch_bounds__(256)
encode_soft_vec_kernel(const uint8_t* __restrict__ x, long long B, int d, Thresholds th,
                       OutT* __restrict__ bits, uint8_t* __restrict__ bits8, bool vec16) {
    __shared__ __align__(16) uint8_t tile[kEncTF][kEncVS];   // feature-major
    __shared__ ThresholdSwar sT[32];
    if (threadIdx.x < th.b) sT[threadIdx.x] = threshold_swar(threshold_at(th, threadIdx.x));
    const long long s0 = (long long)blockIdx.y * kEncVS;
    const int f0 = blockIdx.x * kEncTF;
    const int nf = min(kEncTF, d - f0);
    {   // thread t: sample t / 2, features 16 (t % 2) .. 16 (t % 2) + 15
        const int sl = threadIdx.x >> 1, half = threadIdx.x & 1;
        const long long s = s0 + sl;
        uint32_t v[4] = {0u, 0u, 0u, 0u};
        if (s < B) {
            const uint8_t* p = x + s * d + f0 + 16 * half;
            if (vec16 && nf == kEncTF) {
                const uint4 a = __ldg(reinterpret_cast<const uint4*>(p));
                v[0] = a.x; v[1] = a.y; v[2] = a.z; v[3] = a.w;
            } else {
#pragma unroll
                for (int f = 0; f < 16; ++f)
                    if (16 * half + f < nf) v[f >> 2] |= (uint32_t)__ldg(p + f) << (8 * (f & 3));
            }
        }
#pragma unroll
        for (int f = 0; f < 16; ++f) tile[16 * half + f][sl] = (uint8_t)(v[f >> 2] >> (8 * (f & 3)));
    }
    __syncthreads();
    // warp w: features w, w + 8, ...; per feature one shared load of the
    // lane's 4 samples and, per threshold, a byte-wise test of all four
    const int u = threadIdx.x & 31, rg = threadIdx.x >> 5;
    const long long s = s0 + 4 * u;
    if (s >= B) return;   // B % 4 == 0: the thread's four samples are in range
    for (int f = rg; f < nf; f += 8) {
        const uint32_t q = *reinterpret_cast<const uint32_t*>(&tile[f][4 * u]);
        const uint32_t lo7 = q & 0x7f7f7f7fu;
        const long long o = (long long)(f0 + f) * th.b * B + s;
        OutT* out = bits + o;
        uint8_t* out8 = bits8 ? bits8 + o : nullptr;
        for (int i = 0; i < th.b; ++i) {
            const uint32_t hb = swar_greater(q, lo7, sT[i]);
            put_high_bits4(out + (long long)i * B, hb);
            if (out8) put_high_bits4(out8 + (long long)i * B, hb);   // the same wires as bytes
        }
    }
}

// ------------------------------------------------------------- bit rows --
//
// Layer-1 wires at one bit per sample for the soft layer-1 kernels (a
// thirty-second of fp32 rows, an eighth of byte rows), in the order of those
// kernels' lanes: the batch is cut into 1024-sample blocks of 32 words per
// wire, and bit 8 m + r of word L of a block is the wire of the block's sample
// 128 r + 4 L + m (r < 8, m < 4).  Lane L of a layer-1 kernel, taking samples
// 128 r + 4 L .. + 3 of the block (stage r), finds their four wires as bytes
// 0 .. 3 of (word >> r) & 0x01010101.  Samples past B have wire 0.
//
// A block encodes 8 features (one per warp) over one 1024-sample block: the
// raw bytes go to a feature-major shared tile, then lane L reads its 8
// stages' 4 pixels (one 32-bit word each) and per threshold assembles its
// word from the byte-wise comparisons.
constexpr int kBitsTF = 8;   // features per block (one per warp)

__global__ void __launch_bounds__(256)
encode_bitrows_kernel(const uint8_t* __restrict__ x, long long B, int d, Thresholds th,
                      uint32_t* __restrict__ bits, long long words, bool vec8) {
    __shared__ __align__(16) uint8_t tile[kBitsTF][kBitBlock];   // feature-major
    __shared__ ThresholdSwar sT[32];
    if (threadIdx.x < th.b) sT[threadIdx.x] = threshold_swar(threshold_at(th, threadIdx.x));
    const long long s0 = (long long)blockIdx.y * kBitBlock;
    const int f0 = blockIdx.x * kBitsTF;
    const int nf = min(kBitsTF, d - f0);
#pragma unroll
    for (int q = 0; q < kBitBlock / 256; ++q) {   // thread t: samples t, t + 256, ...
        const int sl = threadIdx.x + 256 * q;
        const long long s = s0 + sl;
        uint32_t lo = 0u, hi = 0u;   // the sample's 8 feature bytes
        if (s < B) {
            const uint8_t* p = x + s * d + f0;
            if (vec8 && nf == kBitsTF) {
                const uint2 v = __ldg(reinterpret_cast<const uint2*>(p));
                lo = v.x;
                hi = v.y;
            } else {
                for (int f = 0; f < nf; ++f) {
                    const uint32_t v = __ldg(p + f);
                    if (f < 4) lo |= v << (8 * f);
                    else hi |= v << (8 * (f - 4));
                }
            }
        }
#pragma unroll
        for (int f = 0; f < kBitsTF; ++f) tile[f][sl] = (uint8_t)((f < 4 ? lo : hi) >> (8 * (f & 3)));
    }
    __syncthreads();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (warp >= nf) return;
    uint32_t q[8], lo7[8];
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        q[r] = *reinterpret_cast<const uint32_t*>(&tile[warp][128 * r + 4 * lane]);
        lo7[r] = q[r] & 0x7f7f7f7fu;
    }
    uint32_t* out = bits + (long long)(f0 + warp) * th.b * words + (long long)blockIdx.y * 32 + lane;
    for (int i = 0; i < th.b; ++i) {
        const ThresholdSwar t = sT[i];
        uint32_t word = 0u;
#pragma unroll
        for (int r = 0; r < 8; ++r) word |= (swar_greater(q[r], lo7[r], t) >> 7) << r;
        out[(long long)i * words] = word;
    }
}

// --------------------------------------------------------------- packed --
//
// One lane per output word (32 samples), so every store is a coalesced
// 128-byte run of a wire row.  A block takes 1024 samples x 32 features.
// Sample group (q, r) of word q holds samples 32q + r + 8j (j < 4): a 32-bit
// register of one feature over those four samples is one byte per sample.
//
// Fill: thread 8q + r loads the 32 feature bytes of the four samples of group
// (q, r) and transposes each 4 x 4 byte block (4 samples x 4 features) with
// two rounds of byte permutes into four words, one per feature.  The shared
// tile is [feature quad][sample group][feature in quad]: the four words of a
// block are one 16-byte cell, written with one 16-byte store (8 per thread).
// Cells are XOR-swizzled within each word's 8 groups (cell r ^ (q & 7)), so
// the 8 lanes of a 16-byte access phase always hit 8 different bank groups,
// both in the fill (lanes = the 8 groups of one word) and in the compare
// (lanes = 8 words, one group each).
//
// Compare: warp w takes feature quad w; lane q reads the 8 cells of its word
// (8 sixteen-byte loads: four features x 32 samples), and for a threshold T
// every register yields its four comparisons v > T as the high bits of its
// bytes by byte-wise SWAR arithmetic (no carry crosses a byte):
//   T < 127:  v > T  <=>  v >= 128 or (v & 127) + (127 - T) >= 128
//   T >= 127: v > T  <=>  v >= 128 and (v & 127) + (255 - T) >= 128
// and register r's high bits, moved right by 7 - r, put sample r + 8j at bit
// r + 8j of the word.  The move is a multiply-high by 2^(25 + r), which runs
// on the FMA pipe and leaves the logic pipe to the comparisons.  Per 128
// input bytes: 8 global loads, 8 shared stores, 8 shared loads.

constexpr int kPackWords = 32;             // words per tile (1024 samples)
constexpr int kPackTS = kPackWords * 32;   // samples per tile
constexpr int kPackTF = 32;                // features per tile
constexpr int kPackQuads = kPackTF / 4;    // feature quads per tile
constexpr int kPackWarps = 8;              // warp w: feature quad w
static_assert(kPackWarps * 32 == kPackWords * 8, "fill: 8 threads per word");
static_assert(kPackWarps == kPackQuads, "compare: one feature quad per warp");

__device__ __forceinline__ int pack_cell(int q, int r) { return 8 * q + (r ^ (q & 7)); }

__global__ void __launch_bounds__(kPackWarps * 32)
pack_bits_kernel(const uint8_t* __restrict__ x, long long N, int d, Thresholds th,
                 uint32_t* __restrict__ xp, long long W, bool vec16) {
    __shared__ __align__(16) uint4 tile[kPackQuads][kPackWords * 8];   // [quad][swizzled group]
    __shared__ uint32_t sC[32], sOr[32];   // per-threshold SWAR constants
    if (threadIdx.x < th.b) {
        const uint32_t T = threshold_at(th, threadIdx.x);
        // T == 255: nothing exceeds it (C = 0, AND form: the sum never reaches 128)
        sC[threadIdx.x] = (T < 127u ? 127u - T : 255u - T) * 0x01010101u;
        sOr[threadIdx.x] = T < 127u ? 0x80808080u : 0u;
    }
    const long long s0 = (long long)blockIdx.y * kPackTS;
    const int f0 = blockIdx.x * kPackTF;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int nf = min(kPackTF, d - f0);
    {
        const int wq = threadIdx.x >> 3, r = threadIdx.x & 7;
        uint32_t v[4][8];   // [sample j][feature quad]
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const long long s = s0 + 32 * wq + r + 8 * j;
#pragma unroll
            for (int f4 = 0; f4 < 8; ++f4) v[j][f4] = 0u;
            if (s < N) {
                const uint8_t* p = x + s * d + f0;
                if (vec16 && nf == kPackTF) {
                    const uint4 a = __ldg(reinterpret_cast<const uint4*>(p));
                    const uint4 b = __ldg(reinterpret_cast<const uint4*>(p) + 1);
                    v[j][0] = a.x; v[j][1] = a.y; v[j][2] = a.z; v[j][3] = a.w;
                    v[j][4] = b.x; v[j][5] = b.y; v[j][6] = b.z; v[j][7] = b.w;
                } else {
#pragma unroll
                    for (int f = 0; f < kPackTF; ++f)
                        if (f < nf) v[j][f >> 2] |= (uint32_t)__ldg(p + f) << (8 * (f & 3));
                }
            }
        }
        const int cell = pack_cell(wq, r);
#pragma unroll
        for (int f4 = 0; f4 < 8; ++f4) {
            // bytes (s0 f0, s1 f0, s0 f1, s1 f1) and (s0 f2, s1 f2, s0 f3, s1 f3), likewise s2/s3
            const uint32_t a0 = __byte_perm(v[0][f4], v[1][f4], 0x5140);
            const uint32_t a1 = __byte_perm(v[0][f4], v[1][f4], 0x7362);
            const uint32_t b0 = __byte_perm(v[2][f4], v[3][f4], 0x5140);
            const uint32_t b1 = __byte_perm(v[2][f4], v[3][f4], 0x7362);
            tile[f4][cell] = make_uint4(__byte_perm(a0, b0, 0x5410), __byte_perm(a0, b0, 0x7632),
                                        __byte_perm(a1, b1, 0x5410), __byte_perm(a1, b1, 0x7632));
        }
    }
    __syncthreads();
    const long long q = (long long)blockIdx.y * kPackWords + lane;   // this lane's word
    if (q >= W) return;
    const int fq = warp;   // this warp's feature quad: features 4 fq .. 4 fq + 3
    if (4 * fq >= nf) return;
    uint32_t reg[4][8];    // [feature in quad][sample group r]
#pragma unroll
    for (int r = 0; r < 8; ++r) {
        const uint4 c = tile[fq][pack_cell(lane, r)];
        reg[0][r] = c.x; reg[1][r] = c.y; reg[2][r] = c.z; reg[3][r] = c.w;
    }
#pragma unroll
    for (int fi = 0; fi < 4; ++fi) {
        if (4 * fq + fi >= nf) break;
        uint32_t lo7[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) lo7[i] = reg[fi][i] & 0x7f7f7f7fu;
        uint32_t* out = xp + (long long)(f0 + 4 * fq + fi) * th.b * W + q;
        for (int i = 0; i < th.b; ++i) {
            const uint32_t C = sC[i];
            uint32_t word = 0u;
            if (sOr[i]) {   // T < 127: OR form (warp-uniform branch)
#pragma unroll
                for (int i8 = 0; i8 < 8; ++i8) {
                    const uint32_t hb = (reg[fi][i8] | (lo7[i8] + C)) & 0x80808080u;
                    word += i8 < 7 ? __umulhi(hb, 1u << ((25 + i8) & 31)) : hb;   // disjoint bits
                }
            } else {        // T >= 127: AND form
#pragma unroll
                for (int i8 = 0; i8 < 8; ++i8) {
                    const uint32_t hb = (reg[fi][i8] & (lo7[i8] + C)) & 0x80808080u;
                    word += i8 < 7 ? __umulhi(hb, 1u << ((25 + i8) & 31)) : hb;
                }
            }
            out[(long long)i * W] = word;
        }
    }
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(encode)

namespace {
template <typename OutT>
int encode_impl(const uint8_t* x, int64_t B, int32_t d, const uint8_t* thr_host, int32_t b, OutT* bits,
                uint8_t* bits8, cudaStream_t stream) {
    Thresholds th;
    int st = make_thresholds(thr_host, b, &th);
    if (st) return st;
    if (B < 0 || d <= 0) return BITLOGIC_ERR_SHAPE;
    if (B == 0) return BITLOGIC_OK;   // an empty batch may come as NULL
    if (!x || !bits) return BITLOGIC_ERR_NULL;
    if (B % 4 == 0 && aligned16(bits) && (!bits8 || aligned16(bits8))) {
        const long long gy = (B + kEncVS - 1) / kEncVS;
        if (gy > 65535) return BITLOGIC_ERR_SHAPE;
        const bool vec16 = (d % 16 == 0) && aligned16(x);
        dim3 grid((unsigned)((d + kEncTF - 1) / kEncTF), (unsigned)gy);
        encode_soft_vec_kernel<OutT><<<grid, 256, 0, stream>>>(x, B, d, th, bits, bits8, vec16);
        return launch_status();
    }
    const long long gy = (B + kEncTS - 1) / kEncTS;
    if (gy > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((d + kEncTF - 1) / kEncTF), (unsigned)gy);
    encode_soft_kernel<OutT><<<grid, 256, 0, stream>>>(x, B, d, th, bits, bits8);
    return launch_status();
}
}  // namespace

extern "C" int bitlogic_encode_thermometer(const uint8_t* x, int64_t B, int32_t d,
                                           const uint8_t* thr_host, int32_t b,
                                           float* bits, cudaStream_t stream) {
    return encode_impl(x, B, d, thr_host, b, bits, nullptr, stream);
}

extern "C" int bitlogic_encode_thermometer_u8(const uint8_t* x, int64_t B, int32_t d,
                                              const uint8_t* thr_host, int32_t b,
                                              uint8_t* bits, cudaStream_t stream) {
    return encode_impl(x, B, d, thr_host, b, bits, nullptr, stream);
}

extern "C" int bitlogic_encode_thermometer_both(const uint8_t* x, int64_t B, int32_t d,
                                                const uint8_t* thr_host, int32_t b,
                                                float* bits, uint8_t* bits8, cudaStream_t stream) {
    if (B > 0 && !bits8) return BITLOGIC_ERR_NULL;
    return encode_impl(x, B, d, thr_host, b, bits, bits8, stream);
}

extern "C" int bitlogic_encode_thermometer_bitrows(const uint8_t* x, int64_t B, int32_t d,
                                                   const uint8_t* thr_host, int32_t b,
                                                   uint32_t* bits, cudaStream_t stream) {
    Thresholds th;
    int st = make_thresholds(thr_host, b, &th);
    if (st) return st;
    if (B < 0 || d <= 0) return BITLOGIC_ERR_SHAPE;
    if (B == 0) return BITLOGIC_OK;   // an empty batch may come as NULL
    if (!x || !bits) return BITLOGIC_ERR_NULL;
    const long long nblk = (B + kBitBlock - 1) / kBitBlock;
    if (nblk > 65535) return BITLOGIC_ERR_SHAPE;
    const bool vec8 = (d % 8 == 0) && (reinterpret_cast<uintptr_t>(x) & 7u) == 0;
    dim3 grid((unsigned)((d + kBitsTF - 1) / kBitsTF), (unsigned)nblk);
    encode_bitrows_kernel<<<grid, 256, 0, stream>>>(x, B, d, th, bits, nblk * 32, vec8);
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
    const bool vec16 = (d % 16 == 0) && aligned16(x);
    dim3 grid((unsigned)((d + kPackTF - 1) / kPackTF), (unsigned)gy);
    pack_bits_kernel<<<grid, kPackWarps * 32, 0, stream>>>(x, N, d, th, xp, W, vec16);
    return launch_status();
}
