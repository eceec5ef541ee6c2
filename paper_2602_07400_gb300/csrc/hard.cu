// Hard (inference) mode on bit-packed activations (paper App. C.1
// "Bit-packed inference": tables discretized once per layer, samples packed
// along the batch into words, each layer's LUT evaluation a bitwise op on
// the packed tensors; here 32 samples per uint32).
//
// A node's output word is a bit-sliced Shannon expansion of its table over
// its k input words: level 0 selects between the two table bits of each pair
// with x_0 (as all-zero / all-one masks), level l muxes the level-(l-1)
// results with x_l, each mux one LOP3 (x & hi) | (~x & lo); 2^k - 1 per node
// and word.  The popcount GroupSum head (§3) is fused into the last layer:
// every lane keeps carry-save (Harley-Seal) bit-sliced counters over its
// group's nodes, so the last layer's packed outputs never reach memory.
#include "common.cuh"

namespace bitlogic {
namespace {

// ------------------------------------------------------------ binarize --

__global__ void __launch_bounds__(256)
binarize_kernel(const float* __restrict__ theta, int w, int k, uint64_t* __restrict__ table) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * 8 + warp;
    if (j >= w) return;
    const int K = 1 << k;
    const float* t = theta + (long long)j * K;
    const bool b0 = lane < K && __ldg(t + lane) > 0.0f;
    const bool b1 = lane + 32 < K && __ldg(t + lane + 32) > 0.0f;
    const uint32_t lo = __ballot_sync(0xffffffffu, b0);
    const uint32_t hi = __ballot_sync(0xffffffffu, b1);
    if (lane == 0) table[j] = (uint64_t)lo | ((uint64_t)hi << 32);
}

// ------------------------------------------------------------ mux tree --

// Level 0 selects between the two table bits of each pair with x_0.  With
// table bits (t0, t1) of pair m the bit-sliced x_0 ? t1 : t0 is one of
// 0, ~0, x_0, ~x_0, which in 32-bit arithmetic is x_0 * p + q with
// (p, q) = (t1 - t0, -t0): (0,0) -> 0, (1,1) -> -1, (0,1) -> x_0,
// (1,0) -> -x_0 - 1 = ~x_0.  So level 0 runs as integer multiply-adds on the
// FMA pipe, and only the 2^(k-1) - 1 upper muxes are logic ops.
template <int L, int M, int H, int k>
__device__ __forceinline__ uint32_t mux_tree(const int (&p)[H], const int (&q)[H],
                                             const uint32_t (&x)[k]) {
    if constexpr (L == 0) {
        return (uint32_t)((int)x[0] * p[M] + q[M]);
    } else {
        const uint32_t a = mux_tree<L - 1, 2 * M>(p, q, x);
        const uint32_t b = mux_tree<L - 1, 2 * M + 1>(p, q, x);
        return (x[L] & b) | (~x[L] & a);
    }
}

// Per-warp node set-up: lane m derives (p, q) of pair m from the table, the
// warp shares them through shared memory.
template <int k>
__device__ __forceinline__ void node_pairs(uint64_t T, int lane, int2* sPQ,
                                           int (&p)[1 << (k - 1)], int (&q)[1 << (k - 1)]) {
    constexpr int H = 1 << (k - 1);
    if (lane < H) {
        const int t0 = (int)((T >> (2 * lane)) & 1u), t1 = (int)((T >> (2 * lane + 1)) & 1u);
        sPQ[lane] = make_int2(t1 - t0, -t0);
    }
    __syncwarp();
#pragma unroll
    for (int m = 0; m < H; m += 2) {
        if constexpr (H >= 2) {
            const int4 v = *reinterpret_cast<const int4*>(sPQ + m);
            p[m] = v.x; q[m] = v.y; p[m + 1] = v.z; q[m + 1] = v.w;
        } else {
            const int2 v = sPQ[m];
            p[m] = v.x; q[m] = v.y;
        }
    }
    __syncwarp();
}

template <int k>
__device__ __forceinline__ void node_rows(const int* __restrict__ conn, int j, int w_in,
                                          int lane, int (&rows)[k]) {
    bool bad = false;
#pragma unroll
    for (int i = 0; i < k; ++i) {
        int c = __ldg(conn + (long long)j * k + i);
        if ((unsigned)c >= (unsigned)w_in) { bad = true; c = 0; }
        rows[i] = c;
    }
    if (bad && lane == 0) flag_index_error();
}

template <int R>
struct Words;
template <> struct Words<1> { using T = uint32_t; };
template <> struct Words<2> { using T = uint2; };
template <> struct Words<4> { using T = uint4; };

template <int R>
__device__ __forceinline__ void load_words(const uint32_t* p, uint32_t (&o)[R]) {
    if constexpr (R == 1) {
        o[0] = __ldg(p);
    } else if constexpr (R == 2) {
        const uint2 v = __ldg(reinterpret_cast<const uint2*>(p));
        o[0] = v.x; o[1] = v.y;
    } else {
        const uint4 v = __ldg(reinterpret_cast<const uint4*>(p));
        o[0] = v.x; o[1] = v.y; o[2] = v.z; o[3] = v.w;
    }
}

template <int R>
__device__ __forceinline__ void store_words(uint32_t* p, const uint32_t (&o)[R]) {
    if constexpr (R == 1) *p = o[0];
    else if constexpr (R == 2) *reinterpret_cast<uint2*>(p) = make_uint2(o[0], o[1]);
    else *reinterpret_cast<uint4*>(p) = make_uint4(o[0], o[1], o[2], o[3]);
}

// ------------------------------------------------- layer without head --

constexpr int kHardWarps = 8;

// One warp per node, each lane R consecutive words (R = 4: 16-byte loads
// and stores, four independent trees); the block's y index selects a range
// of words so that the gathered rows of the resident blocks stay in L2.
template <int k, int R>
__global__ void __launch_bounds__(kHardWarps * 32)
hard_layer_kernel(const uint32_t* __restrict__ xp, int w_in, long long W,
                  const int* __restrict__ conn, const uint64_t* __restrict__ table, int w,
                  uint32_t* __restrict__ yp, long long wchunk, uint32_t tail_mask) {
    constexpr int H = 1 << (k - 1);
    __shared__ __align__(16) int2 sPQ[kHardWarps][H < 2 ? 2 : H];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kHardWarps + warp;
    if (j >= w) return;
    int rows[k];
    node_rows<k>(conn, j, w_in, lane, rows);
    int p[H], q[H];
    node_pairs<k>(__ldg(table + j), lane, sPQ[warp], p, q);
    const long long q0 = (long long)blockIdx.y * wchunk;
    const long long q1 = min(W, q0 + wchunk);
    uint32_t* out = yp + (long long)j * W;
    for (long long w0 = q0 + (long long)R * lane; w0 < q1; w0 += 32 * R) {
        uint32_t x[R][k];
#pragma unroll
        for (int i = 0; i < k; ++i) {
            uint32_t v[R];
            load_words<R>(xp + (long long)rows[i] * W + w0, v);
#pragma unroll
            for (int r = 0; r < R; ++r) x[r][i] = v[r];
        }
        uint32_t y[R];
#pragma unroll
        for (int r = 0; r < R; ++r) {
            y[r] = mux_tree<k - 1, 0>(p, q, x[r]);
            if (w0 + r == W - 1) y[r] &= tail_mask;
        }
        store_words<R>(out + w0, y);
    }
}

// ------------------------------------------------- layer + popcount head --

// Carry-save adder on bit-sliced words: (a + b + c) = 2*carry + sum.
__device__ __forceinline__ void csa(uint32_t& carry, uint32_t& sum, uint32_t a, uint32_t b,
                                    uint32_t c) {
    const uint32_t u = a ^ b;
    carry = (a & b) | (u & c);
    sum = u ^ c;
}

constexpr int kHeadWarps = 8;
constexpr int kBigPlanes = 10;   // weight-8 planes: up to 8 * 1023 + 7 nodes per warp
constexpr int kHeadR = 2;        // words per lane in the head kernel

// grid.x: groups of 32 * kHeadR words, grid.y: class c x split.  Lane l
// covers words kHeadR * l .. kHeadR * l + kHeadR - 1 of the group.  Warp r of
// a block takes nodes n0 + r, n0 + r + 8, ... of its slice and feeds their
// output words, eight nodes at a time, through a Harley-Seal carry-save tree
// into per-lane bit-sliced counters.  At the end every lane turns its
// counters into per-sample counts, the block adds its 8 warps in shared
// memory and one integer atomicAdd per (sample, class) publishes the block's
// total (exact and order-independent).
template <int k, int R>
__global__ void __launch_bounds__(kHeadWarps * 32, 2)
hard_head_kernel(const uint32_t* __restrict__ xp, int w_in, long long W, long long N,
                 const int* __restrict__ conn, const uint64_t* __restrict__ table,
                 int C, int g, int splits, int per_split, uint32_t* __restrict__ yp,
                 int* __restrict__ counts, uint32_t tail_mask) {
    constexpr int H = 1 << (k - 1);
    __shared__ int sCount[32 * R * 32];   // [word in block][bit]
    __shared__ __align__(16) int2 sPQ[kHeadWarps][H < 2 ? 2 : H];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.y / splits, sp = blockIdx.y - c * splits;
    const int n0 = c * g + sp * per_split;
    const int n1 = min(c * g + g, n0 + per_split);
    const long long w0 = (long long)blockIdx.x * (32 * R) + (long long)R * lane;   // first word
    const bool active = w0 < W;   // W % R == 0 on this path, so all R words are in range
    for (int t = threadIdx.x; t < 32 * R * 32; t += kHeadWarps * 32) sCount[t] = 0;

    uint32_t ones[R], twos[R], fours[R], big[R][kBigPlanes];
#pragma unroll
    for (int r = 0; r < R; ++r) {
        ones[r] = twos[r] = fours[r] = 0;
#pragma unroll
        for (int b = 0; b < kBigPlanes; ++b) big[r][b] = 0;
    }

    int j = n0 + warp;
    while (j < n1) {
        uint32_t y[8][R];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
#pragma unroll
            for (int r = 0; r < R; ++r) y[u][r] = 0;
            if (j < n1) {
                int rows[k];
                node_rows<k>(conn, j, w_in, lane, rows);
                int p[H], q[H];
                node_pairs<k>(__ldg(table + j), lane, sPQ[warp], p, q);
                if (active) {
                    uint32_t x[R][k];
#pragma unroll
                    for (int i = 0; i < k; ++i) {
                        uint32_t v[R];
                        load_words<R>(xp + (long long)rows[i] * W + w0, v);
#pragma unroll
                        for (int r = 0; r < R; ++r) x[r][i] = v[r];
                    }
#pragma unroll
                    for (int r = 0; r < R; ++r) {
                        uint32_t v = mux_tree<k - 1, 0>(p, q, x[r]);
                        if (w0 + r == W - 1) v &= tail_mask;
                        y[u][r] = v;
                    }
                    if (yp) store_words<R>(yp + (long long)j * W + w0, y[u]);
                }
            }
            j += kHeadWarps;
        }
#pragma unroll
        for (int r = 0; r < R; ++r) {
            uint32_t tA, tB, fA, fB, e;
            csa(tA, ones[r], ones[r], y[0][r], y[1][r]);
            csa(tB, ones[r], ones[r], y[2][r], y[3][r]);
            csa(fA, twos[r], twos[r], tA, tB);
            csa(tA, ones[r], ones[r], y[4][r], y[5][r]);
            csa(tB, ones[r], ones[r], y[6][r], y[7][r]);
            csa(fB, twos[r], twos[r], tA, tB);
            csa(e, fours[r], fours[r], fA, fB);
#pragma unroll
            for (int b = 0; b < kBigPlanes; ++b) {   // ripple-add the weight-8 word
                const uint32_t cy = big[r][b] & e;
                big[r][b] ^= e;
                e = cy;
            }
        }
    }
    __syncthreads();
    if (active) {
#pragma unroll
        for (int r = 0; r < R; ++r) {
            for (int bit = 0; bit < 32; ++bit) {
                int cnt = (int)((ones[r] >> bit) & 1u) + 2 * (int)((twos[r] >> bit) & 1u) +
                          4 * (int)((fours[r] >> bit) & 1u);
#pragma unroll
                for (int b = 0; b < kBigPlanes; ++b) cnt += (int)((big[r][b] >> bit) & 1u) << (b + 3);
                if (cnt) atomicAdd(&sCount[(R * lane + r) * 32 + bit], cnt);
            }
        }
    }
    __syncthreads();
    for (int t = threadIdx.x; t < 32 * R * 32; t += kHeadWarps * 32) {
        const long long s = (long long)blockIdx.x * (32 * R * 32) + t;
        if (s < N && sCount[t]) atomicAdd(counts + s * C + c, sCount[t]);
    }
}

__global__ void __launch_bounds__(256)
argmax_kernel(const int* __restrict__ counts, long long N, int C, int* __restrict__ pred) {
    const long long s = (long long)blockIdx.x * 256 + threadIdx.x;
    if (s >= N) return;
    const int* row = counts + s * C;
    int best = row[0], bc = 0;
    for (int c = 1; c < C; ++c) {
        const int v = row[c];
        if (v > best) { best = v; bc = c; }
    }
    pred[s] = bc;
}

// Words per block of the headless layer: enough that the node set-up is
// amortised, small enough that the gathered input slice stays in L2.
long long hard_word_chunk(int w_in, long long W) {
    const long long l2_budget = 48ll << 20;
    if ((long long)w_in * W * 4 <= l2_budget) return W;
    long long c = l2_budget / ((long long)w_in * 4);
    c = (c / 128) * 128;
    if (c < 512) c = 512;
    return c < W ? c : W;
}

template <int k>
int launch_hard(const uint32_t* xp, int w_in, long long N, const int* conn, const uint64_t* table,
                int w, uint32_t* yp, int C, int* counts, int* pred, cudaStream_t st) {
    const long long W = (N + 31) / 32;
    const uint32_t tail_mask = (N % 32) ? ((1u << (N % 32)) - 1u) : 0xffffffffu;
    if (C == 0) {
        const bool vec = (W % 4 == 0) && aligned16(xp) && aligned16(yp);
        const long long chunk = hard_word_chunk(w_in, W);
        const long long ny = (W + chunk - 1) / chunk;
        if (ny > 65535) return BITLOGIC_ERR_SHAPE;
        dim3 grid((unsigned)((w + kHardWarps - 1) / kHardWarps), (unsigned)ny);
        if (vec)
            hard_layer_kernel<k, 4><<<grid, kHardWarps * 32, 0, st>>>(xp, w_in, W, conn, table, w, yp, chunk, tail_mask);
        else
            hard_layer_kernel<k, 1><<<grid, kHardWarps * 32, 0, st>>>(xp, w_in, W, conn, table, w, yp, chunk, tail_mask);
        return launch_status();
    }
    const int g = w / C;
    const bool vec = (W % kHeadR == 0) && ((reinterpret_cast<uintptr_t>(xp) & 7u) == 0) &&
                     (!yp || (reinterpret_cast<uintptr_t>(yp) & 7u) == 0);
    const int R = vec ? kHeadR : 1;
    const long long wg = (W + 32 * R - 1) / (32 * R);
    // split a class over several blocks when there are few word groups, so
    // that at least ~4 blocks per SM are in flight
    int splits = 1;
    while (wg * C * splits < 608 && g / (splits * 2) >= 64) splits *= 2;
    int per_split = (g + splits - 1) / splits;
    // each warp's slice must fit the counters
    while ((per_split + kHeadWarps - 1) / kHeadWarps > 8 * ((1 << kBigPlanes) - 1)) {
        splits *= 2;
        per_split = (g + splits - 1) / splits;
    }
    if ((long long)C * splits > 65535) return BITLOGIC_ERR_SHAPE;
    if (cudaMemsetAsync(counts, 0, sizeof(int) * (size_t)N * (size_t)C, st) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    dim3 grid((unsigned)wg, (unsigned)(C * splits));
    if (vec)
        hard_head_kernel<k, kHeadR><<<grid, kHeadWarps * 32, 0, st>>>(xp, w_in, W, N, conn, table, C, g, splits,
                                                                      per_split, yp, counts, tail_mask);
    else
        hard_head_kernel<k, 1><<<grid, kHeadWarps * 32, 0, st>>>(xp, w_in, W, N, conn, table, C, g, splits,
                                                                 per_split, yp, counts, tail_mask);
    if (pred) argmax_kernel<<<(unsigned)((N + 255) / 256), 256, 0, st>>>(counts, N, C, pred);
    return launch_status();
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(hard)

extern "C" int bitlogic_binarize_tables(const float* theta, int32_t w, int32_t k,
                                        uint64_t* table, cudaStream_t stream) {
    if (!theta || !table) return BITLOGIC_ERR_NULL;
    if (w <= 0) return BITLOGIC_ERR_SHAPE;
    if (k < 1 || k > 6) return BITLOGIC_ERR_FANIN;
    binarize_kernel<<<(unsigned)((w + 7) / 8), 256, 0, stream>>>(theta, w, k, table);
    return launch_status();
}

extern "C" int bitlogic_hard_forward(const uint32_t* xp, int32_t w_in, int64_t N,
                                     const int32_t* conn, const uint64_t* table,
                                     int32_t w, int32_t k, uint32_t* yp,
                                     int32_t C, int32_t* counts, int32_t* pred,
                                     cudaStream_t stream) {
    if (!conn || !table) return BITLOGIC_ERR_NULL;
    if (w_in <= 0 || w <= 0 || N < 0 || C < 0) return BITLOGIC_ERR_SHAPE;
    if (k < 1 || k > 6 || k > w_in) return BITLOGIC_ERR_FANIN;
    if (C > 0 && w % C != 0) return BITLOGIC_ERR_SHAPE;
    if (N == 0) return BITLOGIC_OK;   // an empty batch may come as NULL
    if (!xp) return BITLOGIC_ERR_NULL;
    if (C == 0 && !yp) return BITLOGIC_ERR_NULL;
    if (C > 0 && !counts) return BITLOGIC_ERR_NULL;
    if ((N + 31) / 32 > (1ll << 40)) return BITLOGIC_ERR_SHAPE;
    switch (k) {
        case 1: return launch_hard<1>(xp, w_in, N, conn, table, w, yp, C, counts, pred, stream);
        case 2: return launch_hard<2>(xp, w_in, N, conn, table, w, yp, C, counts, pred, stream);
        case 3: return launch_hard<3>(xp, w_in, N, conn, table, w, yp, C, counts, pred, stream);
        case 4: return launch_hard<4>(xp, w_in, N, conn, table, w, yp, C, counts, pred, stream);
        case 5: return launch_hard<5>(xp, w_in, N, conn, table, w, yp, C, counts, pred, stream);
        default: return launch_hard<6>(xp, w_in, N, conn, table, w, yp, C, counts, pred, stream);
    }
}
