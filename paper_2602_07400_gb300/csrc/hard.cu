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

template <int L, int M, int H, int k>
__device__ __forceinline__ uint32_t mux_tree(const uint32_t (&lo)[H], const uint32_t (&hi)[H],
                                             const uint32_t (&x)[k]) {
    if constexpr (L == 0) {
        return (x[0] & hi[M]) | (~x[0] & lo[M]);
    } else {
        const uint32_t a = mux_tree<L - 1, 2 * M>(lo, hi, x);
        const uint32_t b = mux_tree<L - 1, 2 * M + 1>(lo, hi, x);
        return (x[L] & b) | (~x[L] & a);
    }
}

// Table bits of node j as level-0 masks: lo[m] = -(bit 2m), hi[m] = -(bit 2m+1).
template <int k>
__device__ __forceinline__ void table_masks(uint64_t T, uint32_t (&lo)[1 << (k - 1)],
                                            uint32_t (&hi)[1 << (k - 1)]) {
    const uint32_t tl = (uint32_t)T, th = (uint32_t)(T >> 32);
#pragma unroll
    for (int m = 0; m < (1 << (k - 1)); ++m) {
        const int b0 = 2 * m, b1 = 2 * m + 1;
        const uint32_t w0 = b0 < 32 ? tl : th, w1 = b1 < 32 ? tl : th;
        lo[m] = (uint32_t)((int32_t)(w0 << (31 - (b0 & 31))) >> 31);
        hi[m] = (uint32_t)((int32_t)(w1 << (31 - (b1 & 31))) >> 31);
    }
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

// ------------------------------------------------- layer without head --

constexpr int kHardWarps = 8;

// One warp per node, lanes over words; the block's y index selects a range
// of words so the gathered rows of the resident blocks stay in L2.
template <int k>
__global__ void __launch_bounds__(kHardWarps * 32)
hard_layer_kernel(const uint32_t* __restrict__ xp, int w_in, long long W,
                  const int* __restrict__ conn, const uint64_t* __restrict__ table, int w,
                  uint32_t* __restrict__ yp, long long wchunk, uint32_t tail_mask) {
    constexpr int H = 1 << (k - 1);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kHardWarps + warp;
    if (j >= w) return;
    int rows[k];
    node_rows<k>(conn, j, w_in, lane, rows);
    uint32_t lo[H], hi[H];
    table_masks<k>(__ldg(table + j), lo, hi);
    const long long q0 = (long long)blockIdx.y * wchunk;
    const long long q1 = min(W, q0 + wchunk);
    uint32_t* out = yp + (long long)j * W;
    for (long long q = q0 + lane; q < q1; q += 32) {
        uint32_t x[k];
#pragma unroll
        for (int i = 0; i < k; ++i) x[i] = __ldg(xp + (long long)rows[i] * W + q);
        uint32_t y = mux_tree<k - 1, 0>(lo, hi, x);
        if (q == W - 1) y &= tail_mask;
        out[q] = y;
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

// grid.x: groups of 32 words (lane = word), grid.y: class c x split.
// Warp r of a block takes nodes n0 + r, n0 + r + 8, ... of its slice and
// feeds their output words, eight at a time, through a Harley-Seal
// carry-save tree into per-lane bit-sliced counters.  At the end every lane
// turns its counters into 32 per-sample counts, the block adds its 8 warps in
// shared memory and one integer atomicAdd per (sample, class) publishes the
// block's total (exact and order-independent).
template <int k>
__global__ void __launch_bounds__(kHeadWarps * 32)
hard_head_kernel(const uint32_t* __restrict__ xp, int w_in, long long W, long long N,
                 const int* __restrict__ conn, const uint64_t* __restrict__ table,
                 int C, int g, int splits, int per_split, uint32_t* __restrict__ yp,
                 int* __restrict__ counts, uint32_t tail_mask) {
    constexpr int H = 1 << (k - 1);
    __shared__ int sCount[32 * 32];   // [word in block][bit]
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.y / splits, sp = blockIdx.y - c * splits;
    const int n0 = c * g + sp * per_split;
    const int n1 = min(c * g + g, n0 + per_split);
    const long long q = (long long)blockIdx.x * 32 + lane;
    const bool active = q < W;
    for (int t = threadIdx.x; t < 32 * 32; t += kHeadWarps * 32) sCount[t] = 0;

    uint32_t ones = 0, twos = 0, fours = 0;
    uint32_t big[kBigPlanes];
#pragma unroll
    for (int p = 0; p < kBigPlanes; ++p) big[p] = 0;

    int j = n0 + warp;
    while (j < n1) {
        uint32_t y[8];
#pragma unroll
        for (int u = 0; u < 8; ++u) {
            y[u] = 0;
            if (j < n1) {
                int rows[k];
                node_rows<k>(conn, j, w_in, lane, rows);
                uint32_t lo[H], hi[H];
                table_masks<k>(__ldg(table + j), lo, hi);
                if (active) {
                    uint32_t x[k];
#pragma unroll
                    for (int i = 0; i < k; ++i) x[i] = __ldg(xp + (long long)rows[i] * W + q);
                    uint32_t v = mux_tree<k - 1, 0>(lo, hi, x);
                    if (q == W - 1) v &= tail_mask;
                    if (yp) yp[(long long)j * W + q] = v;
                    y[u] = v;
                }
            }
            j += kHeadWarps;
        }
        uint32_t tA, tB, fA, fB, e;
        csa(tA, ones, ones, y[0], y[1]);
        csa(tB, ones, ones, y[2], y[3]);
        csa(fA, twos, twos, tA, tB);
        csa(tA, ones, ones, y[4], y[5]);
        csa(tB, ones, ones, y[6], y[7]);
        csa(fB, twos, twos, tA, tB);
        csa(e, fours, fours, fA, fB);
#pragma unroll
        for (int p = 0; p < kBigPlanes; ++p) {   // ripple-add the weight-8 word
            const uint32_t cy = big[p] & e;
            big[p] ^= e;
            e = cy;
        }
    }
    __syncthreads();
    if (active) {
        for (int bit = 0; bit < 32; ++bit) {
            int cnt = (int)((ones >> bit) & 1u) + 2 * (int)((twos >> bit) & 1u) +
                      4 * (int)((fours >> bit) & 1u);
#pragma unroll
            for (int p = 0; p < kBigPlanes; ++p) cnt += (int)((big[p] >> bit) & 1u) << (p + 3);
            if (cnt) atomicAdd(&sCount[lane * 32 + bit], cnt);
        }
    }
    __syncthreads();
    for (int t = threadIdx.x; t < 32 * 32; t += kHeadWarps * 32) {
        const long long s = (long long)blockIdx.x * 1024 + t;
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

// Words per block of the headless layer: enough that the mask set-up is
// amortised, small enough that the gathered input slice stays in L2.
long long hard_word_chunk(int w_in, long long W) {
    const long long l2_budget = 48ll << 20;
    if ((long long)w_in * W * 4 <= l2_budget) return W;
    long long c = l2_budget / ((long long)w_in * 4);
    c = (c / 32) * 32;
    if (c < 256) c = 256;
    return c < W ? c : W;
}

template <int k>
int launch_hard(const uint32_t* xp, int w_in, long long N, const int* conn, const uint64_t* table,
                int w, uint32_t* yp, int C, int* counts, int* pred, cudaStream_t st) {
    const long long W = (N + 31) / 32;
    const uint32_t tail_mask = (N % 32) ? ((1u << (N % 32)) - 1u) : 0xffffffffu;
    if (C == 0) {
        const long long chunk = hard_word_chunk(w_in, W);
        const long long ny = (W + chunk - 1) / chunk;
        if (ny > 65535) return BITLOGIC_ERR_SHAPE;
        dim3 grid((unsigned)((w + kHardWarps - 1) / kHardWarps), (unsigned)ny);
        hard_layer_kernel<k><<<grid, kHardWarps * 32, 0, st>>>(xp, w_in, W, conn, table, w, yp, chunk, tail_mask);
        return launch_status();
    }
    const int g = w / C;
    const long long wg = (W + 31) / 32;
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
    hard_head_kernel<k><<<grid, kHeadWarps * 32, 0, st>>>(xp, w_in, W, N, conn, table, C, g, splits,
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
