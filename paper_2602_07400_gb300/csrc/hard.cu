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
        return x[0] * (uint32_t)p[M] + (uint32_t)q[M];   // modulo 2^32
    } else {
        const uint32_t a = mux_tree<L - 1, 2 * M>(p, q, x);
        const uint32_t b = mux_tree<L - 1, 2 * M + 1>(p, q, x);
        return (x[L] & b) | (~x[L] & a);
    }
}

// The tree for four words at once with the level-0 pairs read from shared
// memory (broadcast loads) instead of registers: depth first, so at most one
// partial result per level and word is live.
template <int L, int M, int k>
__device__ __forceinline__ void mux_tree4_smem(const int2* __restrict__ sPQ, const uint32_t (&x)[4][k],
                                               uint32_t (&out)[4]) {
    if constexpr (L == 0) {
        const int2 v = sPQ[M];
#pragma unroll
        for (int r = 0; r < 4; ++r) out[r] = x[r][0] * (uint32_t)v.x + (uint32_t)v.y;
    } else {
        uint32_t lo[4], hi[4];
        mux_tree4_smem<L - 1, 2 * M, k>(sPQ, x, lo);
        mux_tree4_smem<L - 1, 2 * M + 1, k>(sPQ, x, hi);
#pragma unroll
        for (int r = 0; r < 4; ++r) out[r] = (x[r][L] & hi[r]) | (~x[r][L] & lo[r]);
    }
}

// Per-warp node set-up: lane m derives (p, q) of pair m from the table, the
// warp shares them through shared memory (sPQ: 2 * 2^(k-1) ints per warp)
// and every lane reads all pairs into registers (two per 16-byte load).
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

// Pair set-up when the tree reads the pairs from shared memory: lane m
// writes pair m; the warp synchronises before the tree reads them.
template <int k>
__device__ __forceinline__ void node_pairs_smem(uint64_t T, int lane, int2* sPQ) {
    constexpr int H = 1 << (k - 1);
    if (lane < H) {
        const int t0 = (int)((T >> (2 * lane)) & 1u), t1 = (int)((T >> (2 * lane + 1)) & 1u);
        sPQ[lane] = make_int2(t1 - t0, -t0);
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

// ------------------------------------------- staged layer (vector path) --
//
// The vector paths (W % 4 == 0, 16-byte aligned rows) stream the gathered
// input words through a per-warp ring of shared-memory stages filled by
// 16-byte cp.async copies; a stage holds the k input rows of one node over
// 128 words.  Lane l copies, and later reads, only words 4l .. 4l + 3 of each
// row, so the ring is lane-private: a lane waits for its own copies
// (cp.async.wait_group) and no warp synchronisation guards the ring.  The
// ring runs across node boundaries, so the copies of the next node are in
// flight while the current node is evaluated, and the connectivity row and
// table of the next node are loaded one node ahead.

constexpr int kStageWords = 128;  // words per stage (4 per lane)

template <int k>
__device__ __forceinline__ void read_stage(const uint4* slot, uint32_t (&x)[4][k]) {
#pragma unroll
    for (int i = 0; i < k; ++i) {
        const uint4 v = slot[i * 32];
        x[0][i] = v.x; x[1][i] = v.y; x[2][i] = v.z; x[3][i] = v.w;
    }
}

template <int k>
__host__ __device__ constexpr int ring_bytes_per_warp(int stages) { return stages * k * 32 * 16; }

// A node's k input rows as 32-bit offsets, in 16-byte units from the start
// of the packed input, of the lane's first words: (row * W + wl) / 4.  The
// launchers use the staged kernels only when w_in * W / 4 < 2^32.
template <int k>
__device__ __forceinline__ void node_offsets(const int* __restrict__ conn, int j, int w_in, int lane,
                                             uint32_t W4, uint32_t wl4, uint32_t (&off)[k]) {
    int rows[k];
    node_rows<k>(conn, j, w_in, lane, rows);
#pragma unroll
    for (int i = 0; i < k; ++i) off[i] = (uint32_t)rows[i] * W4 + wl4;
}

// Copies of one stage (the lane's 16 bytes of each of the k rows, `s16`
// 16-byte units past the node's offsets) into a ring slot.
template <int k>
__device__ __forceinline__ void issue_stage(uint4* slot, const uint4* __restrict__ xp4,
                                            const uint32_t (&off)[k], uint32_t s16) {
#pragma unroll
    for (int i = 0; i < k; ++i) cp_async16(slot + i * 32, xp4 + (off[i] + s16));
}

// Three stages per node and warp ring, three blocks per SM: the level-0
// pairs are read from shared memory (80 registers per thread), so 24 warps
// per SM hide the latency of the half-rate logic pipe.
#ifndef BITLOGIC_HARD_NS
#define BITLOGIC_HARD_NS 3
#endif
#ifndef BITLOGIC_HARD_MINB
#define BITLOGIC_HARD_MINB 3
#endif
constexpr int kLayerNS = BITLOGIC_HARD_NS;       // stages per node = ring slots per warp
constexpr int kLayerMinBlocks = BITLOGIC_HARD_MINB;

// Warp w of block b evaluates nodes j = 8b + w, j + jstride, ... (jstride =
// 8 * gridDim.x) over the block's chunk of NS * 128 words (blockIdx.y).  A
// node is exactly NS stages and the warp's ring has NS slots, so stage s of
// every node lives in slot s and all slot offsets are compile-time
// constants: while stage s of node j is evaluated, the copies of stage
// s + NS - 1 (the last stage of node j, or stage s - 1 of the warp's next
// node) are in flight.  FULL: the chunk lies inside the words and holds no
// partial tail word, so no lane checks.
template <int k, int NS, bool FULL>
__device__ __forceinline__ void layer_staged_body(const uint4* __restrict__ xp4, int w_in, long long W,
                                                  const int* __restrict__ conn,
                                                  const uint64_t* __restrict__ table, int w,
                                                  uint32_t* __restrict__ yp, uint32_t tail_mask,
                                                  uint4* ring_smem, int2* sPQ) {
    constexpr int H = 1 << (k - 1);
    constexpr int kSlot = k * 32;   // uint4 per stage
    static_assert(NS >= 2, "at least one stage in flight");
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    uint4* ring = ring_smem + (size_t)warp * (NS * kSlot) + lane;
    const long long wl = (long long)blockIdx.y * (NS * kStageWords) + 4 * lane;   // stage 0 words
    const uint32_t W4 = (uint32_t)(W >> 2), wl4 = (uint32_t)(wl >> 2);
    const int jstride = gridDim.x * kHardWarps;
    int j = blockIdx.x * kHardWarps + warp;

    uint32_t oc[k], on[k];   // row offsets of node j and of node j + jstride
#pragma unroll
    for (int i = 0; i < k; ++i) oc[i] = on[i] = 0;
    if (j < w) node_offsets<k>(conn, j, w_in, lane, W4, wl4, oc);
    if (j + jstride < w) node_offsets<k>(conn, j + jstride, w_in, lane, W4, wl4, on);
    // stage s of a node into slot s (W % 4 == 0: a lane's four words are all
    // in range or all out); one commit group per stage
    auto issue = [&](const uint32_t (&off)[k], int node, int s) {
        bool ok = node < w;
        if constexpr (!FULL) ok = ok && wl + s * kStageWords < W;
        if (ok) issue_stage<k>(ring + s * kSlot, xp4, off, (uint32_t)(s * kStageWords / 4));
        cp_async_commit();
    };
#pragma unroll
    for (int s = 0; s < NS - 1; ++s) issue(oc, j, s);
    uint64_t tab = j < w ? __ldg(table + j) : 0ull;
#pragma unroll 1
    for (; j < w; j += jstride) {
        node_pairs_smem<k>(tab, lane, sPQ);
        const int jn = j + jstride;
        if (jn < w) tab = __ldg(table + jn);
        uint32_t* out = yp + (long long)j * W + wl;
#pragma unroll
        for (int s = 0; s < NS; ++s) {
            if (s == 0) {
                issue(oc, j, NS - 1);
                if (jn + jstride < w) node_offsets<k>(conn, jn + jstride, w_in, lane, W4, wl4, oc);
            } else {
                issue(on, jn, s - 1);
            }
            cp_async_wait<NS - 1>();
            bool ok = true;
            if constexpr (!FULL) ok = wl + s * kStageWords < W;
            if (ok) {
                uint32_t x[4][k];
                read_stage<k>(ring + s * kSlot, x);
                uint32_t y[4];
                mux_tree4_smem<k - 1, 0, k>(sPQ, x, y);
                if constexpr (!FULL) {
                    if (wl + s * kStageWords + 4 == W) y[3] &= tail_mask;   // word W - 1 is y[3]
                }
                store_words<4>(out + s * kStageWords, y);
            }
        }
        __syncwarp();   // the pairs are read before the next node rewrites them
#pragma unroll
        for (int i = 0; i < k; ++i) {
            const uint32_t t = oc[i];
            oc[i] = on[i];
            on[i] = t;
        }
    }
    cp_async_wait<0>();
}

template <int k>
__global__ void __launch_bounds__(kHardWarps * 32, kLayerMinBlocks)
hard_layer_staged_kernel(const uint4* __restrict__ xp4, int w_in, long long W,
                         const int* __restrict__ conn, const uint64_t* __restrict__ table, int w,
                         uint32_t* __restrict__ yp, uint32_t tail_mask) {
    constexpr int H = 1 << (k - 1);
    extern __shared__ uint4 ring_smem[];
    __shared__ __align__(16) int2 sPQ[kHardWarps][H < 2 ? 2 : H];
    const long long end = (long long)(blockIdx.y + 1) * (kLayerNS * kStageWords);
    const bool full = end < W || (end == W && tail_mask == 0xffffffffu);
    int2* mine = sPQ[threadIdx.x >> 5];
    if (full)
        layer_staged_body<k, kLayerNS, true>(xp4, w_in, W, conn, table, w, yp, tail_mask,
                                              ring_smem, mine);
    else
        layer_staged_body<k, kLayerNS, false>(xp4, w_in, W, conn, table, w, yp, tail_mask,
                                                         ring_smem, mine);
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

// Scalar path (any W and alignment).  grid.x: groups of 32 * R words,
// grid.y: class c x split.  Lane l covers words R * l .. R * l + R - 1 of
// the group.  Warp r of
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

// ------------------------------------------- staged head (vector path) --
//
// grid.x: class c x split (fast), grid.y: groups of 128 words, so that the
// blocks in flight share a few word groups and the gathered slice of the
// layer input (w_in rows x 128 words) stays in L2.  Warp r of a block takes
// nodes n0 + r, n0 + r + kHSWarps, ... of its slice; one ring stage holds one
// node's k rows over the block's 128 words (4 words per lane), and the
// node's level-0 pairs are read from shared memory (broadcast loads), which
// keeps the kernel at 128 registers and 16 warps per SM.  The node
// outputs feed, four nodes at a time, a carry-save tree into per-lane
// bit-sliced counters (ones, twos, then kHeadNB ripple planes of weight 4,
// 8, ...).  At the end the warps' counters are added bit-sliced in shared
// memory, each lane turns one bit column into a per-sample count, and one
// integer atomicAdd per (sample, class) publishes the block's total (exact
// and order-independent).

#ifndef BITLOGIC_HEAD_WARPS
#define BITLOGIC_HEAD_WARPS 8
#endif
#ifndef BITLOGIC_HEAD_MINB
#define BITLOGIC_HEAD_MINB 2
#endif
constexpr int kHeadMinBlocks = BITLOGIC_HEAD_MINB;
constexpr int kHeadRing = 4;      // node stages per warp ring
constexpr int kHSWarps = BITLOGIC_HEAD_WARPS;     // warps per block of the staged head
constexpr int kHeadNB = 5;      // weight-4 planes: up to 4 * 31 + 3 = 127 nodes per warp
constexpr int kHeadPlanes = 2 + kHeadNB;
constexpr int kSumPlanes = kHeadPlanes + 3;   // sum of kHSWarps <= 8 warps' counts
constexpr int kMaxNodesPerWarp = 4 * ((1 << kHeadNB) - 1) + 3;
static_assert(kHSWarps <= 8, "kSumPlanes assumes at most 8 warps");

// The block's node slice (connectivity rows, checked once, and tables) is
// staged in shared memory behind the ring: at most kHeadSliceNodes nodes.
// Two blocks per SM of 8 warps: 2 x (113664 + 2048 static + 1024) <= 228 KB.
constexpr int kHeadSliceNodes = 60 * kHSWarps;

template <int k>
__host__ __device__ constexpr int head_ring_bytes() {
    const int ring = kHSWarps * ring_bytes_per_warp<k>(kHeadRing);
    const int flush = (kHSWarps * kHeadPlanes + kSumPlanes) * kStageWords * 4;
    return ring > flush ? ring : flush;
}

template <int k>
__host__ __device__ constexpr int head_smem_bytes() {
    return head_ring_bytes<k>() + kHeadSliceNodes * (k * 4 + 8);
}

template <int k, bool FULL>
__device__ __forceinline__ void head_staged_body(const uint4* __restrict__ xp4, int w_in, long long W,
                                                 long long N, const int* __restrict__ conn,
                                                 const uint64_t* __restrict__ table, int C, int g,
                                                 int splits, int per_split, uint32_t* __restrict__ yp,
                                                 int* __restrict__ counts, uint32_t tail_mask,
                                                 uint4* ring_smem, int2* sPQ, const int* sConn,
                                                 const uint64_t* sTab) {
    constexpr int kSlot = k * 32;   // uint4 per stage
    static_assert(kHeadRing == 4, "a loop iteration is kHeadRing node steps");
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int c = blockIdx.x / splits, sp = blockIdx.x - c * splits;
    const int n0 = c * g + sp * per_split;
    const int n1 = min(c * g + g, n0 + per_split);
    const long long wq = (long long)blockIdx.y * kStageWords + 4 * lane;   // this lane's 4 words
    const bool active = FULL || wq < W;   // W % 4 == 0: all four words are in range
    const uint32_t W4 = (uint32_t)(W >> 2), wq4 = (uint32_t)(wq >> 2);
    uint4* ring = ring_smem + (size_t)warp * (kHeadRing * kSlot) + lane;
    const int jfirst = n0 + warp;

    // issue stream: node ji, kHeadRing - 1 nodes ahead of the compute stream;
    // its rows come from the staged slice (broadcast loads)
    int ji = jfirst;
    auto issue = [&](int slot) {
        if (ji < n1) {
            if (active) {
                const int* rr = sConn + (ji - n0) * k;
                uint32_t off[k];
#pragma unroll
                for (int i = 0; i < k; ++i) off[i] = (uint32_t)rr[i] * W4 + wq4;
                issue_stage<k>(ring + slot * kSlot, xp4, off, 0u);
            }
            ji += kHSWarps;
        }
        cp_async_commit();
    };
    issue(0);
    issue(1);
    issue(2);
    uint32_t ones[4], twos[4], big[kHeadNB][4];
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        ones[r] = twos[r] = 0;
#pragma unroll
        for (int b = 0; b < kHeadNB; ++b) big[b][r] = 0;
    }
    // node step u of a loop iteration (node jj): the loop body has kHeadRing
    // steps, so step u reads slot u and refills slot u + 3 (mod kHeadRing).
    // Returns the node's four output words (0 past the slice or the words).
    auto node = [&](int jj, int u, uint32_t (&y)[4]) {
        __syncwarp();   // the previous node's pairs are read
        node_pairs_smem<k>(jj < n1 ? sTab[jj - n0] : 0ull, lane, sPQ);   // 0 past the slice: harmless
        issue((u + kHeadRing - 1) % kHeadRing);
        cp_async_wait<kHeadRing - 1>();
#pragma unroll
        for (int r = 0; r < 4; ++r) y[r] = 0;
        if (jj < n1 && active) {
            uint32_t x[4][k];
            read_stage<k>(ring + u * kSlot, x);
            mux_tree4_smem<k - 1, 0, k>(sPQ, x, y);
            if constexpr (!FULL) {
                if (wq + 4 == W) y[3] &= tail_mask;
            }
            if (yp) store_words<4>(yp + (long long)jj * W + wq, y);
        }
    };
#pragma unroll 1
    for (int j = jfirst; j < n1; j += 4 * kHSWarps) {
        uint32_t ya[4], yb[4], t1[4];
        node(j, 0, ya);
        node(j + kHSWarps, 1, yb);
#pragma unroll
        for (int r = 0; r < 4; ++r) csa(t1[r], ones[r], ones[r], ya[r], yb[r]);
        node(j + 2 * kHSWarps, 2, ya);
        node(j + 3 * kHSWarps, 3, yb);
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            uint32_t t2, e;
            csa(t2, ones[r], ones[r], ya[r], yb[r]);
            csa(e, twos[r], twos[r], t1[r], t2);
#pragma unroll
            for (int b = 0; b < kHeadNB; ++b) {   // ripple-add the weight-4 word
                const uint32_t cy = big[b][r] & e;
                big[b][r] ^= e;
                e = cy;
            }
        }
    }
    cp_async_wait<0>();
    __syncthreads();   // every warp is done with its ring: reuse it for the flush

    // planes [warp][plane][word], then the block sum [plane][word]
    uint32_t* pl = reinterpret_cast<uint32_t*>(ring_smem);
    uint32_t* sum = pl + kHSWarps * kHeadPlanes * kStageWords;
    {
        uint4* mine = reinterpret_cast<uint4*>(pl + warp * kHeadPlanes * kStageWords) + lane;
        mine[0] = make_uint4(ones[0], ones[1], ones[2], ones[3]);
        mine[kStageWords / 4] = make_uint4(twos[0], twos[1], twos[2], twos[3]);
#pragma unroll
        for (int b = 0; b < kHeadNB; ++b)
            mine[(2 + b) * (kStageWords / 4)] = make_uint4(big[b][0], big[b][1], big[b][2], big[b][3]);
    }
    __syncthreads();
    if (threadIdx.x < kStageWords) {
        const int wd = threadIdx.x;
        uint32_t a[kSumPlanes];
#pragma unroll
        for (int pp = 0; pp < kSumPlanes; ++pp) a[pp] = pp < kHeadPlanes ? pl[pp * kStageWords + wd] : 0u;
#pragma unroll
        for (int wr = 1; wr < kHSWarps; ++wr) {   // bit-sliced ripple-carry add of warp wr
            uint32_t cy = 0;
#pragma unroll
            for (int pp = 0; pp < kSumPlanes; ++pp) {
                const uint32_t b = pp < kHeadPlanes ? pl[(wr * kHeadPlanes + pp) * kStageWords + wd] : 0u;
                const uint32_t ao = a[pp], u = ao ^ b;
                a[pp] = u ^ cy;
                cy = (ao & b) | (u & cy);
            }
        }
#pragma unroll
        for (int pp = 0; pp < kSumPlanes; ++pp) sum[pp * kStageWords + wd] = a[pp];
    }
    __syncthreads();
    for (int wd = warp; wd < kStageWords; wd += kHSWarps) {
        int cnt = 0;
#pragma unroll
        for (int pp = 0; pp < kSumPlanes; ++pp) cnt |= (int)((sum[pp * kStageWords + wd] >> lane) & 1u) << pp;
        const long long s = ((long long)blockIdx.y * kStageWords + wd) * 32 + lane;
        if (cnt && s < N) atomicAdd(counts + s * C + c, cnt);
    }
}


template <int k>
__global__ void __launch_bounds__(kHSWarps * 32, kHeadMinBlocks)
hard_head_staged_kernel(const uint4* __restrict__ xp4, int w_in, long long W, long long N,
                        const int* __restrict__ conn, const uint64_t* __restrict__ table,
                        int C, int g, int splits, int per_split, uint32_t* __restrict__ yp,
                        int* __restrict__ counts, uint32_t tail_mask) {
    constexpr int H = 1 << (k - 1);
    extern __shared__ uint4 ring_smem[];
    __shared__ __align__(16) int2 sPQ[kHSWarps][H < 2 ? 2 : H];
    int* sConn = reinterpret_cast<int*>(reinterpret_cast<unsigned char*>(ring_smem) + head_ring_bytes<k>());
    uint64_t* sTab = reinterpret_cast<uint64_t*>(sConn + kHeadSliceNodes * k);
    {   // stage the slice: out-of-range rows read row 0 and raise the flag
        const int c = blockIdx.x / splits, sp = blockIdx.x - c * splits;
        const int n0 = c * g + sp * per_split;
        const int cnt = max(0, min(c * g + g, n0 + per_split) - n0);
        bool bad = false;
        for (int t = threadIdx.x; t < cnt * k; t += kHSWarps * 32) {
            int v = __ldg(conn + (long long)n0 * k + t);
            if ((unsigned)v >= (unsigned)w_in) {
                bad = true;
                v = 0;
            }
            sConn[t] = v;
        }
        for (int t = threadIdx.x; t < cnt; t += kHSWarps * 32) sTab[t] = __ldg(table + n0 + t);
        if (bad) flag_index_error();
        __syncthreads();
    }
    const long long end = (long long)(blockIdx.y + 1) * kStageWords;
    const bool full = end < W || (end == W && tail_mask == 0xffffffffu);
    int2* mine = sPQ[threadIdx.x >> 5];
    if (full)
        head_staged_body<k, true>(xp4, w_in, W, N, conn, table, C, g, splits, per_split, yp, counts,
                                  tail_mask, ring_smem, mine, sConn, sTab);
    else
        head_staged_body<k, false>(xp4, w_in, W, N, conn, table, C, g, splits, per_split, yp, counts,
                                   tail_mask, ring_smem, mine, sConn, sTab);
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

// Opt in to more than the default 48 KB of shared memory per block when the
// dynamic part plus the kernel's static part (a few KB) may exceed it.
template <typename F>
int set_dynamic_smem(F* kernel, int bytes) {
    if (bytes <= 40 * 1024) return BITLOGIC_OK;
    return cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes) == cudaSuccess
               ? BITLOGIC_OK : BITLOGIC_ERR_CUDA;
}

template <int k>
int launch_hard(const uint32_t* xp, int w_in, long long N, const int* conn, const uint64_t* table,
                int w, uint32_t* yp, int C, int* counts, int* pred, cudaStream_t st) {
    const long long W = (N + 31) / 32;
    const uint32_t tail_mask = (N % 32) ? ((1u << (N % 32)) - 1u) : 0xffffffffu;
    // staged kernels: 16-byte rows and 32-bit row offsets in 16-byte units
    const bool vec4 = (W % 4 == 0) && aligned16(xp) && (!yp || aligned16(yp)) &&
                      (unsigned long long)w_in * (unsigned long long)(W / 4) < (1ull << 32);
    if (C == 0) {
        if (vec4) {
            // chunks of kLayerNS stages; nodes per warp: enough blocks for
            // about four waves of two per SM
            const long long gy = (W + kLayerNS * kStageWords - 1) / (kLayerNS * kStageWords);
            if (gy > 65535) return BITLOGIC_ERR_SHAPE;
            const long long groups = (w + kHardWarps - 1) / kHardWarps;
            long long npw = groups * gy / (8ll * sm_count());
            npw = npw < 1 ? 1 : (npw > 8 ? 8 : npw);
            const long long gx = (w + kHardWarps * npw - 1) / (kHardWarps * npw);
            const int smem = kHardWarps * ring_bytes_per_warp<k>(kLayerNS);
            if (set_dynamic_smem(hard_layer_staged_kernel<k>, smem)) return BITLOGIC_ERR_CUDA;
            hard_layer_staged_kernel<k><<<dim3((unsigned)gx, (unsigned)gy), kHardWarps * 32, smem, st>>>(
                reinterpret_cast<const uint4*>(xp), w_in, W, conn, table, w, yp, tail_mask);
        } else {
            const long long chunk = hard_word_chunk(w_in, W);
            const long long ny = (W + chunk - 1) / chunk;
            if (ny > 65535) return BITLOGIC_ERR_SHAPE;
            dim3 grid((unsigned)((w + kHardWarps - 1) / kHardWarps), (unsigned)ny);
            hard_layer_kernel<k, 1><<<grid, kHardWarps * 32, 0, st>>>(xp, w_in, W, conn, table, w, yp, chunk,
                                                                     tail_mask);
        }
        return launch_status();
    }
    const int g = w / C;
    if (cudaMemsetAsync(counts, 0, sizeof(int) * (size_t)N * (size_t)C, st) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    if (vec4) {
        const long long wg = W / kStageWords + (W % kStageWords ? 1 : 0);
        // split a class over several blocks until a word group has about one
        // block per SM (the blocks in flight then share one or two word
        // groups), keeping at least 8 nodes per warp
        int splits = 1;
        while (C * splits < sm_count() && g / (splits * 2) >= 8 * kHSWarps) splits *= 2;
        int per_split = (g + splits - 1) / splits;
        // counter capacity and the staged slice
        while ((per_split + kHSWarps - 1) / kHSWarps > kMaxNodesPerWarp || per_split > kHeadSliceNodes) {
            splits *= 2;
            per_split = (g + splits - 1) / splits;
        }
        if ((long long)C * splits > 0x7fffffffll || wg > 65535) return BITLOGIC_ERR_SHAPE;
        const int smem = head_smem_bytes<k>();
        if (set_dynamic_smem(hard_head_staged_kernel<k>, smem)) return BITLOGIC_ERR_CUDA;
        hard_head_staged_kernel<k><<<dim3((unsigned)(C * splits), (unsigned)wg), kHSWarps * 32, smem, st>>>(
            reinterpret_cast<const uint4*>(xp), w_in, W, N, conn, table, C, g, splits, per_split, yp, counts,
            tail_mask);
    } else {
        const long long wg = (W + 31) / 32;
        int splits = 1;
        while (wg * C * splits < 608 && g / (splits * 2) >= 64) splits *= 2;
        int per_split = (g + splits - 1) / splits;
        // each warp's slice must fit the counters
        while ((per_split + kHeadWarps - 1) / kHeadWarps > 8 * ((1 << kBigPlanes) - 1)) {
            splits *= 2;
            per_split = (g + splits - 1) / splits;
        }
        if ((long long)C * splits > 65535) return BITLOGIC_ERR_SHAPE;
        dim3 grid((unsigned)wg, (unsigned)(C * splits));
        hard_head_kernel<k, 1><<<grid, kHeadWarps * 32, 0, st>>>(xp, w_in, W, N, conn, table, C, g, splits,
                                                                per_split, yp, counts, tail_mask);
    }
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
