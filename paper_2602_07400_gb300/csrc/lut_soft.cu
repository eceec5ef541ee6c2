// Soft (training) forward and backward of a fixed-connectivity LUT layer.
//
// Node (LightLUT, §2 of the paper: Kronecker-indicator basis, 2^k logits per
// node), read as t = sigmoid(theta), y = sum_a t_a prod_i x_i^{a_i}(1-x_i)^{1-a_i}
// with connectivity slot i = bit i of the table index a.  The straight-through
// hard form of the same node (§4 node sweep) takes t_a = [theta_a > 0] in the
// forward and in the input gradient, and the sigmoid slope for dtheta; only
// the per-node table set-up differs between the two forms.
//
// Evaluation: the multilinear form is a complete binary lerp tree over the
// k inputs (level l interpolates with x_l), 2^k - 1 lerps per (node, sample).
// Level 0 uses per-node constants (t_even, t_odd - t_even), so it costs one
// FFMA per lerp; every other lerp is one FADD and one FFMA.  The backward is
// reverse mode through the same tree: the adjoint of each subtree is pushed
// down (two FMULs per lerp), each lerp adds adjoint * (hi - lo) into dx_l, and
// at the leaves the adjoint is g * w_a, accumulated for dtheta.
//
// Data movement: activations are feature-major [rows][B], so the k rows a
// node gathers are contiguous batch segments.  The vector paths stream them
// through a ring of shared-memory stages filled by 16-byte cp.async copies,
// which overlaps the gathers with the trees of earlier stages without
// spending registers.
#include <type_traits>

#include "common.cuh"

namespace bitlogic {
namespace {

#ifndef BITLOGIC_BWD_MIN_BLOCKS
#define BITLOGIC_BWD_MIN_BLOCKS 16  // dtheta-only kernel: blocks per SM (k >= 4)
#endif
#ifndef BITLOGIC_BWD_MIN_BLOCKS_SMALL
#define BITLOGIC_BWD_MIN_BLOCKS_SMALL 24  // dtheta-only kernel: blocks per SM (k <= 3, fewer registers)
#endif
#ifndef BITLOGIC_NODE_MIN_BLOCKS
#define BITLOGIC_NODE_MIN_BLOCKS 12  // backward with input gradient: blocks per SM
#endif
#ifndef BITLOGIC_FWD_WARPS
#define BITLOGIC_FWD_WARPS 1
#endif
#ifndef BITLOGIC_FWD_MIN_CHUNK
#define BITLOGIC_FWD_MIN_CHUNK 1024
#endif
#ifndef BITLOGIC_FWD_WAVES
#define BITLOGIC_FWD_WAVES 2
#endif
constexpr int kFwdWarps = BITLOGIC_FWD_WARPS;
static_assert(kFwdWarps >= 1 && kFwdWarps <= 16, "forward warps per block");
static_assert(BITLOGIC_FWD_MIN_CHUNK % 128 == 0 && BITLOGIC_FWD_MIN_CHUNK >= 128, "whole stages per chunk");
#ifndef BITLOGIC_BWD_WARPS
#define BITLOGIC_BWD_WARPS 1
#endif
constexpr int kBwdWarps = BITLOGIC_BWD_WARPS;   // warps per block in the staged backward
#ifndef BITLOGIC_BWD_WARPS_PER_NODE
#define BITLOGIC_BWD_WARPS_PER_NODE 1
#endif
constexpr int kWarpsPerNode = BITLOGIC_BWD_WARPS_PER_NODE;   // 1, 2 or 4
constexpr int kNodesPerBlock = kBwdWarps / kWarpsPerNode;
static_assert(kWarpsPerNode == 1 || kWarpsPerNode == 2 || kWarpsPerNode == 4, "1, 2 or 4 warps per node");
static_assert(kBwdWarps >= kWarpsPerNode && kBwdWarps % kWarpsPerNode == 0 && kBwdWarps <= 16,
              "whole nodes per block");
// ---------------------------------------------------------------- trees --

template <int L, int M, int H, int k>
__device__ __forceinline__ float fwd_tree(const float (&te)[H], const float (&d)[H],
                                          const float (&x)[k]) {
    if constexpr (L == 0) {
        return fmaf(x[0], d[M], te[M]);
    } else {
        const float lo = fwd_tree<L - 1, 2 * M>(te, d, x);
        const float hi = fwd_tree<L - 1, 2 * M + 1>(te, d, x);
        return fmaf(x[L], hi - lo, lo);
    }
}

// Reverse tree of the subtree at level L, index M; `adj` is the adjoint of
// its output.  Returns the subtree value, adds adjoint * (hi - lo) into
// dx[l] for each lerp at level l (the lerp with M == 0 is the first to touch
// dx[l] and initialises it), and the leaf adjoints into acc.
template <int L, int M, int H, int K, int k>
__device__ __forceinline__ float bwd_tree(const float (&te)[H], const float (&d)[H],
                                          const float (&x)[k], const float (&omx)[k],
                                          float adj, float (&dx)[k], float (&acc)[K]) {
    if constexpr (L == 0) {
        if constexpr (M == 0) dx[0] = adj * d[M];
        else dx[0] = fmaf(adj, d[M], dx[0]);
        acc[2 * M] = fmaf(adj, omx[0], acc[2 * M]);
        acc[2 * M + 1] = fmaf(adj, x[0], acc[2 * M + 1]);
        return fmaf(x[0], d[M], te[M]);
    } else {
        const float lo = bwd_tree<L - 1, 2 * M>(te, d, x, omx, adj * omx[L], dx, acc);
        const float hi = bwd_tree<L - 1, 2 * M + 1>(te, d, x, omx, adj * x[L], dx, acc);
        const float diff = hi - lo;
        if constexpr (M == 0) dx[L] = adj * diff;
        else dx[L] = fmaf(adj, diff, dx[L]);
        return fmaf(x[L], diff, lo);
    }
}

// ------------------------------------------- subtable polynomial forms --
//
// A subtable of 2^L consecutive table entries over x_0..x_{L-1} is the
// multilinear polynomial sum_S c_S prod_{i in S} x_i whose coefficients are
// the subset differences (Moebius transform) of its entries.  Evaluated by
// Horner steps it costs 2^L - 1 FFMA, against 2^L - 1 lerps (about twice the
// instructions) for the same subtable as a lerp tree.  The upper levels stay
// lerps.  |c_S| <= 2^(L-1), so rounding stays at a few ulp of 1.

// In-place subset-difference transform of 2^L values.
template <int L>
__device__ __forceinline__ void moebius(float (&c)[1 << L]) {
#pragma unroll
    for (int b = 0; b < L; ++b)
#pragma unroll
        for (int a = 0; a < (1 << L); ++a)
            if (a & (1 << b)) c[a] -= c[a ^ (1 << b)];
}

// Horner value of the subtable whose coefficients start at cf[O].
template <int L, int O, int N, int k>
__device__ __forceinline__ float poly(const float (&cf)[N], const float (&x)[k]) {
    if constexpr (L == 1) {
        return fmaf(cf[O + 1], x[0], cf[O]);
    } else {
        const float lo = poly<L - 1, O>(cf, x);
        const float hi = poly<L - 1, O + (1 << (L - 1))>(cf, x);
        return fmaf(x[L - 1], hi, lo);
    }
}

// Forward tree with Moebius subtables of 2^L entries at the bottom: value of
// the subtree at level LV (levels below L are inside the subtables).
template <int LV, int M, int L, int N, int k>
__device__ __forceinline__ float fwd_tree_poly(const float (&cf)[N], const float (&x)[k]) {
    if constexpr (LV == L - 1) {
        return poly<L, M * (1 << L)>(cf, x);
    } else {
        const float lo = fwd_tree_poly<LV - 1, 2 * M, L>(cf, x);
        const float hi = fwd_tree_poly<LV - 1, 2 * M + 1, L>(cf, x);
        return fmaf(x[LV], hi - lo, lo);
    }
}

__host__ __device__ constexpr int fwd_poly_levels(int k) { return k < 3 ? k : 3; }

// Reverse tree whose leaves are 4-entry subtables in Moebius form over
// (x_0, x_1): quad m has coefficients cq[4m .. 4m+3] = (c0, c1, c2, c3),
// value v = (c0 + c1 x0) + x1 (c2 + c3 x0), dv/dx0 = c1 + c3 x1,
// dv/dx1 = c2 + c3 x0, and entry a of the quad has corner weight W[a]
// (W = ((1-x0)(1-x1), x0(1-x1), (1-x0)x1, x0 x1), shared by all quads), so
// its leaf adjoint is adj * W[a].  Above the quads the lerps of bwd_tree.
template <int LV, int M, int N, int NA, int k>
__device__ __forceinline__ float bwd_tree_quad(const float (&cq)[N], const float (&x)[k],
                                               const float (&omx)[k], const float (&W)[4],
                                               float adj, float (&dx)[k], float (&acc)[NA]) {
    if constexpr (LV == 1) {
        const float c0 = cq[4 * M], c1 = cq[4 * M + 1], c2 = cq[4 * M + 2], c3 = cq[4 * M + 3];
        const float in0 = fmaf(c1, x[0], c0);
        const float in1 = fmaf(c3, x[0], c2);
        const float dv0 = fmaf(c3, x[1], c1);
        if constexpr (M == 0) {
            dx[0] = adj * dv0;
            dx[1] = adj * in1;
        } else {
            dx[0] = fmaf(adj, dv0, dx[0]);
            dx[1] = fmaf(adj, in1, dx[1]);
        }
#pragma unroll
        for (int a = 0; a < 4; ++a) acc[4 * M + a] = fmaf(adj, W[a], acc[4 * M + a]);
        return fmaf(x[1], in1, in0);
    } else {
        const float lo = bwd_tree_quad<LV - 1, 2 * M>(cq, x, omx, W, adj * omx[LV], dx, acc);
        const float hi = bwd_tree_quad<LV - 1, 2 * M + 1>(cq, x, omx, W, adj * x[LV], dx, acc);
        const float diff = hi - lo;
        if constexpr (M == 0) dx[LV] = adj * diff;
        else dx[LV] = fmaf(adj, diff, dx[LV]);
        return fmaf(x[LV], diff, lo);
    }
}

__device__ __forceinline__ float comp(const float4& v, int c) {
    return c == 0 ? v.x : c == 1 ? v.y : c == 2 ? v.z : v.w;
}

__device__ __forceinline__ float4 ldg4(const float* p) {
    return __ldg(reinterpret_cast<const float4*>(p));
}

__device__ __forceinline__ float4 add4(float4 a, const float4& b) {
    a.x += b.x; a.y += b.y; a.z += b.z; a.w += b.w;
    return a;
}

template <int k>
__device__ __forceinline__ void load_rows(const int* __restrict__ conn, int j, int w_in, int lane,
                                          int (&rows)[k]) {
    bool bad = false;
#pragma unroll
    for (int i = 0; i < k; ++i) {
        int c = __ldg(conn + (long long)j * k + i);
        if ((unsigned)c >= (unsigned)w_in) { bad = true; c = 0; }
        rows[i] = c;
    }
    if (bad && lane == 0) flag_index_error();
}

// Table entry of a node form (bitlogic_node_t): the sigmoid sg of the logit
// th for the soft LightLUT node, the hard sample [th > 0] for the
// straight-through node (whose theta gradient still takes the slope of sg).
__device__ __forceinline__ float table_value(float th, float sg, int node) {
    return node == BITLOGIC_NODE_ST ? (th > 0.f ? 1.f : 0.f) : sg;
}

// Per-warp node set-up: connectivity rows (range-checked), table entries of
// the node form, level-0 constants broadcast to every lane through shared
// memory.  Lane l (l < 2^(k-1)) keeps the sigmoids of entries 2l and 2l+1
// for the dtheta epilogue.
template <int k>
__device__ __forceinline__ void node_setup(const int* __restrict__ conn,
                                           const float* __restrict__ theta, int j, int w_in,
                                           int node, int lane, float2* sPair, int (&rows)[k],
                                           float (&te)[1 << (k - 1)], float (&d)[1 << (k - 1)],
                                           float& t0, float& t1) {
    constexpr int K = 1 << k, H = K / 2;
    load_rows<k>(conn, j, w_in, lane, rows);
    t0 = t1 = 0.f;
    if (lane < H) {
        const float th0 = __ldg(theta + (long long)j * K + 2 * lane);
        const float th1 = __ldg(theta + (long long)j * K + 2 * lane + 1);
        t0 = sigmoidf(th0);
        t1 = sigmoidf(th1);
        const float v0 = table_value(th0, t0, node), v1 = table_value(th1, t1, node);
        sPair[lane] = make_float2(v0, v1 - v0);
    }
    __syncwarp();
#pragma unroll
    for (int m = 0; m < H; ++m) {
        const float2 v = sPair[m];
        te[m] = v.x;
        d[m] = v.y;
    }
    __syncwarp();
}

#ifndef BITLOGIC_STAGES
#define BITLOGIC_STAGES 3
#endif
// samples per pipeline stage: every lane copies and reads one 16-byte chunk
// (4 consecutive samples) of each row, so a stage is exactly 32 x 4 samples;
// the lane offsets of all staged kernels rely on it
constexpr int kStageSamples = 128;
constexpr int kStages = BITLOGIC_STAGES;                // stages in flight per warp
static_assert(kStageSamples == 32 * 4, "a stage is one 16-byte chunk per lane");
static_assert(kStages >= 2 && kStages <= 8, "the rings hold 2 to 8 stages");

// ------------------------------------------------------------- forward --

// Scalar forward (any B, any alignment): one warp per (node, batch slice),
// one sample per lane.
template <int k>
__global__ void __launch_bounds__(kFwdWarps * 32)
lut_forward_kernel(const float* __restrict__ X, int w_in, long long B,
                   const int* __restrict__ conn, const float* __restrict__ theta, int w,
                   int node, float* __restrict__ Y, long long chunk) {
    constexpr int H = 1 << (k - 1);
    __shared__ float2 sPair[kFwdWarps][H];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kFwdWarps + warp;
    if (j >= w) return;
    int rows[k];
    float te[H], d[H], t0, t1;
    node_setup<k>(conn, theta, j, w_in, node, lane, sPair[warp], rows, te, d, t0, t1);
    const long long s0 = (long long)blockIdx.y * chunk;
    const long long s1 = min(B, s0 + chunk);
    const float* xr[k];
#pragma unroll
    for (int i = 0; i < k; ++i) xr[i] = X + (long long)rows[i] * B;
    float* yr = Y + (long long)j * B;
    for (long long s = s0 + lane; s < s1; s += 32) {
        float x[k];
#pragma unroll
        for (int i = 0; i < k; ++i) x[i] = __ldg(xr[i] + s);
        yr[s] = fwd_tree<k - 1, 0>(te, d, x);
    }
}

// Staged forward: one warp per (node, batch slice).  Each lane copies, reads
// back and evaluates its own 4 consecutive samples of a stage (16-byte
// chunks), so the ring needs no warp synchronisation.  Needs B % 4 == 0,
// chunk % 4 == 0 and 16-byte aligned X and Y.
template <int k>
__global__ void __launch_bounds__(kFwdWarps * 32)
lut_forward_staged_kernel(const float* __restrict__ X, int w_in, long long B,
                          const int* __restrict__ conn, const float* __restrict__ theta, int w,
                          int node, float* __restrict__ Y, long long chunk) {
    constexpr int K = 1 << k, CH = kStageSamples, L = fwd_poly_levels(k), S = 1 << L;
    __shared__ __align__(16) float sRing[kFwdWarps][kStages * k * CH];
    __shared__ __align__(16) float sCoef[kFwdWarps][K];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kFwdWarps + warp;
    if (j >= w) return;
    int rows[k];
    load_rows<k>(conn, j, w_in, lane, rows);
    // table entries spread over the lanes (entries l, l + 32), then lane
    // l < K / S turns subtable l into its Moebius coefficients
#pragma unroll
    for (int a = lane; a < K; a += 32) {
        const float th = __ldg(theta + (long long)j * K + a);
        sCoef[warp][a] = table_value(th, sigmoidf(th), node);
    }
    __syncwarp();
    if (lane < K / S) {
        float c[S];
#pragma unroll
        for (int a = 0; a < S; ++a) c[a] = sCoef[warp][lane * S + a];
        moebius<L>(c);
#pragma unroll
        for (int a = 0; a < S; ++a) sCoef[warp][lane * S + a] = c[a];
    }
    __syncwarp();
    float cf[K];
#pragma unroll
    for (int a = 0; a < K; a += 4) {
        const float4 v = *reinterpret_cast<const float4*>(&sCoef[warp][a]);
        cf[a] = v.x; cf[a + 1] = v.y; cf[a + 2] = v.z; cf[a + 3] = v.w;
    }
    float* ring = sRing[warp] + 4 * lane;       // this lane's column of every stage row
    const long long s0 = (long long)blockIdx.y * chunk;
    const long long s1 = min(B, s0 + chunk);
    const float* src[k];
#pragma unroll
    for (int i = 0; i < k; ++i) src[i] = X + (long long)rows[i] * B + s0 + 4 * lane;
    float* yr = Y + (long long)j * B + s0 + 4 * lane;
    const int nst = (int)((s1 - s0 + CH - 1) / CH);
    const long long lim = s1 - s0 - 4 * lane;   // this lane's chunks start below lim

    int ib = 0;   // ring slot of the next stage to issue
    auto issue = [&](int st) {
        if (st < nst && (long long)st * CH < lim) {
            float* buf = ring + ib * (k * CH);
#pragma unroll
            for (int r = 0; r < k; ++r) cp_async16(buf + r * CH, src[r] + (long long)st * CH);
        }
        cp_async_commit();
        ib = (ib + 1 == kStages) ? 0 : ib + 1;
    };
#pragma unroll
    for (int st = 0; st < kStages - 1; ++st) issue(st);
    int rb = 0;   // ring slot of the stage being evaluated
    for (int st = 0; st < nst; ++st) {
        issue(st + kStages - 1);
        cp_async_wait<kStages - 1>();
        if ((long long)st * CH < lim) {
            const float* buf = ring + rb * (k * CH);
            float4 xv[k];
#pragma unroll
            for (int i = 0; i < k; ++i) xv[i] = *reinterpret_cast<const float4*>(buf + i * CH);
            float o[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float x[k];
#pragma unroll
                for (int i = 0; i < k; ++i) x[i] = comp(xv[i], c);
                o[c] = fwd_tree_poly<k - 1, 0, L>(cf, x);
            }
            *reinterpret_cast<float4*>(yr + (long long)st * CH) = make_float4(o[0], o[1], o[2], o[3]);
        }
        rb = (rb + 1 == kStages) ? 0 : rb + 1;
    }
    cp_async_wait<0>();
}

// ------------------------------------------------------------ backward --

// Where a node's output gradient dY[j][.] comes from.
//   rows:  dY + (j / group) * B   (group = 1: one row per node; group = g:
//          the head's per-class gradient, shared by the g nodes of a class)
//   terms: sum over e in [off[j], off[j+1]) of terms[edge[e]][.] in
//          increasing e -- the next layer's input gradient, reduced on the
//          fly from its per-edge terms instead of being materialised.  With
//          edge == nullptr the term rows are stored in CSR order (row e).
struct GradSource {
    const float* dY;
    int group;
    const float* terms;
    const int* off;
    const int* edge;
    int n_edges;
};

// Term row of CSR position e (edge == nullptr: rows in CSR order).
__device__ __forceinline__ int term_row(const GradSource& gs, int e) {
    return gs.edge ? __ldg(gs.edge + e) : e;
}

// Row of edge e's term in the per-edge buffer: e itself, or pos[e] when the
// caller asks for CSR order (an out-of-range position raises the flag and
// falls back to row e, so every store stays inside the buffer).
__device__ __forceinline__ long long edge_row(const int* __restrict__ pos, long long e, long long n) {
    if (!pos) return e;
    const int r = __ldg(pos + e);
    if (r >= 0 && (long long)r < n) return r;
    flag_index_error();
    return e;
}

// CSR range of node j in the upstream terms (range-checked).
__device__ __forceinline__ void term_range(const GradSource& gs, int j, int lane, int& e0, int& e1) {
    e0 = __ldg(gs.off + j);
    e1 = __ldg(gs.off + j + 1);
    if (e0 < 0 || e1 < e0 || e1 > gs.n_edges) {
        if (lane == 0) flag_index_error();
        e0 = e1 = 0;
    }
}

// Scalar backward (any B, any alignment, any k): one warp per node, one
// sample per lane, next sample's gathers issued before this sample's tree.
template <int k, bool WANT_DX, bool TERMS>
__global__ void __launch_bounds__(kFwdWarps * 32)
lut_backward_kernel(const float* __restrict__ X, int w_in, long long B,
                    const int* __restrict__ conn, const float* __restrict__ theta, int w, int node,
                    GradSource gs, float* __restrict__ dtheta, float* __restrict__ P,
                    const int* __restrict__ epos, float* __restrict__ dY_out) {
    constexpr int K = 1 << k, H = K / 2;
    __shared__ float2 sPair[kFwdWarps][H];
    __shared__ float sRed[kFwdWarps][32][K + 1];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kFwdWarps + warp;
    if (j >= w) return;
    int rows[k];
    float te[H], d[H], t0, t1;
    node_setup<k>(conn, theta, j, w_in, node, lane, sPair[warp], rows, te, d, t0, t1);
    int e0 = 0, e1 = 0;
    if constexpr (TERMS) term_range(gs, j, lane, e0, e1);
    const float* gr = TERMS ? nullptr : gs.dY + (long long)(j / gs.group) * B;
    float* pr[WANT_DX ? k : 1];
    if constexpr (WANT_DX) {
#pragma unroll
        for (int i = 0; i < k; ++i) pr[i] = P + edge_row(epos, (long long)j * k + i, (long long)w * k) * B;
    }

    auto grad = [&](long long s) {
        if constexpr (TERMS) {
            float g = 0.f;
            for (int e = e0; e < e1; ++e) {
                const int id = term_row(gs, e);
                if ((unsigned)id < (unsigned)gs.n_edges) g += __ldg(gs.terms + (long long)id * B + s);
                else if (lane == 0) flag_index_error();
            }
            return g;
        } else {
            return __ldg(gr + s);
        }
    };

    float acc[K];
#pragma unroll
    for (int a = 0; a < K; ++a) acc[a] = 0.f;
    float xn[k], gn = 0.f;
#pragma unroll
    for (int i = 0; i < k; ++i) xn[i] = 0.f;
    if (lane < B) {
#pragma unroll
        for (int i = 0; i < k; ++i) xn[i] = __ldg(X + (long long)rows[i] * B + lane);
        gn = grad(lane);
    }
    for (long long s = lane; s < B; s += 32) {
        float x[k], omx[k], dx[k];
        const float g = gn;
#pragma unroll
        for (int i = 0; i < k; ++i) {
            x[i] = xn[i];
            omx[i] = 1.0f - x[i];
        }
        if (s + 32 < B) {
#pragma unroll
            for (int i = 0; i < k; ++i) xn[i] = __ldg(X + (long long)rows[i] * B + s + 32);
            gn = grad(s + 32);
        }
        if (dY_out) dY_out[(long long)j * B + s] = g;
        bwd_tree<k - 1, 0>(te, d, x, omx, g, dx, acc);
        if constexpr (WANT_DX) {
#pragma unroll
            for (int i = 0; i < k; ++i) pr[i][s] = dx[i];
        }
    }
#pragma unroll
    for (int a = 0; a < K; ++a) sRed[warp][lane][a] = acc[a];
    __syncwarp();
    if (lane < H) {
        float s0 = 0.f, s1 = 0.f;
#pragma unroll 8
        for (int r = 0; r < 32; ++r) {
            s0 += sRed[warp][r][2 * lane];
            s1 += sRed[warp][r][2 * lane + 1];
        }
        float* out = dtheta + (long long)j * K + 2 * lane;
        out[0] = t0 * (1.0f - t0) * s0;
        out[1] = t1 * (1.0f - t1) * s1;
    }
}

// ---------------------------------------- backward, one block per node --

constexpr int kGatherStages = 4;   // stages whose upstream rows are gathered together

// Per-warp shared memory of the staged backward: the cp.async ring (k input
// rows, plus the gradient row for a dY source) and, for a CSR-terms source,
// the summed gradient of kGatherStages stages; reused for the dtheta
// transpose at the end.
template <int k, bool TERMS>
__host__ __device__ constexpr int ring_floats() {
    return kStages * (TERMS ? k : k + 1) * kStageSamples;
}
template <int k, bool TERMS>
__host__ __device__ constexpr int node_floats_per_warp() {
    constexpr int rows = ring_floats<k, TERMS>() + (TERMS ? kGatherStages * kStageSamples : 0);
    constexpr int red = 32 * ((1 << (k - 1)) + 1);
    return rows > red ? rows : red;
}

template <int k, bool TERMS>
constexpr size_t node_smem_bytes() {
    return (size_t)kBwdWarps * node_floats_per_warp<k, TERMS>() * sizeof(float) +
           (size_t)kNodesPerBlock * (1 << k) * sizeof(float);
}

// Staged backward.  A block holds kNodesPerBlock nodes with kWarpsPerNode
// warps each (by default one warp per node and per block, over the whole
// batch); each warp of a node takes a contiguous range of its 128-sample
// stages.
//
// Within a warp every sample is split over two lanes: lane h = lane & 1 owns
// the half of the table whose top input x_{k-1} equals h, i.e. one of the two
// subtrees under the root lerp.  Each lane runs the reverse tree of its
// subtree (adjoint g * (h ? x_{k-1} : 1 - x_{k-1})) and accumulates the leaf
// adjoints of its half for dtheta; the pair exchanges one value per stored
// slot by shuffle (the partner's partial dx_i, or the subtree value that
// gives dx_{k-1} = g * (v_1 - v_0)).  Lane h stores the slots i with
// i % 2 == h.  Halving the per-thread table and accumulators doubles the
// resident warps.
//
// The k gathered rows (and, for a dY source, the node's gradient row) stream
// through a kStages-deep cp.async ring.  For a CSR-terms source the node's
// edge ids are read once into lanes; every kGatherStages stages the warp
// sums the upstream rows in increasing edge order, 2 KB contiguous per row
// (random rows in DRAM want long contiguous reads), into a shared buffer the
// stages then read.  dtheta: each lane's partials, then the lanes of each
// parity, then the node's warps, in a fixed order.  Needs k >= 2,
// B % 4 == 0 and 16-byte aligned X and sources.
template <int k, bool WANT_DX, bool TERMS, bool POS>
__global__ void __launch_bounds__(kBwdWarps * 32, BITLOGIC_NODE_MIN_BLOCKS)
lut_backward_node_kernel(const float* __restrict__ X, int w_in, long long B,
                         const int* __restrict__ conn, const float* __restrict__ theta, int w,
                         int node, GradSource gs, float* __restrict__ dtheta, float* __restrict__ P,
                         const int* __restrict__ epos, float* __restrict__ dY_out) {
    constexpr int K = 1 << k, H = K / 2, H2 = K / 4, R = k + 1, CH = kStageSamples;
    constexpr int NQ = (k + 1) / 2;   // slots stored per lane (rounded up)
    extern __shared__ __align__(16) float smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = lane & 1, pair = lane >> 1;
    const int nb = warp / kWarpsPerNode, sub = warp % kWarpsPerNode;   // node in block, warp in node
    constexpr int FPW = node_floats_per_warp<k, TERMS>();
    float* ring = smem + warp * FPW;
    float* gbuf = ring + ring_floats<k, TERMS>();   // summed upstream gradient (terms source)
    float* sT = smem + kBwdWarps * FPW + nb * K;   // the node's table entries
    const int j = blockIdx.x * kNodesPerBlock + nb;
    const bool live = j < w;   // a dead warp still reaches the block barriers

    int rows[k];
#pragma unroll
    for (int i = 0; i < k; ++i) rows[i] = 0;
    float t0 = 0.f, t1 = 0.f;
    if (live) {
        load_rows<k>(conn, j, w_in, lane, rows);
        if (sub == 0 && lane < H) {   // t0, t1: sigmoids, for the dtheta epilogue
            const float th0 = __ldg(theta + (long long)j * K + 2 * lane);
            const float th1 = __ldg(theta + (long long)j * K + 2 * lane + 1);
            t0 = sigmoidf(th0);
            t1 = sigmoidf(th1);
            *reinterpret_cast<float2*>(sT + 2 * lane) =
                make_float2(table_value(th0, t0, node), table_value(th1, t1, node));
        }
    }
    __syncthreads();
    // this lane's half of the table: entries h*H .. h*H + H - 1, as 4-entry
    // Moebius quads (k >= 3) or as level-0 lerp constants (k == 2)
    constexpr bool QUADS = k >= 3;
    float cq[QUADS ? H : 1];
    float te[QUADS ? 1 : H2], d[QUADS ? 1 : H2];
    if constexpr (QUADS) {
#pragma unroll
        for (int m = 0; m < H / 4; ++m) {
            const float4 t = live ? *reinterpret_cast<const float4*>(sT + h * H + 4 * m)
                                  : make_float4(0.f, 0.f, 0.f, 0.f);
            const float c1 = t.y - t.x;
            cq[4 * m] = t.x;
            cq[4 * m + 1] = c1;
            cq[4 * m + 2] = t.z - t.x;
            cq[4 * m + 3] = (t.w - t.z) - c1;
        }
    } else {
#pragma unroll
        for (int m = 0; m < H2; ++m) {
            const float2 t = live ? *reinterpret_cast<const float2*>(sT + h * H + 2 * m) : make_float2(0.f, 0.f);
            te[m] = t.x;
            d[m] = t.y - t.x;
        }
    }
    // upstream edges of node j: ids held one per lane (the first 32)
    int e0 = 0, deg = 0, my_id = 0;
    if constexpr (TERMS) {
        if (live) {
            int e1;
            term_range(gs, j, lane, e0, e1);
            deg = e1 - e0;
            if (lane < deg) {
                my_id = term_row(gs, e0 + lane);
                if ((unsigned)my_id >= (unsigned)gs.n_edges) {
                    flag_index_error();
                    my_id = -1;   // read as a zero row
                }
            }
        }
    }

    const int jj = live ? j : 0;
    const float* src[R];
#pragma unroll
    for (int i = 0; i < k; ++i) src[i] = X + (long long)rows[i] * B + 4 * lane;
    src[k] = TERMS ? nullptr : gs.dY + (long long)(jj / gs.group) * B + 4 * lane;
    float* pst[NQ];   // this lane's stored slots 2q + h, at its first sample
#pragma unroll
    for (int q = 0; q < NQ; ++q) {
        const long long e = (long long)jj * k + (2 * q + h < k ? 2 * q + h : 0);
        if constexpr (POS) pst[q] = P + (live ? edge_row(epos, e, (long long)w * k) : e) * B + pair;
        else pst[q] = P + e * B + pair;
    }
    const int nst = (int)((B + CH - 1) / CH);
    const int per = (nst + kWarpsPerNode - 1) / kWarpsPerNode;
    const int first = sub * per;
    const int mine = !live ? 0 : max(0, min(nst, first + per) - first);
    auto stage_base = [&](int i) { return (long long)(first + i) * CH; };
    constexpr int RR = TERMS ? k : R;   // rows per ring stage

    int ib = 0;
    auto issue = [&](int i) {   // i-th stage of this warp
        if (i < mine) {
            const long long sb = stage_base(i);
            if (sb + 4 * lane < B) {
                float* buf = ring + ib * (RR * CH) + 4 * lane;
#pragma unroll
                for (int r = 0; r < RR; ++r) cp_async16(buf + r * CH, src[r] + sb);
            }
        }
        cp_async_commit();
        ib = (ib + 1 == kStages) ? 0 : ib + 1;
    };

    // gradient of stages i .. i + kGatherStages - 1 from the upstream terms:
    // lane covers samples 4 lane + 128 u (u < kGatherStages), so one row is
    // read as kGatherStages x 512 contiguous bytes; rows in edge order, from 0
    auto gather = [&](int i) {
        if constexpr (TERMS) {
            float4 g[kGatherStages];
#pragma unroll
            for (int u = 0; u < kGatherStages; ++u) g[u] = make_float4(0.f, 0.f, 0.f, 0.f);
            const long long s0 = stage_base(i) + 4 * lane;
            const int nu = min(kGatherStages, mine - i);
#pragma unroll 2
            for (int q = 0; q < deg; ++q) {
                const int id = q < 32 ? __shfl_sync(0xffffffffu, my_id, q) : term_row(gs, e0 + q);
                if (id >= 0 && (unsigned)id < (unsigned)gs.n_edges) {
                    const float* row = gs.terms + (long long)id * B + s0;
#pragma unroll
                    for (int u = 0; u < kGatherStages; ++u)
                        if (u < nu && s0 + u * CH < B) g[u] = add4(g[u], ldg4(row + u * CH));
                } else if (q >= 32 && lane == 0) {
                    flag_index_error();
                }
            }
#pragma unroll
            for (int u = 0; u < kGatherStages; ++u) {
                const long long s = s0 + u * CH;
                if (u < nu && s < B) {
                    *reinterpret_cast<float4*>(gbuf + u * CH + 4 * lane) = g[u];
                    if (dY_out) *reinterpret_cast<float4*>(dY_out + (long long)jj * B + s) = g[u];
                }
            }
        }
    };

    float acc[H];
#pragma unroll
    for (int a = 0; a < H; ++a) acc[a] = 0.f;

#pragma unroll
    for (int i = 0; i < kStages - 1; ++i) issue(i);
    int rb = 0;
    for (int i = 0; i < mine; ++i) {
        issue(i + kStages - 1);
        const long long sbase = stage_base(i);
        float* buf = ring + rb * (RR * CH);
        if constexpr (TERMS) {
            if (i % kGatherStages == 0) {
                __syncwarp();   // previous readers of gbuf are done
                gather(i);
            }
        } else {
            const long long s4 = sbase + 4 * lane;   // this lane's 16-byte chunk
            if (dY_out && s4 < B)
                *reinterpret_cast<float4*>(dY_out + (long long)jj * B + s4) = ldg4(src[k] + sbase);
        }
        cp_async_wait<kStages - 1>();
        __syncwarp();
        const bool full = sbase + CH <= B;
        const float* rbuf = buf + pair;
        const float* gsrc = TERMS ? gbuf + (i % kGatherStages) * CH + pair : rbuf + k * CH;
        // full stages (all but a ragged last one) compile without range checks
        auto stage = [&](auto full_stage) {
        constexpr bool kFull = decltype(full_stage)::value;
        auto sample = [&](int c) {
            const bool in = kFull || sbase + 16 * c + pair < B;
            float x[k], omx[k], dx[k];
#pragma unroll
            for (int q = 0; q < k; ++q) {
                x[q] = in ? rbuf[q * CH + 16 * c] : 0.f;
                omx[q] = 1.0f - x[q];
            }
            const float g = in ? gsrc[16 * c] : 0.f;
            const float adj = g * (h ? x[k - 1] : omx[k - 1]);
            float v;
            if constexpr (QUADS) {
                const float W[4] = {omx[0] * omx[1], x[0] * omx[1], omx[0] * x[1], x[0] * x[1]};
                v = bwd_tree_quad<k - 2, 0>(cq, x, omx, W, adj, dx, acc);
            } else {
                v = bwd_tree<k - 2, 0>(te, d, x, omx, adj, dx, acc);
            }
            if constexpr (WANT_DX) {
#pragma unroll
                for (int q = 0; q < NQ; ++q) {
                    const int ev = 2 * q, od = 2 * q + 1;   // lane 0 stores ev, lane 1 stores od
                    float send;
                    if (ev == k - 1)      send = v;                      // lane 0 needs v_1
                    else if (od == k - 1) send = h ? dx[ev] : v;         // lane 1 needs v_0
                    else if (od < k)      send = h ? dx[ev] : dx[od];
                    else                  send = dx[ev];
                    const float recv = __shfl_xor_sync(0xffffffffu, send, 1);
                    float full_dx;
                    if (h == 0) full_dx = (ev == k - 1) ? g * (recv - v) : dx[ev] + recv;
                    else        full_dx = (od == k - 1) ? g * (v - recv) : (od < k ? dx[od] + recv : 0.f);
                    if (in && (h == 0 || od < k)) pst[q][sbase + 16 * c] = full_dx;
                }
            }
        };
        if constexpr (kFull) {
#pragma unroll 4
            for (int c = 0; c < CH / 16; ++c) sample(c);
        } else {
#pragma unroll 2
            for (int c = 0; c < CH / 16; ++c) sample(c);
        }
        };
        if (full) stage(std::true_type{});
        else stage(std::false_type{});
        __syncwarp();
        rb = (rb + 1 == kStages) ? 0 : rb + 1;
    }
    cp_async_wait<0>();
    __syncwarp();

    // dtheta: entry a lives in half a / H at offset a % H of the lanes with
    // that parity; sum those 16 lanes, then the node's warps, in a fixed order
    float* red = ring;   // [32][H + 1] per warp
#pragma unroll
    for (int a = 0; a < H; ++a) red[lane * (H + 1) + a] = acc[a];
    __syncthreads();
    if (live && sub == 0 && lane < H) {
        float s0 = 0.f, s1 = 0.f;
        const int a0 = 2 * lane, hh = a0 / H, ao = a0 % H;
#pragma unroll
        for (int q = 0; q < kWarpsPerNode; ++q) {
            const float* rq = smem + (warp + q) * FPW;
#pragma unroll 4
            for (int p = 0; p < 16; ++p) {
                s0 += rq[(2 * p + hh) * (H + 1) + ao];
                s1 += rq[(2 * p + hh) * (H + 1) + ao + 1];
            }
        }
        float* out = dtheta + (long long)j * K + a0;
        out[0] = t0 * (1.0f - t0) * s0;
        out[1] = t1 * (1.0f - t1) * s1;
    }
}

// ------------------------------------- dtheta only, one lane per sample --
//
// Without an input gradient the backward needs no table values:
// dtheta_a = t_a (1 - t_a) sum_s g_s w_a(x_s), w_a the corner weight of
// entry a.  With the slots split into a low half (0 .. kl-1, kl = k/2) and a
// high half, w_a = u(a_lo) v(a_hi): per sample the lane builds U = g times
// the corner weights of the low half and V = the corner weights of the high
// half by doubling products, then adds the outer product U V^T into its 2^k
// accumulators (k = 6: 6 FADD + 14 + 12 FMUL + 64 FFMA = 96 FP32 operations
// per sample, against 190 for the separate corner-weight tree).
//
// Persistent warps: warp g of the grid takes nodes g, g + G, ... (G warps in
// the grid, sized to one wave) over the whole batch, 4 consecutive samples
// per lane in each 128-sample stage.  Its k input rows and gradient row
// stream through a lane-private cp.async ring (a lane reads only the 16
// bytes per row it copied) that runs across node boundaries, so the next
// node's first stages load while the current node finishes.  A node's
// dtheta is reduced inside the warp by a fixed butterfly of shuffles, with
// no block barrier.  Needs B % 4 == 0 and 16-byte aligned X, dY and dY_out.

#ifndef BITLOGIC_THETA_WARPS
#define BITLOGIC_THETA_WARPS 1
#endif
constexpr int kThetaWarps = BITLOGIC_THETA_WARPS;   // warps per block of the dtheta-only kernel
static_assert(kThetaWarps >= 1 && kThetaWarps <= 16, "dtheta-only warps per block");

template <int k>
__host__ __device__ constexpr int theta_floats_per_warp() {
    return kStages * (k + 1) * kStageSamples;
}

// Reduce-scatter of N values per lane over the lane offsets O, O/2, ..., 1:
// at each step a lane keeps half of its values (the upper half when lane bit
// O is set), adds its partner's copy of that half and hands over the other
// half; once one value is left the remaining steps add it across lanes.
// Afterwards, for N0 = 2^k >= 32 values, lane l holds the sums of entries
// l N0/32 .. l N0/32 + N0/32 - 1; for N0 < 32, of entry l >> (5 - k).  The
// order of every addition is fixed.
template <int N, int O, int M>
__device__ __forceinline__ void warp_reduce_scatter(float (&v)[M], int lane) {
    if constexpr (O > 0) {
        if constexpr (N > 1) {
            const bool up = (lane & O) != 0;
#pragma unroll
            for (int i = 0; i < N / 2; ++i) {
                const float send = up ? v[i] : v[i + N / 2];
                const float keep = up ? v[i + N / 2] : v[i];
                v[i] = keep + __shfl_xor_sync(0xffffffffu, send, O);
            }
            warp_reduce_scatter<N / 2, O / 2>(v, lane);
        } else {
            v[0] += __shfl_xor_sync(0xffffffffu, v[0], O);
            warp_reduce_scatter<1, O / 2>(v, lane);
        }
    }
}

template <int k>
__host__ __device__ constexpr int theta_min_blocks() {
    return k <= 3 ? BITLOGIC_BWD_MIN_BLOCKS_SMALL : BITLOGIC_BWD_MIN_BLOCKS;
}

template <int k>
__global__ void __launch_bounds__(kThetaWarps * 32, theta_min_blocks<k>())
lut_backward_theta_kernel(const float* __restrict__ X, int w_in, long long B,
                          const int* __restrict__ conn, const float* __restrict__ theta, int w,
                          const float* __restrict__ dY, int group, float* __restrict__ dtheta,
                          float* __restrict__ dY_out) {
    constexpr int K = 1 << k, KL = k / 2, NU = 1 << KL, NV = 1 << (k - KL), R = k + 1;
    constexpr int CH = kStageSamples;
    extern __shared__ __align__(16) float smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    float* ring = smem + warp * theta_floats_per_warp<k>();
    const int G = gridDim.x * kThetaWarps;
    const int jfirst = blockIdx.x * kThetaWarps + warp;
    const int nst = (int)((B + CH - 1) / CH);

    // issue stream: stage si of node ji, kStages - 1 stages ahead of the
    // compute stream; rows of the warp's node after ji are loaded ahead
    int ji = jfirst, si = 0, ib = 0;
    int ri[k], rn[k];
#pragma unroll
    for (int i = 0; i < k; ++i) ri[i] = rn[i] = 0;
    if (ji < w) load_rows<k>(conn, ji, w_in, lane, ri);
    if (ji + G < w) load_rows<k>(conn, ji + G, w_in, lane, rn);
    auto issue = [&]() {
        if (ji < w) {
            const long long s4 = (long long)si * CH + 4 * lane;
            if (s4 < B) {
                float* buf = ring + ib * (R * CH) + 4 * lane;
#pragma unroll
                for (int r = 0; r < k; ++r) cp_async16(buf + r * CH, X + (long long)ri[r] * B + s4);
                cp_async16(buf + k * CH, dY + (long long)(ji / group) * B + s4);
            }
            if (++si == nst) {
                si = 0;
                ji += G;
#pragma unroll
                for (int i = 0; i < k; ++i) ri[i] = rn[i];
                if (ji + G < w) load_rows<k>(conn, ji + G, w_in, lane, rn);
            }
        }
        cp_async_commit();
        ib = (ib + 1 == kStages) ? 0 : ib + 1;
    };
#pragma unroll 1
    for (int i = 0; i < kStages - 1; ++i) issue();

    int rb = 0;
#pragma unroll 1
    for (int j = jfirst; j < w; j += G) {
        float acc[K];
#pragma unroll
        for (int a = 0; a < K; ++a) acc[a] = 0.f;
#pragma unroll 1
        for (int sc = 0; sc < nst; ++sc) {
            issue();
            cp_async_wait<kStages - 1>();
            const long long s4 = (long long)sc * CH + 4 * lane;   // this lane's 4 samples
            if (s4 < B) {   // B % 4 == 0: all four samples are in range
                const float* buf = ring + rb * (R * CH) + 4 * lane;
                float4 xv[k];
#pragma unroll
                for (int q = 0; q < k; ++q) xv[q] = *reinterpret_cast<const float4*>(buf + q * CH);
                const float4 gv = *reinterpret_cast<const float4*>(buf + k * CH);
                if (dY_out) *reinterpret_cast<float4*>(dY_out + (long long)j * B + s4) = gv;
#pragma unroll
                for (int r = 0; r < 4; ++r) {
                    float x[k], omx[k];
#pragma unroll
                    for (int q = 0; q < k; ++q) {
                        x[q] = comp(xv[q], r);
                        omx[q] = 1.0f - x[q];
                    }
                    float U[NU], V[NV];
                    U[0] = comp(gv, r);
#pragma unroll
                    for (int q = 0; q < KL; ++q) {   // slot q doubles U: index bit q
#pragma unroll
                        for (int m = 0; m < (1 << q); ++m) {
                            U[m + (1 << q)] = U[m] * x[q];
                            U[m] = U[m] * omx[q];
                        }
                    }
                    V[0] = omx[KL];
                    V[1] = x[KL];
#pragma unroll
                    for (int q = KL + 1; q < k; ++q) {   // slot q doubles V: index bit q - KL
#pragma unroll
                        for (int m = 0; m < (1 << (q - KL)); ++m) {
                            V[m + (1 << (q - KL))] = V[m] * x[q];
                            V[m] = V[m] * omx[q];
                        }
                    }
#pragma unroll
                    for (int b = 0; b < NV; ++b)
#pragma unroll
                        for (int a = 0; a < NU; ++a) acc[a + b * NU] = fmaf(U[a], V[b], acc[a + b * NU]);
                }
            }
            rb = (rb + 1 == kStages) ? 0 : rb + 1;
        }
        // the node's dtheta: butterfly over the lanes, then t (1 - t)
        warp_reduce_scatter<K, 16>(acc, lane);
        constexpr int NF = K >= 32 ? K / 32 : 1;   // entries per lane
        constexpr int SH = K >= 32 ? 0 : 5 - k;    // lanes sharing an entry (K < 32)
        if ((lane & ((1 << SH) - 1)) == 0) {
#pragma unroll
            for (int i = 0; i < NF; ++i) {
                const int a = K >= 32 ? lane * NF + i : lane >> SH;
                const float t = sigmoidf(__ldg(theta + (long long)j * K + a));
                dtheta[(long long)j * K + a] = t * (1.0f - t) * acc[i];
            }
        }
    }
    cp_async_wait<0>();
}

// dX[i][s] = sum over the CSR positions p of input i (increasing p) of
// P[edge[p]][s].  One block per input row i (and batch slice); warp r of the
// block owns 128 samples (vector path: 4 per lane) or 32 (scalar path) and
// issues the loads of all of the row's terms back to back, so each warp has
// deg x 512 bytes in flight.  The row's ids are read once, one per lane.
constexpr int kCsrWarps = 8;

template <bool VEC>
__global__ void __launch_bounds__(kCsrWarps * 32)
csr_reduce_kernel(const float* __restrict__ P, long long B, const int* __restrict__ off,
                  const int* __restrict__ edge, int w_in, int nE, float* __restrict__ dX) {
    constexpr int SPW = VEC ? 128 : 32;   // samples per warp
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int i = blockIdx.x;
    int e0 = __ldg(off + i), e1 = __ldg(off + i + 1);
    if (e0 < 0 || e1 < e0 || e1 > nE) {
        if (threadIdx.x == 0) flag_index_error();
        e0 = e1 = 0;
    }
    const int deg = e1 - e0;
    int my_id = -1;   // ids of the first 32 positions, -1 when out of range
    if (lane < deg) {
        my_id = edge ? __ldg(edge + e0 + lane) : e0 + lane;
        if ((unsigned)my_id >= (unsigned)nE) {
            if (warp == 0) flag_index_error();
            my_id = -1;
        }
    }
    auto edge_id = [&](int q) {   // warp-uniform call
        if (q < 32) return __shfl_sync(0xffffffffu, my_id, q);
        const int id = edge ? __ldg(edge + e0 + q) : e0 + q;
        if ((unsigned)id >= (unsigned)nE) {
            if (lane == 0 && warp == 0) flag_index_error();
            return -1;
        }
        return id;
    };
    const long long s = ((long long)blockIdx.y * kCsrWarps + warp) * SPW + (VEC ? 4 : 1) * lane;
    const bool in = s < B;   // vector path: B % 4 == 0, all four samples in range
    float* out = dX + (long long)i * B + s;
    // loads of up to kCsrBatch rows are issued before the first add; the
    // adds keep increasing position order
    constexpr int kCsrBatch = 8;
    if constexpr (VEC) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        for (int q0 = 0; q0 < deg; q0 += kCsrBatch) {
            float4 v[kCsrBatch];
#pragma unroll
            for (int u = 0; u < kCsrBatch; ++u) {
                const int id = q0 + u < deg ? edge_id(q0 + u) : -1;   // warp-uniform condition
                v[u] = (in && id >= 0) ? ldg4(P + (long long)id * B + s) : make_float4(0.f, 0.f, 0.f, 0.f);
            }
#pragma unroll
            for (int u = 0; u < kCsrBatch; ++u)
                if (q0 + u < deg) acc = add4(acc, v[u]);
        }
        if (in) *reinterpret_cast<float4*>(out) = acc;
    } else {
        float acc = 0.f;
        for (int q0 = 0; q0 < deg; q0 += kCsrBatch) {
            float v[kCsrBatch];
#pragma unroll
            for (int u = 0; u < kCsrBatch; ++u) {
                const int id = q0 + u < deg ? edge_id(q0 + u) : -1;
                v[u] = (in && id >= 0) ? __ldg(P + (long long)id * B + s) : 0.f;
            }
#pragma unroll
            for (int u = 0; u < kCsrBatch; ++u)
                if (q0 + u < deg) acc += v[u];
        }
        if (in) *out = acc;
    }
}

// ----------------------------------------------------------- launchers --

// Samples per forward work item (node x batch slice): a warp keeps a node
// over the whole batch (the per-node set-up, the sigmoids and Moebius
// coefficients, is paid once) unless that leaves fewer than about
// BITLOGIC_FWD_WAVES waves of warps; the slices keep at least
// BITLOGIC_FWD_MIN_CHUNK samples.
long long forward_chunk(int w_in, int w, long long B) {
    (void)w_in;
    const long long items_wanted = (long long)BITLOGIC_FWD_WAVES * sm_count() * 16;
    long long c = (long long)w * B / items_wanted;
    c = (c / 128) * 128;
    if (c < BITLOGIC_FWD_MIN_CHUNK) c = BITLOGIC_FWD_MIN_CHUNK;
    return c < B ? c : B;
}

template <int k>
int launch_forward(const float* X, int w_in, long long B, const int* conn, const float* theta,
                   int w, int node, float* Y, bool vec, cudaStream_t st) {
    long long chunk = forward_chunk(w_in, w, B);
    if (vec) chunk = (chunk + 3) / 4 * 4;
    const long long ny = (B + chunk - 1) / chunk;
    if (ny > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((w + kFwdWarps - 1) / kFwdWarps), (unsigned)ny);
    if (vec)
        lut_forward_staged_kernel<k><<<grid, kFwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, node, Y, chunk);
    else
        lut_forward_kernel<k><<<grid, kFwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, node, Y, chunk);
    return launch_status();
}

template <int k, bool WANT_DX, bool TERMS>
int launch_backward_impl(const float* X, int w_in, long long B, const int* conn, const float* theta,
                         int w, int node, const GradSource& gs, float* dtheta, float* P, const int* epos,
                         float* dY_out, bool staged, cudaStream_t st) {
    if constexpr (k >= 2) {
        if (staged) {
            constexpr size_t smem = node_smem_bytes<k, TERMS>();
            // term rows at caller-given positions: a separate instantiation,
            // so the common form compiles without the position lookups
            auto kern = (WANT_DX && epos) ? lut_backward_node_kernel<k, WANT_DX, TERMS, WANT_DX>
                                          : lut_backward_node_kernel<k, WANT_DX, TERMS, false>;
            if (smem > 48 * 1024 &&
                cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
                return BITLOGIC_ERR_CUDA;
            kern<<<(unsigned)((w + kNodesPerBlock - 1) / kNodesPerBlock), kBwdWarps * 32, smem, st>>>(
                X, w_in, B, conn, theta, w, node, gs, dtheta, P, epos, dY_out);
            return launch_status();
        }
    }
    dim3 grid((unsigned)((w + kFwdWarps - 1) / kFwdWarps));
    lut_backward_kernel<k, WANT_DX, TERMS><<<grid, kFwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, node,
                                                                            gs, dtheta, P, epos, dY_out);
    return launch_status();
}

template <int k>
int launch_backward(const float* X, int w_in, long long B, const int* conn, const float* theta,
                    int w, int node, const GradSource& gs, float* dtheta, float* P, const int* epos,
                    float* dY_out, cudaStream_t st) {
    const bool terms = gs.terms != nullptr;
    const bool staged = (B % 4 == 0) && aligned16(X) && aligned16(terms ? gs.terms : gs.dY) &&
                        (!dY_out || aligned16(dY_out)) && (!P || aligned16(P));
    // dtheta only, from dY rows: the table entries are not needed, so both
    // node forms run the same kernel
    if (staged && !P && !terms) {
        constexpr size_t smem = (size_t)kThetaWarps * theta_floats_per_warp<k>() * sizeof(float);
        auto kern = lut_backward_theta_kernel<k>;
        if (smem > 40 * 1024 &&
            cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
            return BITLOGIC_ERR_CUDA;
        // one wave of persistent warps filling every SM alike (nodes dealt
        // round-robin, so warps differ by at most one node)
        const long long resident = (long long)sm_count() * theta_min_blocks<k>() * kThetaWarps;
        const long long warps = w < resident ? w : resident;
        kern<<<(unsigned)((warps + kThetaWarps - 1) / kThetaWarps), kThetaWarps * 32, smem, st>>>(
            X, w_in, B, conn, theta, w, gs.dY, gs.group, dtheta, dY_out);
        return launch_status();
    }
    if (P) {
        return terms ? launch_backward_impl<k, true, true>(X, w_in, B, conn, theta, w, node, gs, dtheta, P, epos, dY_out,
                                                           staged, st)
                     : launch_backward_impl<k, true, false>(X, w_in, B, conn, theta, w, node, gs, dtheta, P, epos, dY_out,
                                                            staged, st);
    }
    return terms ? launch_backward_impl<k, false, true>(X, w_in, B, conn, theta, w, node, gs, dtheta, P, epos, dY_out,
                                                        staged, st)
                 : launch_backward_impl<k, false, false>(X, w_in, B, conn, theta, w, node, gs, dtheta, P, epos, dY_out,
                                                         staged, st);
}

int check_layer(const void* X, int32_t w_in, int64_t B, const void* conn, const void* theta,
                int32_t w, int32_t k) {
    if (!conn || !theta) return BITLOGIC_ERR_NULL;
    if (B > 0 && !X) return BITLOGIC_ERR_NULL;   // an empty batch may come as NULL
    if (w_in <= 0 || w <= 0 || B < 0) return BITLOGIC_ERR_SHAPE;
    if (k < 1 || k > 6 || k > w_in) return BITLOGIC_ERR_FANIN;
    if ((int64_t)w * k > 0x7fffffffLL) return BITLOGIC_ERR_SHAPE;
    return BITLOGIC_OK;
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(lut_soft)

extern "C" int bitlogic_lut_forward_node(const float* X, int32_t w_in, int64_t B,
                                         const int32_t* conn, const float* theta,
                                         int32_t w, int32_t k, int32_t node, float* Y,
                                         cudaStream_t stream) {
    int st = check_layer(X, w_in, B, conn, theta, w, k);
    if (st) return st;
    if (node != BITLOGIC_NODE_SOFT && node != BITLOGIC_NODE_ST) return BITLOGIC_ERR_NODE;
    if (B == 0) return BITLOGIC_OK;
    if (!Y) return BITLOGIC_ERR_NULL;
    const bool vec = (B % 4 == 0) && aligned16(X) && aligned16(Y);
    switch (k) {
        case 1: return launch_forward<1>(X, w_in, B, conn, theta, w, node, Y, vec, stream);
        case 2: return launch_forward<2>(X, w_in, B, conn, theta, w, node, Y, vec, stream);
        case 3: return launch_forward<3>(X, w_in, B, conn, theta, w, node, Y, vec, stream);
        case 4: return launch_forward<4>(X, w_in, B, conn, theta, w, node, Y, vec, stream);
        case 5: return launch_forward<5>(X, w_in, B, conn, theta, w, node, Y, vec, stream);
        default: return launch_forward<6>(X, w_in, B, conn, theta, w, node, Y, vec, stream);
    }
}

extern "C" int bitlogic_lut_forward(const float* X, int32_t w_in, int64_t B,
                                    const int32_t* conn, const float* theta,
                                    int32_t w, int32_t k, float* Y, cudaStream_t stream) {
    return bitlogic_lut_forward_node(X, w_in, B, conn, theta, w, k, BITLOGIC_NODE_SOFT, Y, stream);
}

extern "C" size_t bitlogic_lut_backward_workspace(int32_t w_in, int64_t B, int32_t w,
                                                  int32_t k, int32_t want_dx) {
    (void)w_in;
    if (!want_dx || B <= 0 || w <= 0 || k <= 0) return 0;
    return (size_t)w * (size_t)k * (size_t)B * sizeof(float);
}

extern "C" int bitlogic_lut_backward_node(const float* X, int32_t w_in, int64_t B,
                                          const int32_t* conn, const float* theta,
                                          int32_t w, int32_t k, int32_t node,
                                          const float* dY, int32_t dy_group,
                                          const float* up_terms, const int32_t* up_off,
                                          const int32_t* up_edge, int32_t up_edges,
                                          float* dtheta, float* edge_terms, const int32_t* edge_pos,
                                          float* dY_out, cudaStream_t stream) {
    int st = check_layer(X, w_in, B, conn, theta, w, k);
    if (st) return st;
    if (node != BITLOGIC_NODE_SOFT && node != BITLOGIC_NODE_ST) return BITLOGIC_ERR_NODE;
    if (!dtheta) return BITLOGIC_ERR_NULL;
    const bool terms = up_terms != nullptr;
    if (B > 0 && terms == (dY != nullptr)) return BITLOGIC_ERR_NULL;   // exactly one source
    if (terms) {
        if (!up_off) return BITLOGIC_ERR_NULL;   // up_edge NULL: terms in CSR order
        if (up_edges < 0) return BITLOGIC_ERR_SHAPE;
    } else if (dy_group < 1 || dy_group > w) {
        return BITLOGIC_ERR_SHAPE;
    }
    if (B == 0) {
        // empty batch: the batch sums are zero
        if (cudaMemsetAsync(dtheta, 0, sizeof(float) * (size_t)w * ((size_t)1 << k), stream) != cudaSuccess)
            return BITLOGIC_ERR_CUDA;
        return BITLOGIC_OK;
    }
    GradSource gs{dY, dy_group, up_terms, up_off, up_edge, up_edges};
    switch (k) {
        case 1: return launch_backward<1>(X, w_in, B, conn, theta, w, node, gs, dtheta, edge_terms, edge_pos, dY_out, stream);
        case 2: return launch_backward<2>(X, w_in, B, conn, theta, w, node, gs, dtheta, edge_terms, edge_pos, dY_out, stream);
        case 3: return launch_backward<3>(X, w_in, B, conn, theta, w, node, gs, dtheta, edge_terms, edge_pos, dY_out, stream);
        case 4: return launch_backward<4>(X, w_in, B, conn, theta, w, node, gs, dtheta, edge_terms, edge_pos, dY_out, stream);
        case 5: return launch_backward<5>(X, w_in, B, conn, theta, w, node, gs, dtheta, edge_terms, edge_pos, dY_out, stream);
        default: return launch_backward<6>(X, w_in, B, conn, theta, w, node, gs, dtheta, edge_terms, edge_pos, dY_out, stream);
    }
}

extern "C" int bitlogic_lut_backward_ex(const float* X, int32_t w_in, int64_t B,
                                        const int32_t* conn, const float* theta,
                                        int32_t w, int32_t k,
                                        const float* dY, int32_t dy_group,
                                        const float* up_terms, const int32_t* up_off,
                                        const int32_t* up_edge, int32_t up_edges,
                                        float* dtheta, float* edge_terms, const int32_t* edge_pos,
                                        float* dY_out, cudaStream_t stream) {
    return bitlogic_lut_backward_node(X, w_in, B, conn, theta, w, k, BITLOGIC_NODE_SOFT, dY, dy_group,
                                      up_terms, up_off, up_edge, up_edges, dtheta, edge_terms, edge_pos,
                                      dY_out, stream);
}

extern "C" int bitlogic_lut_backward_edges(const float* X, int32_t w_in, int64_t B,
                                           const int32_t* conn, const float* theta,
                                           int32_t w, int32_t k, const float* dY,
                                           float* dtheta, float* edge_terms,
                                           cudaStream_t stream) {
    if (B > 0 && !dY) return BITLOGIC_ERR_NULL;
    return bitlogic_lut_backward_ex(X, w_in, B, conn, theta, w, k, dY, 1,
                                    nullptr, nullptr, nullptr, 0, dtheta, edge_terms, nullptr, nullptr, stream);
}

extern "C" int bitlogic_csr_reduce(const float* edge_terms, int64_t B, const int32_t* csr_off,
                                   const int32_t* csr_edge, int32_t w_in, int32_t n_edges,
                                   float* dX, cudaStream_t stream) {
    if (B < 0 || w_in <= 0 || n_edges < 0) return BITLOGIC_ERR_SHAPE;
    if (B == 0) return BITLOGIC_OK;
    if (!edge_terms || !csr_off || !dX) return BITLOGIC_ERR_NULL;   // csr_edge NULL: terms in CSR order
    const bool vec = (B % 4 == 0) && aligned16(edge_terms) && aligned16(dX);
    const long long per_block = (long long)kCsrWarps * (vec ? 128 : 32);
    const long long gy = (B + per_block - 1) / per_block;
    if (gy > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)w_in, (unsigned)gy);
    if (vec)
        csr_reduce_kernel<true><<<grid, kCsrWarps * 32, 0, stream>>>(edge_terms, B, csr_off, csr_edge, w_in, n_edges, dX);
    else
        csr_reduce_kernel<false><<<grid, kCsrWarps * 32, 0, stream>>>(edge_terms, B, csr_off, csr_edge, w_in, n_edges, dX);
    return launch_status();
}

extern "C" int bitlogic_lut_backward(const float* X, int32_t w_in, int64_t B,
                                     const int32_t* conn, const float* theta,
                                     int32_t w, int32_t k, const float* dY,
                                     const int32_t* csr_off, const int32_t* csr_edge,
                                     float* dtheta, float* dX,
                                     void* workspace, size_t ws_bytes, cudaStream_t stream) {
    int st = check_layer(X, w_in, B, conn, theta, w, k);
    if (st) return st;
    if (!dtheta || (B > 0 && !dY)) return BITLOGIC_ERR_NULL;
    const bool want_dx = dX != nullptr && B > 0;
    if (want_dx) {
        if (!csr_off || !csr_edge) return BITLOGIC_ERR_NULL;
        if (!workspace) return BITLOGIC_ERR_NULL;
        if (!aligned16(workspace)) return BITLOGIC_ERR_ALIGN;
        if (ws_bytes < bitlogic_lut_backward_workspace(w_in, B, w, k, 1)) return BITLOGIC_ERR_WORKSPACE;
    }
    float* P = want_dx ? static_cast<float*>(workspace) : nullptr;
    st = bitlogic_lut_backward_edges(X, w_in, B, conn, theta, w, k, dY, dtheta, P, stream);
    if (st || !want_dx) return st;
    return bitlogic_csr_reduce(P, B, csr_off, csr_edge, w_in, w * k, dX, stream);
}
