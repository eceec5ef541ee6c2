// Soft (training) forward and backward of a fixed-connectivity LUT layer.
//
// Node (LightLUT, §2 of the paper: Kronecker-indicator basis, 2^k logits per
// node), read as t = sigmoid(theta), y = sum_a t_a prod_i x_i^{a_i}(1-x_i)^{1-a_i}
// with connectivity slot i = bit i of the table index a.
//
// Evaluation: the multilinear form is a complete binary lerp tree over the
// k inputs (level l interpolates with x_l), 2^k - 1 lerps per (node, sample).
// Level 0 uses per-node constants (t_even, t_odd - t_even), so it costs one
// FFMA per lerp; every other lerp is one FADD and one FFMA.  The backward is
// reverse mode through the same tree: the adjoint of each subtree is pushed
// down (two FMULs per lerp), each lerp adds adjoint * (hi - lo) into dx_l, and
// at the leaves the adjoint is g * w_a, accumulated for dtheta.
//
// Work split: one warp per node, lanes over samples (batch-contiguous rows,
// so every gathered row segment is a coalesced 128/512-byte access).  The
// table lives in registers for the whole sweep of the node.
#include "common.cuh"

namespace bitlogic {
namespace {

constexpr int kFwdWarps = 4;
constexpr int kBwdWarps = 4;
constexpr int kCsrWarps = 8;

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

// Returns the subtree value; `adj` is the adjoint of this subtree's output.
template <int L, int M, int H, int K, int k>
__device__ __forceinline__ float bwd_tree(const float (&te)[H], const float (&d)[H],
                                          const float (&x)[k], const float (&omx)[k],
                                          float adj, float (&dx)[k], float (&acc)[K]) {
    if constexpr (L == 0) {
        dx[0] = fmaf(adj, d[M], dx[0]);
        acc[2 * M] = fmaf(adj, omx[0], acc[2 * M]);
        acc[2 * M + 1] = fmaf(adj, x[0], acc[2 * M + 1]);
        return fmaf(x[0], d[M], te[M]);
    } else {
        const float lo = bwd_tree<L - 1, 2 * M>(te, d, x, omx, adj * omx[L], dx, acc);
        const float hi = bwd_tree<L - 1, 2 * M + 1>(te, d, x, omx, adj * x[L], dx, acc);
        const float diff = hi - lo;
        dx[L] = fmaf(adj, diff, dx[L]);
        return fmaf(x[L], diff, lo);
    }
}

__device__ __forceinline__ float comp(const float4& v, int c) {
    return c == 0 ? v.x : c == 1 ? v.y : c == 2 ? v.z : v.w;
}

__device__ __forceinline__ float4 ldg4(const float* p) {
    return __ldg(reinterpret_cast<const float4*>(p));
}

// Per-warp node set-up: connectivity rows (range-checked), sigmoid of the
// table logits, level-0 constants broadcast to every lane through shared
// memory.  Lane l (l < 2^(k-1)) keeps t[2l] and t[2l+1] for the dtheta
// epilogue.
template <int k>
__device__ __forceinline__ void node_setup(const int* __restrict__ conn,
                                           const float* __restrict__ theta, int j, int w_in,
                                           int lane, float2* sPair, int (&rows)[k],
                                           float (&te)[1 << (k - 1)], float (&d)[1 << (k - 1)],
                                           float& t0, float& t1) {
    constexpr int K = 1 << k, H = K / 2;
    bool bad = false;
#pragma unroll
    for (int i = 0; i < k; ++i) {
        int c = __ldg(conn + (long long)j * k + i);
        if ((unsigned)c >= (unsigned)w_in) { bad = true; c = 0; }
        rows[i] = c;
    }
    if (bad && lane == 0) flag_index_error();
    t0 = t1 = 0.f;
    if (lane < H) {
        t0 = sigmoidf(__ldg(theta + (long long)j * K + 2 * lane));
        t1 = sigmoidf(__ldg(theta + (long long)j * K + 2 * lane + 1));
        sPair[lane] = make_float2(t0, t1 - t0);
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

// ---------------------------------------------------- async copy helpers --

// Asynchronous 16-byte global -> shared copies (L2 only), grouped per stage.
__device__ __forceinline__ void cp_async16(void* smem, const void* gmem) {
    const unsigned s = (unsigned)__cvta_generic_to_shared(smem);
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16;\n" ::"r"(s), "l"(gmem) : "memory");
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;\n" ::: "memory"); }
template <int N>
__device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;\n" ::"n"(N) : "memory"); }

constexpr int kStageSamples = 128;   // samples per pipeline stage
constexpr int kStages = 3;           // stages in flight per warp

// ------------------------------------------------------------- forward --

template <int k, bool VEC>
__global__ void __launch_bounds__(kFwdWarps * 32)
lut_forward_kernel(const float* __restrict__ X, int w_in, long long B,
                   const int* __restrict__ conn, const float* __restrict__ theta, int w,
                   float* __restrict__ Y, long long chunk) {
    constexpr int H = 1 << (k - 1);
    __shared__ float2 sPair[kFwdWarps][H];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kFwdWarps + warp;
    if (j >= w) return;
    int rows[k];
    float te[H], d[H], t0, t1;
    node_setup<k>(conn, theta, j, w_in, lane, sPair[warp], rows, te, d, t0, t1);

    const long long s0 = (long long)blockIdx.y * chunk;
    const long long s1 = min(B, s0 + chunk);
    const float* xr[k];
#pragma unroll
    for (int i = 0; i < k; ++i) xr[i] = X + (long long)rows[i] * B;
    float* yr = Y + (long long)j * B;

    if constexpr (VEC) {
        // B % 4 == 0 and chunk % 4 == 0: every float4 is in range
        for (long long s = s0 + 4 * lane; s < s1; s += 128) {
            float4 xv[k];
#pragma unroll
            for (int i = 0; i < k; ++i) xv[i] = ldg4(xr[i] + s);
            float o[4];
#pragma unroll
            for (int c = 0; c < 4; ++c) {
                float x[k];
#pragma unroll
                for (int i = 0; i < k; ++i) x[i] = comp(xv[i], c);
                o[c] = fwd_tree<k - 1, 0>(te, d, x);
            }
            *reinterpret_cast<float4*>(yr + s) = make_float4(o[0], o[1], o[2], o[3]);
        }
    } else {
        for (long long s = s0 + lane; s < s1; s += 32) {
            float x[k];
#pragma unroll
            for (int i = 0; i < k; ++i) x[i] = __ldg(xr[i] + s);
            yr[s] = fwd_tree<k - 1, 0>(te, d, x);
        }
    }
}

// Forward with the k gathered input rows streamed through a ring of
// shared-memory stages (cp.async).  Each lane copies, reads back and
// evaluates its own 4 consecutive samples of a stage (16-byte chunks), so
// the ring needs no warp synchronisation.  The block's y index selects a
// batch slice (see forward_chunk).  Needs B % 4 == 0, chunk % 4 == 0 and
// 16-byte aligned X and Y.
template <int k>
__global__ void __launch_bounds__(kFwdWarps * 32)
lut_forward_staged_kernel(const float* __restrict__ X, int w_in, long long B,
                          const int* __restrict__ conn, const float* __restrict__ theta, int w,
                          float* __restrict__ Y, long long chunk) {
    constexpr int H = 1 << (k - 1), CH = kStageSamples;
    __shared__ __align__(16) float sRing[kFwdWarps][kStages * k * CH];
    __shared__ float2 sPair[kFwdWarps][H];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kFwdWarps + warp;
    if (j >= w) return;
    int rows[k];
    float te[H], d[H], t0, t1;
    node_setup<k>(conn, theta, j, w_in, lane, sPair[warp], rows, te, d, t0, t1);
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
                o[c] = fwd_tree<k - 1, 0>(te, d, x);
            }
            *reinterpret_cast<float4*>(yr + (long long)st * CH) = make_float4(o[0], o[1], o[2], o[3]);
        }
        rb = (rb + 1 == kStages) ? 0 : rb + 1;
    }
    cp_async_wait<0>();
}

// ------------------------------------------------------------ backward --

template <int k, bool WANT_DX>
__global__ void __launch_bounds__(kBwdWarps * 32)
lut_backward_kernel(const float* __restrict__ X, int w_in, long long B,
                    const int* __restrict__ conn, const float* __restrict__ theta, int w,
                    const float* __restrict__ dY, float* __restrict__ dtheta,
                    float* __restrict__ P) {
    constexpr int K = 1 << k, H = K / 2;
    __shared__ float2 sPair[kBwdWarps][H];
    __shared__ float sRed[kBwdWarps][32][K + 1];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kBwdWarps + warp;
    if (j >= w) return;
    int rows[k];
    float te[H], d[H], t0, t1;
    node_setup<k>(conn, theta, j, w_in, lane, sPair[warp], rows, te, d, t0, t1);

    const float* gr = dY + (long long)j * B;
    float* pr = P + (long long)j * k * B;   // rows j*k + i of the per-edge terms

    float acc[K];
#pragma unroll
    for (int a = 0; a < K; ++a) acc[a] = 0.f;

    // one sample per lane per step (coalesced 128-byte rows), with the next
    // step's gathers issued before this step's tree
    float xn[k], gn = 0.f;
    if (lane < B) {
#pragma unroll
        for (int i = 0; i < k; ++i) xn[i] = __ldg(X + (long long)rows[i] * B + lane);
        gn = __ldg(gr + lane);
    }
    for (long long s = lane; s < B; s += 32) {
        float x[k], omx[k], dx[k];
        const float g = gn;
#pragma unroll
        for (int i = 0; i < k; ++i) {
            x[i] = xn[i];
            omx[i] = 1.0f - x[i];
            dx[i] = 0.f;
        }
        if (s + 32 < B) {
#pragma unroll
            for (int i = 0; i < k; ++i) xn[i] = __ldg(X + (long long)rows[i] * B + s + 32);
            gn = __ldg(gr + s + 32);
        }
        bwd_tree<k - 1, 0>(te, d, x, omx, g, dx, acc);
        if constexpr (WANT_DX) {
#pragma unroll
            for (int i = 0; i < k; ++i) pr[(long long)i * B + s] = dx[i];
        }
    }

    // dtheta: sum the per-lane partials over the 32 lanes in lane order
    // (transpose through shared memory), then scale by t (1 - t).
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

// ---------------------------------------- backward, shared-memory staged --

template <int k>
__host__ __device__ constexpr int staged_floats_per_warp() {
    constexpr int rows = kStages * (k + 1) * kStageSamples;
    constexpr int red = 32 * ((1 << (k - 1)) + 1);
    return rows > red ? rows : red;
}

template <int k>
constexpr size_t staged_smem_bytes() {
    return (size_t)kBwdWarps * staged_floats_per_warp<k>() * sizeof(float) +
           (size_t)kBwdWarps * (1 << (k - 1)) * sizeof(float2);
}

// Backward with two lanes per sample: lane h = lane & 1 owns the half of
// the table whose top input x_{k-1} equals h, i.e. one of the two subtrees
// under the root lerp.  Each lane runs the reverse tree of its subtree
// (adjoint g * (h ? x_{k-1} : 1 - x_{k-1})), accumulates the leaf adjoints of
// its half for dtheta, and the pair exchanges three values by shuffle: the
// partial dx_i of the slots the partner stores, and the subtree value that
// gives dx_{k-1} = g * (v_1 - v_0).  Lane h stores the slots i with
// i % 2 == h.  Halving the per-thread table and accumulators doubles the
// resident warps.  The k gathered rows and the dY row stream through a
// kStages-deep cp.async ring as 16-byte chunks (each lane copies one chunk
// per row; the pair partners read them after a warp sync).  Needs k >= 2,
// B % 4 == 0 and 16-byte aligned X and dY.
template <int k, bool WANT_DX>
__global__ void __launch_bounds__(kBwdWarps * 32)
lut_backward_staged_kernel(const float* __restrict__ X, int w_in, long long B,
                           const int* __restrict__ conn, const float* __restrict__ theta, int w,
                           const float* __restrict__ dY, float* __restrict__ dtheta,
                           float* __restrict__ P) {
    constexpr int K = 1 << k, H = K / 2, H2 = K / 4, R = k + 1, CH = kStageSamples;
    constexpr int NQ = (k + 1) / 2;   // slots stored per lane (rounded up)
    extern __shared__ __align__(16) float smem[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int h = lane & 1, pair = lane >> 1;
    float* ring = smem + warp * staged_floats_per_warp<k>();
    float2* sPair = reinterpret_cast<float2*>(smem + kBwdWarps * staged_floats_per_warp<k>()) + warp * H;
    const int j = blockIdx.x * kBwdWarps + warp;
    if (j >= w) return;

    int rows[k];
    bool bad = false;
#pragma unroll
    for (int i = 0; i < k; ++i) {
        int c = __ldg(conn + (long long)j * k + i);
        if ((unsigned)c >= (unsigned)w_in) { bad = true; c = 0; }
        rows[i] = c;
    }
    if (bad && lane == 0) flag_index_error();
    float t0 = 0.f, t1 = 0.f;
    if (lane < H) {
        t0 = sigmoidf(__ldg(theta + (long long)j * K + 2 * lane));
        t1 = sigmoidf(__ldg(theta + (long long)j * K + 2 * lane + 1));
        sPair[lane] = make_float2(t0, t1 - t0);
    }
    __syncwarp();
    float te[H2], d[H2];
#pragma unroll
    for (int m = 0; m < H2; ++m) {
        const float2 v = sPair[h * H2 + m];
        te[m] = v.x;
        d[m] = v.y;
    }
    __syncwarp();

    const float* src[R];
#pragma unroll
    for (int i = 0; i < k; ++i) src[i] = X + (long long)rows[i] * B + 4 * lane;
    src[k] = dY + (long long)j * B + 4 * lane;
    float* pst[NQ];   // this lane's stored slots 2q + h, at its first sample
#pragma unroll
    for (int q = 0; q < NQ; ++q) pst[q] = P + ((long long)j * k + (2 * q + h < k ? 2 * q + h : 0)) * B + pair;
    const int nst = (int)((B + CH - 1) / CH);

    int ib = 0;
    auto issue = [&](int st) {
        if (st < nst && (long long)st * CH + 4 * lane < B) {
            float* buf = ring + ib * (R * CH) + 4 * lane;
#pragma unroll
            for (int r = 0; r < R; ++r) cp_async16(buf + r * CH, src[r] + (long long)st * CH);
        }
        cp_async_commit();
        ib = (ib + 1 == kStages) ? 0 : ib + 1;
    };

    float acc[H];
#pragma unroll
    for (int a = 0; a < H; ++a) acc[a] = 0.f;

#pragma unroll
    for (int st = 0; st < kStages - 1; ++st) issue(st);
    int rb = 0;
    for (int st = 0; st < nst; ++st) {
        issue(st + kStages - 1);
        cp_async_wait<kStages - 1>();
        __syncwarp();
        const float* buf = ring + rb * (R * CH) + pair;
        const long long sbase = (long long)st * CH;
#pragma unroll 2
        for (int c = 0; c < CH / 16; ++c) {
            const bool in = sbase + 16 * c + pair < B;
            float x[k], omx[k], dx[k];
#pragma unroll
            for (int i = 0; i < k; ++i) {
                x[i] = in ? buf[i * CH + 16 * c] : 0.f;
                omx[i] = 1.0f - x[i];
                dx[i] = 0.f;
            }
            const float g = in ? buf[k * CH + 16 * c] : 0.f;
            const float adj = g * (h ? x[k - 1] : omx[k - 1]);
            const float v = bwd_tree<k - 2, 0>(te, d, x, omx, adj, dx, acc);
            if constexpr (WANT_DX) {
#pragma unroll
                for (int q = 0; q < NQ; ++q) {
                    const int e = 2 * q, o = 2 * q + 1;   // lane 0 stores e, lane 1 stores o
                    // what the partner needs from this lane
                    float send;
                    if (e == k - 1)      send = v;                    // lane 0 needs v_1
                    else if (o == k - 1) send = h ? dx[e] : v;        // lane 1 needs v_0
                    else if (o < k)      send = h ? dx[e] : dx[o];
                    else                 send = dx[e];
                    const float recv = __shfl_xor_sync(0xffffffffu, send, 1);
                    float full;
                    if (h == 0) full = (e == k - 1) ? g * (recv - v) : dx[e] + recv;
                    else        full = (o == k - 1) ? g * (v - recv) : (o < k ? dx[o] + recv : 0.f);
                    if (in && (h == 0 || o < k)) pst[q][sbase + 16 * c] = full;
                }
            }
        }
        __syncwarp();
        rb = (rb + 1 == kStages) ? 0 : rb + 1;
    }
    cp_async_wait<0>();
    __syncwarp();

    // dtheta: entry a lives in half a / H at offset a % H of the lanes with
    // that parity; sum those 16 lanes in lane order through the ring
    float* red = ring;   // [32][H + 1]
#pragma unroll
    for (int a = 0; a < H; ++a) red[lane * (H + 1) + a] = acc[a];
    __syncwarp();
    if (lane < H) {
        float s0 = 0.f, s1 = 0.f;
        const int a0 = 2 * lane, hh = a0 / H, ao = a0 % H;
#pragma unroll 4
        for (int p = 0; p < 16; ++p) {
            s0 += red[(2 * p + hh) * (H + 1) + ao];
            s1 += red[(2 * p + hh) * (H + 1) + ao + 1];
        }
        float* out = dtheta + (long long)j * K + a0;
        out[0] = t0 * (1.0f - t0) * s0;
        out[1] = t1 * (1.0f - t1) * s1;
    }
}

// dX[i][s] = sum over the CSR edges of input i (increasing edge id) of
// P[edge][s].  One warp per input row, lanes over samples.
template <bool VEC>
__global__ void __launch_bounds__(kCsrWarps * 32)
csr_reduce_kernel(const float* __restrict__ P, long long B, const int* __restrict__ off,
                  const int* __restrict__ edge, int w_in, int nE, float* __restrict__ dX) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int i = blockIdx.x * kCsrWarps + warp;
    if (i >= w_in) return;
    int e0 = __ldg(off + i), e1 = __ldg(off + i + 1);
    if (e0 < 0 || e1 < e0 || e1 > nE) {
        if (lane == 0) flag_index_error();
        e0 = e1 = 0;
    }
    float* out = dX + (long long)i * B;
    if constexpr (VEC) {
        for (long long base = 0; base < B; base += 512) {
            float4 acc[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) acc[q] = make_float4(0.f, 0.f, 0.f, 0.f);
            for (int e = e0; e < e1; ++e) {
                int eid = __ldg(edge + e);
                if ((unsigned)eid >= (unsigned)nE) {
                    if (lane == 0) flag_index_error();
                    continue;
                }
                const float* pr = P + (long long)eid * B;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const long long s = base + 128 * q + 4 * lane;
                    if (s < B) {
                        const float4 v = ldg4(pr + s);
                        acc[q].x += v.x; acc[q].y += v.y; acc[q].z += v.z; acc[q].w += v.w;
                    }
                }
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const long long s = base + 128 * q + 4 * lane;
                if (s < B) *reinterpret_cast<float4*>(out + s) = acc[q];
            }
        }
    } else {
        for (long long base = 0; base < B; base += 128) {
            float acc[4] = {0.f, 0.f, 0.f, 0.f};
            for (int e = e0; e < e1; ++e) {
                int eid = __ldg(edge + e);
                if ((unsigned)eid >= (unsigned)nE) {
                    if (lane == 0) flag_index_error();
                    continue;
                }
                const float* pr = P + (long long)eid * B;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const long long s = base + 32 * q + lane;
                    if (s < B) acc[q] += __ldg(pr + s);
                }
            }
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                const long long s = base + 32 * q + lane;
                if (s < B) out[s] = acc[q];
            }
        }
    }
}

// ----------------------------------------------------------- launchers --

// Samples per forward block: the whole batch when the layer input fits in
// a fraction of L2, else a batch slice so that the gathered working set of
// the blocks resident at one time stays in L2.
long long forward_chunk(int w_in, long long B) {
    const long long l2_budget = 48ll << 20;
    if ((long long)w_in * B * 4 <= l2_budget) return B;
    long long c = l2_budget / ((long long)w_in * 4);
    c = (c / 128) * 128;
    if (c < 256) c = 256;
    return c < B ? c : B;
}

template <int k>
int launch_forward(const float* X, int w_in, long long B, const int* conn, const float* theta,
                   int w, float* Y, bool vec, cudaStream_t st) {
    long long chunk = forward_chunk(w_in, B);
    if (vec) chunk = (chunk + 3) / 4 * 4;
    const long long ny = (B + chunk - 1) / chunk;
    if (ny > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((w + kFwdWarps - 1) / kFwdWarps), (unsigned)ny);
    if (vec)
        lut_forward_staged_kernel<k><<<grid, kFwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, Y, chunk);
    else
        lut_forward_kernel<k, false><<<grid, kFwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, Y, chunk);
    return launch_status();
}

template <int k, bool WANT_DX>
int launch_staged(const float* X, int w_in, long long B, const int* conn, const float* theta,
                  int w, const float* dY, float* dtheta, float* P, cudaStream_t st) {
    constexpr size_t smem = staged_smem_bytes<k>();
    auto kern = lut_backward_staged_kernel<k, WANT_DX>;
    if (smem > 48 * 1024 &&
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    dim3 grid((unsigned)((w + kBwdWarps - 1) / kBwdWarps));
    kern<<<grid, kBwdWarps * 32, smem, st>>>(X, w_in, B, conn, theta, w, dY, dtheta, P);
    return launch_status();
}

template <int k>
int launch_backward(const float* X, int w_in, long long B, const int* conn, const float* theta,
                    int w, const float* dY, float* dtheta, float* P, bool want_dx,
                    cudaStream_t st) {
    if constexpr (k >= 2) {
        const bool staged = (B % 4 == 0) && aligned16(X) && aligned16(dY);
        if (staged)
            return want_dx ? launch_staged<k, true>(X, w_in, B, conn, theta, w, dY, dtheta, P, st)
                           : launch_staged<k, false>(X, w_in, B, conn, theta, w, dY, dtheta, P, st);
    }
    dim3 grid((unsigned)((w + kBwdWarps - 1) / kBwdWarps));
    if (want_dx)
        lut_backward_kernel<k, true><<<grid, kBwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, dY, dtheta, P);
    else
        lut_backward_kernel<k, false><<<grid, kBwdWarps * 32, 0, st>>>(X, w_in, B, conn, theta, w, dY, dtheta, P);
    return launch_status();
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

extern "C" int bitlogic_lut_forward(const float* X, int32_t w_in, int64_t B,
                                    const int32_t* conn, const float* theta,
                                    int32_t w, int32_t k, float* Y, cudaStream_t stream) {
    int st = check_layer(X, w_in, B, conn, theta, w, k);
    if (st) return st;
    if (B == 0) return BITLOGIC_OK;
    if (!Y) return BITLOGIC_ERR_NULL;
    const bool vec = (B % 4 == 0) && aligned16(X) && aligned16(Y);
    switch (k) {
        case 1: return launch_forward<1>(X, w_in, B, conn, theta, w, Y, vec, stream);
        case 2: return launch_forward<2>(X, w_in, B, conn, theta, w, Y, vec, stream);
        case 3: return launch_forward<3>(X, w_in, B, conn, theta, w, Y, vec, stream);
        case 4: return launch_forward<4>(X, w_in, B, conn, theta, w, Y, vec, stream);
        case 5: return launch_forward<5>(X, w_in, B, conn, theta, w, Y, vec, stream);
        default: return launch_forward<6>(X, w_in, B, conn, theta, w, Y, vec, stream);
    }
}

extern "C" size_t bitlogic_lut_backward_workspace(int32_t w_in, int64_t B, int32_t w,
                                                  int32_t k, int32_t want_dx) {
    (void)w_in;
    if (!want_dx || B <= 0 || w <= 0 || k <= 0) return 0;
    return (size_t)w * (size_t)k * (size_t)B * sizeof(float);
}

extern "C" int bitlogic_lut_backward_edges(const float* X, int32_t w_in, int64_t B,
                                           const int32_t* conn, const float* theta,
                                           int32_t w, int32_t k, const float* dY,
                                           float* dtheta, float* edge_terms,
                                           cudaStream_t stream) {
    int st = check_layer(X, w_in, B, conn, theta, w, k);
    if (st) return st;
    if (!dtheta || (B > 0 && !dY)) return BITLOGIC_ERR_NULL;
    if (B == 0) {
        // empty batch: the batch sums are zero
        if (cudaMemsetAsync(dtheta, 0, sizeof(float) * (size_t)w * ((size_t)1 << k), stream) != cudaSuccess)
            return BITLOGIC_ERR_CUDA;
        return BITLOGIC_OK;
    }
    const bool want = edge_terms != nullptr;
    switch (k) {
        case 1: return launch_backward<1>(X, w_in, B, conn, theta, w, dY, dtheta, edge_terms, want, stream);
        case 2: return launch_backward<2>(X, w_in, B, conn, theta, w, dY, dtheta, edge_terms, want, stream);
        case 3: return launch_backward<3>(X, w_in, B, conn, theta, w, dY, dtheta, edge_terms, want, stream);
        case 4: return launch_backward<4>(X, w_in, B, conn, theta, w, dY, dtheta, edge_terms, want, stream);
        case 5: return launch_backward<5>(X, w_in, B, conn, theta, w, dY, dtheta, edge_terms, want, stream);
        default: return launch_backward<6>(X, w_in, B, conn, theta, w, dY, dtheta, edge_terms, want, stream);
    }
}

extern "C" int bitlogic_csr_reduce(const float* edge_terms, int64_t B, const int32_t* csr_off,
                                   const int32_t* csr_edge, int32_t w_in, int32_t n_edges,
                                   float* dX, cudaStream_t stream) {
    if (B < 0 || w_in <= 0 || n_edges < 0) return BITLOGIC_ERR_SHAPE;
    if (B == 0) return BITLOGIC_OK;
    if (!edge_terms || !csr_off || !csr_edge || !dX) return BITLOGIC_ERR_NULL;
    const bool vec = (B % 4 == 0) && aligned16(edge_terms) && aligned16(dX);
    dim3 grid((unsigned)((w_in + kCsrWarps - 1) / kCsrWarps));
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
