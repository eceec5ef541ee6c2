// Table gradient of a LUT layer whose output gradient is recomputed from the
// next layer (chain rule through a next layer of small fan-in), so that
// neither the next layer's per-edge input-gradient terms nor this layer's
// output gradient are stored.
//
// For the node j of this layer, output row j is an input of the next layer;
// its gradient (the next layer's input gradient, summed over the consumers)
// is
//   g_j[s] = sum over the consumer edges e = (j2, slot) of j, in increasing
//            CSR position (node order), of dY2[j2][s] * d y_j2 / d x_slot (s),
// and for a next-layer node of fan-in ku the derivative with respect to one
// input is a multilinear function of its other ku - 1 inputs:
//   d y / d x_slot = sum over the corners b of the other inputs of
//                    (t[b, slot = 1] - t[b, slot = 0]) * prod_m x_m^b_m (1 - x_m)^(1 - b_m),
// i.e. a constant (ku = 1), c0 + c1 u (ku = 2), or
// c0 + c1 u + c2 v + c3 u v (ku = 3, Moebius coefficients of the corner
// differences), with u, v the other inputs in slot order.  Every consumer
// costs ku - 1 gathered values of this layer's output (one row each, held in
// L2 by the step) and one output-gradient row of the next layer (the head's
// per-class rows: a handful of rows), instead of the per-edge term written
// by the next layer's backward and read back by a reduction.
//
// The table gradient itself is the dtheta-only form of the soft backward:
//   dtheta_a = t_a (1 - t_a) sum_s g_s w_a(x_s),
// with the corner weights w_a built per sample as the outer product of the
// low-half and high-half corner weights of the node's own k inputs.
//
// Layout and scheduling follow the dtheta-only kernel: persistent one-warp
// blocks, a node over the whole batch, 4 consecutive samples per lane in each
// 128-sample stage, the node's k input rows streamed through a lane-private
// cp.async ring that runs across node boundaries, and a fixed butterfly of
// shuffles for the batch reduction.  The consumers' rows are gathered for
// several stages at a time (eight for k <= 3), so a warp has eight (ku = 1)
// to twenty-four (ku = 3) independent loads in flight per consumer.  Needs B % 4 == 0 and 16-byte aligned
// X, Y, the next layer's gradient rows and dY_out.
#include "common.cuh"

namespace bitlogic {
namespace {

constexpr int kTStageSamples = 128;   // one 16-byte chunk per lane and row
constexpr int kTStages = 3;           // ring stages in flight per warp
constexpr int kTMinBlocks = 16;       // one-warp blocks per SM
// stages whose consumer rows are gathered together: fewer for the wider
// tables, whose 2^k accumulators already take most registers
template <int k>
__host__ __device__ constexpr int through_chunk() { return k <= 3 ? 8 : (k == 4 ? 4 : (k == 5 ? 2 : 1)); }

__device__ __forceinline__ float4 ldg4t(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }

__device__ __forceinline__ float comp4(const float4& v, int c) {
    return c == 0 ? v.x : c == 1 ? v.y : c == 2 ? v.z : v.w;
}

// Table entry of a node form: the sigmoid of the logit (soft LightLUT), or
// the hard sample [theta > 0] (straight-through node).
__device__ __forceinline__ float table_entry(float th, int node) {
    return node == BITLOGIC_NODE_ST ? (th > 0.f ? 1.f : 0.f) : sigmoidf(th);
}

// Reduce-scatter of N values per lane over the lane offsets O, O/2, ..., 1
// (fixed order): afterwards lane l holds the sums of entries
// l N0/32 .. l N0/32 + N0/32 - 1 for N0 = 2^k >= 32 values, of entry
// l >> (5 - k) for N0 < 32.
template <int N, int O, int M>
__device__ __forceinline__ void reduce_scatter(float (&v)[M], int lane) {
    if constexpr (O > 0) {
        if constexpr (N > 1) {
            const bool up = (lane & O) != 0;
#pragma unroll
            for (int i = 0; i < N / 2; ++i) {
                const float send = up ? v[i] : v[i + N / 2];
                const float keep = up ? v[i + N / 2] : v[i];
                v[i] = keep + __shfl_xor_sync(0xffffffffu, send, O);
            }
            reduce_scatter<N / 2, O / 2>(v, lane);
        } else {
            v[0] += __shfl_xor_sync(0xffffffffu, v[0], O);
            reduce_scatter<1, O / 2>(v, lane);
        }
    }
}

// One consumer edge of a row: the next layer's gradient row, the rows of the
// consumer's other inputs, and the coefficients of its derivative.
template <int ku>
struct Consumer {
    int grow;                              // next-layer gradient row (-1: no contribution)
    int orow[ku > 1 ? ku - 1 : 1];         // other inputs' rows
    float c[1 << (ku - 1)];                // derivative coefficients
};

template <int ku>
__device__ __forceinline__ Consumer<ku> load_consumer(int p, const int* __restrict__ up_edge, int n_up,
                                                      const int* __restrict__ up_conn,
                                                      const float* __restrict__ up_theta, int up_group,
                                                      int w, int node, bool& bad) {
    constexpr int KU = 1 << ku, H = KU / 2;
    Consumer<ku> q;
    q.grow = -1;
#pragma unroll
    for (int m = 0; m < (ku > 1 ? ku - 1 : 1); ++m) q.orow[m] = 0;
#pragma unroll
    for (int b = 0; b < H; ++b) q.c[b] = 0.f;
    const int id = up_edge ? __ldg(up_edge + p) : p;
    if ((unsigned)id >= (unsigned)n_up) {
        bad = true;
        return q;
    }
    const int j2 = id / ku, slot = id - j2 * ku;
    q.grow = j2 / up_group;
    // other input o (in slot order) is slot o below `slot`, slot o + 1 above
#pragma unroll
    for (int o = 0; o < ku - 1; ++o) {
        int r = __ldg(up_conn + (long long)j2 * ku + (o < slot ? o : o + 1));
        if ((unsigned)r >= (unsigned)w) {
            bad = true;
            r = 0;
        }
        q.orow[o] = r;
    }
    // corner differences over the other inputs (b: their bits in slot order)
    float d[H];
#pragma unroll
    for (int b = 0; b < H; ++b) {
        // table index with the slot bit inserted at position `slot`
        const int lowmask = (1 << slot) - 1;
        const int a0 = (b & lowmask) | ((b & ~lowmask) << 1);
        const int a1 = a0 | (1 << slot);
        d[b] = table_entry(__ldg(up_theta + (long long)j2 * KU + a1), node) -
               table_entry(__ldg(up_theta + (long long)j2 * KU + a0), node);
    }
    if constexpr (ku == 1) {
        q.c[0] = d[0];
    } else if constexpr (ku == 2) {
        q.c[0] = d[0];
        q.c[1] = d[1] - d[0];
    } else {
        q.c[0] = d[0];
        q.c[1] = d[1] - d[0];
        q.c[2] = d[2] - d[0];
        q.c[3] = (d[3] - d[2]) - (d[1] - d[0]);
    }
    return q;
}

template <int ku>
__device__ __forceinline__ Consumer<ku> shfl_consumer(const Consumer<ku>& q, int src) {
    Consumer<ku> r;
    r.grow = __shfl_sync(0xffffffffu, q.grow, src);
#pragma unroll
    for (int m = 0; m < (ku > 1 ? ku - 1 : 1); ++m) r.orow[m] = __shfl_sync(0xffffffffu, q.orow[m], src);
#pragma unroll
    for (int b = 0; b < (1 << (ku - 1)); ++b) r.c[b] = __shfl_sync(0xffffffffu, q.c[b], src);
    return r;
}

// g += dY2 * derivative for the lane's four samples at s4.
template <int ku>
__device__ __forceinline__ void add_consumer(float4& g, const Consumer<ku>& q, const float* __restrict__ Y,
                                             const float* __restrict__ up_dY, long long B, long long s4) {
    if (q.grow < 0) return;
    const float4 dy = ldg4t(up_dY + (long long)q.grow * B + s4);
    if constexpr (ku == 1) {
        g.x = fmaf(dy.x, q.c[0], g.x);
        g.y = fmaf(dy.y, q.c[0], g.y);
        g.z = fmaf(dy.z, q.c[0], g.z);
        g.w = fmaf(dy.w, q.c[0], g.w);
    } else if constexpr (ku == 2) {
        const float4 u = ldg4t(Y + (long long)q.orow[0] * B + s4);
        g.x = fmaf(dy.x, fmaf(q.c[1], u.x, q.c[0]), g.x);
        g.y = fmaf(dy.y, fmaf(q.c[1], u.y, q.c[0]), g.y);
        g.z = fmaf(dy.z, fmaf(q.c[1], u.z, q.c[0]), g.z);
        g.w = fmaf(dy.w, fmaf(q.c[1], u.w, q.c[0]), g.w);
    } else {
        const float4 u = ldg4t(Y + (long long)q.orow[0] * B + s4);
        const float4 v = ldg4t(Y + (long long)q.orow[1] * B + s4);
        g.x = fmaf(dy.x, fmaf(v.x, fmaf(q.c[3], u.x, q.c[2]), fmaf(q.c[1], u.x, q.c[0])), g.x);
        g.y = fmaf(dy.y, fmaf(v.y, fmaf(q.c[3], u.y, q.c[2]), fmaf(q.c[1], u.y, q.c[0])), g.y);
        g.z = fmaf(dy.z, fmaf(v.z, fmaf(q.c[3], u.z, q.c[2]), fmaf(q.c[1], u.z, q.c[0])), g.z);
        g.w = fmaf(dy.w, fmaf(v.w, fmaf(q.c[3], u.w, q.c[2]), fmaf(q.c[1], u.w, q.c[0])), g.w);
    }
}

template <int k>
__host__ __device__ constexpr int through_floats_per_warp() {
    return kTStages * k * kTStageSamples;
}

template <int k, int ku>
__global__ void __launch_bounds__(32, kTMinBlocks)
lut_theta_through_kernel(const float* __restrict__ X, int w_in, long long B, const int* __restrict__ conn,
                         const float* __restrict__ theta, int w, const float* __restrict__ Y,
                         const int* __restrict__ up_conn, const float* __restrict__ up_theta, int up_w,
                         const float* __restrict__ up_dY, int up_group, const int* __restrict__ up_off,
                         const int* __restrict__ up_edge, int node, float* __restrict__ dtheta,
                         float* __restrict__ dY_out) {
    constexpr int K = 1 << k, KL = k / 2, NU = 1 << KL, NV = 1 << (k - KL);
    constexpr int CH = kTStageSamples;
    constexpr int kTChunk = through_chunk<k>();
    extern __shared__ __align__(16) float smem[];
    const int lane = threadIdx.x & 31;
    float* ring = smem;
    const int G = gridDim.x;
    const int jfirst = blockIdx.x;
    const int nst = (int)((B + CH - 1) / CH);
    const int n_up = up_w * ku;

    // issue stream: stage si of node ji, kTStages - 1 stages ahead of the
    // compute stream; rows of the warp's node after ji are loaded ahead
    int ji = jfirst, si = 0, ib = 0;
    int ri[k], rn[k];
    auto rows_of = [&](int j, int (&r)[k]) {
        bool bad = false;
#pragma unroll
        for (int i = 0; i < k; ++i) {
            int c = __ldg(conn + (long long)j * k + i);
            if ((unsigned)c >= (unsigned)w_in) {
                bad = true;
                c = 0;
            }
            r[i] = c;
        }
        if (bad && lane == 0) flag_index_error();
    };
#pragma unroll
    for (int i = 0; i < k; ++i) ri[i] = rn[i] = 0;
    if (ji < w) rows_of(ji, ri);
    if (ji + G < w) rows_of(ji + G, rn);
    auto issue = [&]() {
        if (ji < w) {
            const long long s4 = (long long)si * CH + 4 * lane;
            if (s4 < B) {
                float* buf = ring + ib * (k * CH) + 4 * lane;
#pragma unroll
                for (int r = 0; r < k; ++r) cp_async16(buf + r * CH, X + (long long)ri[r] * B + s4);
            }
            if (++si == nst) {
                si = 0;
                ji += G;
#pragma unroll
                for (int i = 0; i < k; ++i) ri[i] = rn[i];
                if (ji + G < w) rows_of(ji + G, rn);
            }
        }
        cp_async_commit();
        ib = (ib + 1 == kTStages) ? 0 : ib + 1;
    };
#pragma unroll 1
    for (int i = 0; i < kTStages - 1; ++i) issue();

    int rb = 0;
#pragma unroll 1
    for (int j = jfirst; j < w; j += G) {
        // the node's consumers in the next layer (CSR positions e0 .. e1 - 1)
        int e0 = __ldg(up_off + j), e1 = __ldg(up_off + j + 1);
        if (e0 < 0 || e1 < e0 || e1 > n_up) {
            if (lane == 0) flag_index_error();
            e0 = e1 = 0;
        }
        const int deg = e1 - e0;
        bool bad = false;
        Consumer<ku> mine;
        mine.grow = -1;
        if (lane < deg)
            mine = load_consumer<ku>(e0 + lane, up_edge, n_up, up_conn, up_theta, up_group, w, node, bad);
        if (__any_sync(0xffffffffu, bad) && lane == 0) flag_index_error();

        float acc[K];
#pragma unroll
        for (int a = 0; a < K; ++a) acc[a] = 0.f;
#pragma unroll 1
        for (int sc0 = 0; sc0 < nst; sc0 += kTChunk) {
            // the node's output gradient over kTChunk stages, consumers in
            // increasing CSR position: each consumer's rows are gathered for
            // all the chunk's stages at once (kTChunk loads per row in flight)
            float4 gv[kTChunk];
#pragma unroll
            for (int t = 0; t < kTChunk; ++t) gv[t] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
            for (int c0 = 0; c0 < deg; c0 += 32) {
                Consumer<ku> cur = mine;
                if (c0 > 0) {   // more than 32 consumers: this chunk's edges
                    bool bad2 = false;
                    cur.grow = -1;
                    if (c0 + lane < deg)
                        cur = load_consumer<ku>(e0 + c0 + lane, up_edge, n_up, up_conn, up_theta, up_group, w,
                                                node, bad2);
                    if (__any_sync(0xffffffffu, bad2) && lane == 0) flag_index_error();
                }
                const int n = min(32, deg - c0);
#pragma unroll 1
                for (int e = 0; e < n; ++e) {
                    const Consumer<ku> q = shfl_consumer<ku>(cur, e);
#pragma unroll
                    for (int t = 0; t < kTChunk; ++t) {
                        const long long s4 = (long long)(sc0 + t) * CH + 4 * lane;
                        if (s4 < B) add_consumer<ku>(gv[t], q, Y, up_dY, B, s4);
                    }
                }
            }
            // the chunk's stages: the table gradient from the node's inputs
#pragma unroll
            for (int t = 0; t < kTChunk; ++t) {
                if (sc0 + t < nst) {
                    issue();
                    cp_async_wait<kTStages - 1>();
                    const long long s4 = (long long)(sc0 + t) * CH + 4 * lane;   // this lane's 4 samples
                    if (s4 < B) {   // B % 4 == 0: all four samples are in range
                        if (dY_out) *reinterpret_cast<float4*>(dY_out + (long long)j * B + s4) = gv[t];
                        const float* buf = ring + rb * (k * CH) + 4 * lane;
                        float4 xv[k];
#pragma unroll
                        for (int q = 0; q < k; ++q) xv[q] = *reinterpret_cast<const float4*>(buf + q * CH);
#pragma unroll
                        for (int r = 0; r < 4; ++r) {
                            float x[k], omx[k];
#pragma unroll
                            for (int q = 0; q < k; ++q) {
                                x[q] = comp4(xv[q], r);
                                omx[q] = 1.0f - x[q];
                            }
                            float U[NU], V[NV];
                            U[0] = comp4(gv[t], r);
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
                    rb = (rb + 1 == kTStages) ? 0 : rb + 1;
                }
            }
        }
        // the node's dtheta: butterfly over the lanes, then t (1 - t)
        reduce_scatter<K, 16>(acc, lane);
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

template <int k, int ku>
int launch_through(const float* X, int w_in, long long B, const int* conn, const float* theta, int w,
                   const float* Y, const int* up_conn, const float* up_theta, int up_w, const float* up_dY,
                   int up_group, const int* up_off, const int* up_edge, int node, float* dtheta, float* dY_out,
                   cudaStream_t st) {
    constexpr size_t smem = (size_t)through_floats_per_warp<k>() * sizeof(float);
    auto kern = lut_theta_through_kernel<k, ku>;
    if (smem > 40 * 1024 &&
        cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    // one wave of persistent one-warp blocks (nodes dealt round-robin)
    const long long resident = (long long)sm_count() * kTMinBlocks;
    const long long blocks = w < resident ? w : resident;
    kern<<<(unsigned)blocks, 32, smem, st>>>(X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY,
                                             up_group, up_off, up_edge, node, dtheta, dY_out);
    return launch_status();
}

template <int k>
int launch_through_k(int up_k, const float* X, int w_in, long long B, const int* conn, const float* theta, int w,
                     const float* Y, const int* up_conn, const float* up_theta, int up_w, const float* up_dY,
                     int up_group, const int* up_off, const int* up_edge, int node, float* dtheta,
                     float* dY_out, cudaStream_t st) {
    switch (up_k) {
        case 1:
            return launch_through<k, 1>(X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY, up_group,
                                        up_off, up_edge, node, dtheta, dY_out, st);
        case 2:
            return launch_through<k, 2>(X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY, up_group,
                                        up_off, up_edge, node, dtheta, dY_out, st);
        default:
            return launch_through<k, 3>(X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY, up_group,
                                        up_off, up_edge, node, dtheta, dY_out, st);
    }
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(lut_through)

extern "C" int bitlogic_lut_backward_through(const float* X, int32_t w_in, int64_t B, const int32_t* conn,
                                             const float* theta, int32_t w, int32_t k, int32_t node,
                                             const float* Y, const int32_t* up_conn, const float* up_theta,
                                             int32_t up_w, int32_t up_k, const float* up_dY, int32_t up_group,
                                             const int32_t* up_off, const int32_t* up_edge, float* dtheta,
                                             float* dY_out, cudaStream_t stream) {
    if (!conn || !theta || !up_conn || !up_theta || !up_off || !dtheta) return BITLOGIC_ERR_NULL;
    if (w_in <= 0 || w <= 0 || B < 0 || up_w <= 0) return BITLOGIC_ERR_SHAPE;
    if (k < 1 || k > 6 || k > w_in || up_k < 1 || up_k > 3 || up_k > w) return BITLOGIC_ERR_FANIN;
    if ((int64_t)w * k > 0x7fffffffLL || (int64_t)up_w * up_k > 0x7fffffffLL) return BITLOGIC_ERR_SHAPE;
    if (up_group < 1 || up_group > up_w || up_w % up_group != 0) return BITLOGIC_ERR_SHAPE;
    if (node != BITLOGIC_NODE_SOFT && node != BITLOGIC_NODE_ST) return BITLOGIC_ERR_NODE;
    if (B == 0) {
        if (cudaMemsetAsync(dtheta, 0, sizeof(float) * (size_t)w * ((size_t)1 << k), stream) != cudaSuccess)
            return BITLOGIC_ERR_CUDA;
        return BITLOGIC_OK;
    }
    if (!X || !Y || !up_dY) return BITLOGIC_ERR_NULL;
    if (B % 4 != 0 || !aligned16(X) || !aligned16(Y) || !aligned16(up_dY) || (dY_out && !aligned16(dY_out)))
        return BITLOGIC_ERR_ALIGN;
    switch (k) {
        case 1: return launch_through_k<1>(up_k, X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY,
                                           up_group, up_off, up_edge, node, dtheta, dY_out, stream);
        case 2: return launch_through_k<2>(up_k, X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY,
                                           up_group, up_off, up_edge, node, dtheta, dY_out, stream);
        case 3: return launch_through_k<3>(up_k, X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY,
                                           up_group, up_off, up_edge, node, dtheta, dY_out, stream);
        case 4: return launch_through_k<4>(up_k, X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY,
                                           up_group, up_off, up_edge, node, dtheta, dY_out, stream);
        case 5: return launch_through_k<5>(up_k, X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY,
                                           up_group, up_off, up_edge, node, dtheta, dY_out, stream);
        default: return launch_through_k<6>(up_k, X, w_in, B, conn, theta, w, Y, up_conn, up_theta, up_w, up_dY,
                                            up_group, up_off, up_edge, node, dtheta, dY_out, stream);
    }
}
