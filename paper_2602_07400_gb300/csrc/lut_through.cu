// Table gradient of a LUT layer (the dtheta-only backward: no input
// gradient), for the inputs and output-gradient sources the training step
// uses on its first layer:
//
// * the layer input as fp32 rows or as byte rows (binary wires, e.g. the
//   thermometer encoder's output written by bitlogic_encode_thermometer_u8);
// * the output gradient
//   - recomputed from the next layer itself (through: chain rule through a
//     next layer of small fan-in), so that neither the next layer's per-edge
//     terms nor this layer's output gradient are stored (fp32 or byte rows);
//   - from rows: row j / group of dY (byte rows);
//   - from terms: the next layer's per-edge input-gradient terms, summed over
//     the node's consumers in increasing CSR position (the order of
//     bitlogic_csr_reduce, so the sum is the same bit for bit; byte rows).
//
// Through: for the node j of this layer, output row j is an input of the
// next layer; its gradient (the next layer's input gradient, summed over
// the consumers) is
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
// low-half and high-half corner weights of the node's own k inputs.  On byte
// rows (binary wires) the corner weights of a sample are one-hot: w_a is 1
// for the corner a = sum_i x_i 2^i the inputs sit on and 0 elsewhere (the
// identity behind "a soft node on binary inputs returns its table entry",
// §2), so the sum adds g_s to one entry per sample.  Each lane keeps its
// 2^k partial sums in its own column of a shared [2^k][32] array (no bank
// conflicts) and adds each sample's g to the entry its index selects, in the
// sample order of the register form; since g * 1 and g * 0 are exact, the
// partial sums, and after the same butterfly dtheta, are the fp32 form's bit
// for bit, for a few instructions per sample instead of ~2^k multiply-adds.
//
// The through kernel follows the dtheta-only kernel's layout: persistent
// one-warp blocks, a node over the whole batch, 4 consecutive samples per
// lane in each 128-sample stage, the node's k input rows streamed through a
// lane-private cp.async ring that runs across node boundaries (16 bytes per
// lane and row for fp32 rows, 4 for byte rows), and a fixed butterfly of
// shuffles for the batch reduction; the output gradient is formed for
// several stages at a time (a chunk), so the consumer rows it reads have
// several independent loads in flight.  The rows and terms sources on byte
// rows have a streaming kernel of their own (below).  Needs B % 4 == 0 and
// 16-byte aligned X, the gradient rows, the terms, Y and dY_out.
#include "common.cuh"

namespace bitlogic {
namespace {

constexpr int kTStageSamples = 128;   // one 16-byte chunk per lane and row
constexpr int kTStages = 3;           // ring stages in flight per warp
#ifndef BITLOGIC_THROUGH_MIN_BLOCKS
#define BITLOGIC_THROUGH_MIN_BLOCKS 16
#endif
#ifndef BITLOGIC_THROUGH_CHUNK
#define BITLOGIC_THROUGH_CHUNK 8
#endif
constexpr int kTMinBlocks = BITLOGIC_THROUGH_MIN_BLOCKS;   // one-warp blocks per SM
static_assert(kTMinBlocks >= 1 && kTMinBlocks <= 32, "one-warp blocks per SM");
static_assert(BITLOGIC_THROUGH_CHUNK >= 1 && BITLOGIC_THROUGH_CHUNK <= 16, "stages gathered together");
// stages whose consumer rows are gathered together: fewer for the wider
// tables, whose 2^k accumulators already take most registers
template <int k>
__host__ __device__ constexpr int through_chunk() {
    return k <= 3 ? BITLOGIC_THROUGH_CHUNK : (k == 4 ? 4 : (k == 5 ? 2 : 1));
}

__device__ __forceinline__ float4 ldg4t(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }

__device__ __forceinline__ float comp4(const float4& v, int c) {
    return c == 0 ? v.x : c == 1 ? v.y : c == 2 ? v.z : v.w;
}

// Binary wires: the corner index of the lane's 4 samples of a stage, one
// per byte (byte r = sum_i bit(x_i[s + r]) 2^i); `xb` points at the lane's 4
// bytes of row 0 in a ring slot whose rows are `stride` bytes apart.  A byte
// is read by its lowest bit.
template <int k>
__device__ __forceinline__ uint32_t corner_index4(const uint8_t* xb, int stride) {
    uint32_t v = *reinterpret_cast<const uint32_t*>(xb + (k - 1) * stride) & 0x01010101u;
#pragma unroll
    for (int q = k - 2; q >= 0; --q) v = (v << 1) | (*reinterpret_cast<const uint32_t*>(xb + q * stride) & 0x01010101u);
    return v;
}

// Adds the 4 samples' gradients to the entries their indices select in the
// lane's column (`col` = the [2^k][32] array + lane), in sample order.
__device__ __forceinline__ void corner_add4(float* col, uint32_t v, const float4& g) {
    col[(v & 0xffu) * 32] += g.x;
    col[((v >> 8) & 0xffu) * 32] += g.y;
    col[((v >> 16) & 0xffu) * 32] += g.z;
    col[(v >> 24) * 32] += g.w;
}

// Moves the lane's column into registers (for the butterfly) and, with
// CLEAR, clears it for the warp's next node.
template <int K, bool CLEAR = true>
__device__ __forceinline__ void corner_take(float* col, float (&acc)[K]) {
#pragma unroll
    for (int a = 0; a < K; ++a) {
        acc[a] = col[a * 32];
        if constexpr (CLEAR) col[a * 32] = 0.f;
    }
}

template <typename TX>
__host__ __device__ constexpr bool byte_rows() { return sizeof(TX) == 1; }

// Shared bytes of the per-lane corner sums (byte rows only).
template <typename TX>
__host__ __device__ constexpr int corner_bytes(int k) {
    return byte_rows<TX>() ? (1 << k) * 32 * (int)sizeof(float) : 0;
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

struct GradIn {
    const float* dY;        // rows: [w / group][B]
    int group;
    const float* terms;     // terms: [n_terms][B]
    int n_terms;
    const int* off;         // terms, through: CSR positions of this layer's rows [w + 1]
    const int* edge;        // terms, through: edge ids in CSR order (NULL: identity)
    const float* Y;         // through: this layer's output [w][B]
    const int* up_conn;     // through: the next layer [up_w][up_k]
    const float* up_theta;
    int up_w;
    const float* up_dY;     // through: the next layer's gradient rows [up_w / up_group][B]
    int up_group;
};

template <typename TX>
__host__ __device__ constexpr int ring_bytes_per_warp(int k) {
    return kTStages * k * kTStageSamples * (int)sizeof(TX);
}

// The lane's 16 (fp32) or 4 (bytes) bytes of one row of one stage.
__device__ __forceinline__ void copy_row_part(float* dst, const float* src) { cp_async16(dst, src); }
__device__ __forceinline__ void copy_row_part(uint8_t* dst, const uint8_t* src) {
    const unsigned sa = (unsigned)__cvta_generic_to_shared(dst);
    asm volatile("cp.async.ca.shared.global [%0], [%1], 4;\n" ::"r"(sa), "l"(src) : "memory");
}
// Its four samples (fp32 rows; byte rows take the one-hot form).
__device__ __forceinline__ float4 read_row_part(const float* p) { return *reinterpret_cast<const float4*>(p); }

template <int k, int ku, typename TX>
__global__ void __launch_bounds__(32, kTMinBlocks)
lut_theta_through_kernel(const TX* __restrict__ X, int w_in, long long B, const int* __restrict__ conn,
                         const float* __restrict__ theta, int w, GradIn gi, int node, float* __restrict__ dtheta,
                         float* __restrict__ dY_out) {
    constexpr int K = 1 << k, KL = k / 2, NU = 1 << KL, NV = 1 << (k - KL);
    constexpr int CH = kTStageSamples;
    constexpr int kTChunk = through_chunk<k>();
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int lane = threadIdx.x & 31;
    TX* ring = reinterpret_cast<TX*>(smem_raw);
    constexpr bool BIN = byte_rows<TX>();   // one-hot corner weights
    float* corners = reinterpret_cast<float*>(smem_raw + ring_bytes_per_warp<TX>(k)) + lane;
    if constexpr (BIN) {
#pragma unroll
        for (int a = 0; a < K; ++a) corners[a * 32] = 0.f;
    }
    const int G = gridDim.x;
    const int jfirst = blockIdx.x;
    const int nst = (int)((B + CH - 1) / CH);
    const int n_up = gi.up_w * ku;   // CSR positions

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
                TX* buf = ring + ib * (k * CH) + 4 * lane;
#pragma unroll
                for (int r = 0; r < k; ++r) copy_row_part(buf + r * CH, X + (long long)ri[r] * B + s4);
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
        // the node's upstream edges (terms, through: CSR positions e0 .. e1 - 1)
        int e0 = __ldg(gi.off + j), e1 = __ldg(gi.off + j + 1);
        if (e0 < 0 || e1 < e0 || e1 > n_up) {
            if (lane == 0) flag_index_error();
            e0 = e1 = 0;
        }
        const int deg = e1 - e0;
        // per lane one consumer (through), for the positions e0 .. e0 + 31
        Consumer<ku> mine;
        mine.grow = -1;
        auto load_edges = [&](int c0) {
            bool bad = false;
            mine.grow = -1;
            if (c0 + lane < deg)
                mine = load_consumer<ku>(e0 + c0 + lane, gi.edge, n_up, gi.up_conn, gi.up_theta, gi.up_group, w,
                                         node, bad);
            if (__any_sync(0xffffffffu, bad) && lane == 0) flag_index_error();
        };
        load_edges(0);

        float acc[K];
#pragma unroll
        for (int a = 0; a < K; ++a) acc[a] = 0.f;
#pragma unroll 1
        for (int sc0 = 0; sc0 < nst; sc0 += kTChunk) {
            // the node's output gradient over kTChunk stages
            float4 gv[kTChunk];
#pragma unroll
            for (int t = 0; t < kTChunk; ++t) gv[t] = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll 1
            for (int c0 = 0; c0 < deg; c0 += 32) {
                if (c0 > 0) load_edges(c0);   // more than 32 upstream edges: this chunk's
                const int n = min(32, deg - c0);
                {
                    // consumers in increasing CSR position: each consumer's rows
                    // for all the chunk's stages at once
#pragma unroll 1
                    for (int e = 0; e < n; ++e) {
                        const Consumer<ku> q = shfl_consumer<ku>(mine, e);
#pragma unroll
                        for (int t = 0; t < kTChunk; ++t) {
                            const long long s4 = (long long)(sc0 + t) * CH + 4 * lane;
                            if (s4 < B) add_consumer<ku>(gv[t], q, gi.Y, gi.up_dY, B, s4);
                        }
                    }
                }
            }
            if (deg > 32) load_edges(0);   // the next chunk of stages starts again at position e0
            // the chunk's stages: the table gradient from the node's inputs
#pragma unroll
            for (int t = 0; t < kTChunk; ++t) {
                if (sc0 + t < nst) {
                    issue();
                    cp_async_wait<kTStages - 1>();
                    const long long s4 = (long long)(sc0 + t) * CH + 4 * lane;   // this lane's 4 samples
                    if (s4 < B) {   // B % 4 == 0: all four samples are in range
                        if (dY_out) *reinterpret_cast<float4*>(dY_out + (long long)j * B + s4) = gv[t];
                        const TX* buf = ring + rb * (k * CH) + 4 * lane;
                        if constexpr (BIN) {
                            corner_add4(corners, corner_index4<k>(reinterpret_cast<const uint8_t*>(buf), CH), gv[t]);
                        } else {
                            float4 xv[k];
#pragma unroll
                            for (int q = 0; q < k; ++q) xv[q] = read_row_part(buf + q * CH);
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
                    }
                    rb = (rb + 1 == kTStages) ? 0 : rb + 1;
                }
            }
        }
        // the node's dtheta: butterfly over the lanes, then t (1 - t)
        if constexpr (BIN) corner_take<K>(corners, acc);
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

// Byte rows (binary wires) with the output gradient from dY rows or from
// the next layer's per-edge terms: the one-hot table gradient, streaming
// form.  The arithmetic per sample is one add, so the kernel moves data: a
// warp per node over the whole batch in chunks of kBytesChunk stages (128
// samples each, 4 per lane); per chunk each lane loads its output-gradient
// segments (a dY row, or the node's consumer term rows summed in increasing
// CSR position, the order of bitlogic_csr_reduce) and its k input words per
// stage straight into registers, so a warp has a few KB of independent loads
// in flight and no ring to wait on, and then adds each sample's gradient to
// the entry its bits select in the lane's column of a shared [2^k][32] array.
// The lane visits its samples in the order of the fp32 kernels and the lanes
// are combined by the same butterfly, so dtheta is theirs bit for bit.
#ifndef BITLOGIC_BYTES_WARPS
#define BITLOGIC_BYTES_WARPS 2
#endif
#ifndef BITLOGIC_BYTES_CHUNK
#define BITLOGIC_BYTES_CHUNK 4
#endif
#ifndef BITLOGIC_BYTES_STREAM
#define BITLOGIC_BYTES_STREAM 1
#endif
#ifndef BITLOGIC_BYTES_UNROLL
#define BITLOGIC_BYTES_UNROLL 4
#endif
constexpr int kBytesWarps = BITLOGIC_BYTES_WARPS;   // warps (nodes) per block
constexpr int kBytesChunk = BITLOGIC_BYTES_CHUNK;   // stages per chunk
constexpr int kBytesUnroll = BITLOGIC_BYTES_UNROLL;   // term rows whose loads are issued together

// BITS: the input is wire bit rows (one bit per sample, `words` 32-bit words
// per row; see kBitBlock) instead of byte rows: a chunk's 4 stages lie in one
// 1024-sample block, so each lane loads one word per input row per chunk and
// finds stage r's 4 wires as bytes of (word >> r) & 0x01010101.
static_assert((kBitBlock / kTStageSamples) % kBytesChunk == 0, "a chunk's stages lie in one bit-row block");

// order (or NULL): the warp at position p takes node order[p] (a permutation
// of the nodes, e.g. by decreasing term count so that the longest nodes start
// first); only the schedule changes.  With an order the terms' CSR map is
// the one in the order's sequence (position p's rows at off[p] ..
// off[p+1] - 1), so a node's range does not wait for its index.
template <int k, bool TERMS, bool BITS>
__global__ void __launch_bounds__(kBytesWarps * 32)
lut_theta_bytes_kernel(const void* __restrict__ Xv, int w_in, long long B, long long words,
                       const int* __restrict__ conn, const float* __restrict__ theta, int w, GradIn gi,
                       float* __restrict__ dtheta, float* __restrict__ dY_out, const int* __restrict__ order) {
    constexpr int K = 1 << k, CH = kTStageSamples;
    extern __shared__ __align__(16) unsigned char smem_raw[];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int p = blockIdx.x * kBytesWarps + warp;
    if (p >= w) return;   // warp-uniform; the block has no barrier
    const int j = order ? __ldg(order + p) : p;
    if ((unsigned)j >= (unsigned)w) {   // not a node: flagged, nothing written
        if (lane == 0) flag_index_error();
        return;
    }
    float* col = reinterpret_cast<float*>(smem_raw) + warp * K * 32 + lane;
#pragma unroll
    for (int a = 0; a < K; ++a) col[a * 32] = 0.f;
    bool bad = false;
    const uint8_t* xr[k];                 // byte rows: the lane's first 4 bytes
    const uint32_t* xb[k];                // bit rows: the lane's word of block 0
#pragma unroll
    for (int i = 0; i < k; ++i) {
        int c = __ldg(conn + (long long)j * k + i);
        if ((unsigned)c >= (unsigned)w_in) {
            bad = true;
            c = 0;
        }
        if constexpr (BITS) xb[i] = static_cast<const uint32_t*>(Xv) + (long long)c * words + lane;
        else xr[i] = static_cast<const uint8_t*>(Xv) + (long long)c * B + 4 * lane;
    }
    // the node's term rows: CSR positions e0 .. e0 + deg - 1, ids of the
    // first 32 one per lane
    int e0 = 0, deg = 0, my_id = -1;
    if constexpr (TERMS) {
        int e1;
        const int r = order ? p : j;   // the node's entry in the CSR map
        e0 = __ldg(gi.off + r);
        e1 = __ldg(gi.off + r + 1);
        if (e0 < 0 || e1 < e0 || e1 > gi.n_terms) {
            bad = true;
            e0 = e1 = 0;
        }
        deg = e1 - e0;
        if (lane < deg) {
            my_id = gi.edge ? __ldg(gi.edge + e0 + lane) : e0 + lane;
            if ((unsigned)my_id >= (unsigned)gi.n_terms) {
                bad = true;
                my_id = -1;
            }
        }
    }
    if (__any_sync(0xffffffffu, bad) && lane == 0) flag_index_error();
    const float* grow = TERMS ? nullptr : gi.dY + (long long)(j / gi.group) * B + 4 * lane;
    const int nst = (int)((B + CH - 1) / CH);
#pragma unroll 1
    for (int c0 = 0; c0 < nst; c0 += kBytesChunk) {
        // stage c0 + c of this lane: samples (c0 + c) * CH + 4 lane .. + 3,
        // all in range when the first is (B % 4 == 0)
        bool in[kBytesChunk];
#pragma unroll
        for (int c = 0; c < kBytesChunk; ++c) in[c] = c0 + c < nst && (long long)(c0 + c) * CH + 4 * lane < B;
        uint32_t xw[BITS ? 1 : kBytesChunk][k];
        if constexpr (BITS) {
#pragma unroll
            for (int i = 0; i < k; ++i) xw[0][i] = __ldg(xb[i] + (long long)(c0 / 8) * 32);
        } else {
#pragma unroll
            for (int c = 0; c < kBytesChunk; ++c)
#pragma unroll
                for (int i = 0; i < k; ++i)
                    xw[c][i] = in[c] ? __ldg(reinterpret_cast<const uint32_t*>(xr[i] + (long long)(c0 + c) * CH)) : 0u;
        }
        float4 g[kBytesChunk];
#pragma unroll
        for (int c = 0; c < kBytesChunk; ++c) g[c] = make_float4(0.f, 0.f, 0.f, 0.f);
        if constexpr (TERMS) {
#pragma unroll kBytesUnroll
            for (int e = 0; e < deg; ++e) {   // warp-uniform count; every lane takes the shuffle
                int id;
                if (e < 32) {
                    id = __shfl_sync(0xffffffffu, my_id, e);
                } else {
                    id = gi.edge ? __ldg(gi.edge + e0 + e) : e0 + e;
                    if ((unsigned)id >= (unsigned)gi.n_terms) {
                        if (lane == 0) flag_index_error();
                        id = -1;
                    }
                }
                if (id >= 0) {
                    const float* row = gi.terms + (long long)id * B + 4 * lane;
#pragma unroll
                    for (int c = 0; c < kBytesChunk; ++c) {
                        if (in[c]) {
#if BITLOGIC_BYTES_STREAM
                            const float4 v = __ldcs(reinterpret_cast<const float4*>(row + (long long)(c0 + c) * CH));
#else
                            const float4 v = ldg4t(row + (long long)(c0 + c) * CH);
#endif
                            g[c].x += v.x; g[c].y += v.y; g[c].z += v.z; g[c].w += v.w;
                        }
                    }
                }
            }
        } else {
#pragma unroll
            for (int c = 0; c < kBytesChunk; ++c)
                if (in[c]) g[c] = ldg4t(grow + (long long)(c0 + c) * CH);
        }
#pragma unroll
        for (int c = 0; c < kBytesChunk; ++c) {
            if (in[c]) {
                if (dY_out) *reinterpret_cast<float4*>(dY_out + (long long)j * B + (long long)(c0 + c) * CH + 4 * lane) = g[c];
                // the 4 samples' wires of input i, as bytes 0 / 1
                auto wire4 = [&](int i) {
                    if constexpr (BITS) return (xw[0][i] >> ((c0 & 7) + c)) & 0x01010101u;
                    else return xw[c][i] & 0x01010101u;
                };
                uint32_t v = wire4(k - 1);
#pragma unroll
                for (int i = k - 2; i >= 0; --i) v = (v << 1) | wire4(i);
                corner_add4(col, v, g[c]);
            }
        }
    }
    // the node's dtheta: butterfly over the lanes, then t (1 - t)
    float acc[K];
    corner_take<K, false>(col, acc);   // the warp's only node
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

template <int k, bool BITS>
int launch_bytes(bool terms, const void* X, int w_in, long long B, const int* conn, const float* theta, int w,
                 const GradIn& gi, float* dtheta, float* dY_out, const int* order, cudaStream_t st) {
    constexpr int smem = kBytesWarps * (1 << k) * 32 * (int)sizeof(float);
    const unsigned blocks = (unsigned)((w + kBytesWarps - 1) / kBytesWarps);
    const long long words = (B + kBitBlock - 1) / kBitBlock * 32;
    auto kern = terms ? lut_theta_bytes_kernel<k, true, BITS> : lut_theta_bytes_kernel<k, false, BITS>;
    if (smem > 40 * 1024 && cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    kern<<<blocks, kBytesWarps * 32, smem, st>>>(X, w_in, B, words, conn, theta, w, gi, dtheta, dY_out, order);
    return launch_status();
}

template <int k, int ku, typename TX>
int launch_through(const TX* X, int w_in, long long B, const int* conn, const float* theta, int w,
                   const GradIn& gi, int node, float* dtheta, float* dY_out, cudaStream_t st) {
    constexpr int smem = ring_bytes_per_warp<TX>(k) + corner_bytes<TX>(k);
    auto kern = lut_theta_through_kernel<k, ku, TX>;
    if (smem > 40 * 1024 && cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, smem) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    // one wave of persistent one-warp blocks (nodes dealt round-robin)
    const long long resident = (long long)sm_count() * kTMinBlocks;
    const long long blocks = w < resident ? w : resident;
    kern<<<(unsigned)blocks, 32, smem, st>>>(X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out);
    return launch_status();
}

template <int k, typename TX>
int launch_through_k(int up_k, const TX* X, int w_in, long long B, const int* conn, const float* theta, int w,
                     const GradIn& gi, int node, float* dtheta, float* dY_out, cudaStream_t st) {
    switch (up_k) {
        case 1: return launch_through<k, 1, TX>(X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
        case 2: return launch_through<k, 2, TX>(X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
        default: return launch_through<k, 3, TX>(X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
    }
}

template <typename TX>
int run_through(int up_k, const TX* X, int w_in, long long B, const int* conn, const float* theta, int w, int k,
                const GradIn& gi, int node, float* dtheta, float* dY_out, cudaStream_t st) {
    switch (k) {
        case 1: return launch_through_k<1, TX>(up_k, X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
        case 2: return launch_through_k<2, TX>(up_k, X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
        case 3: return launch_through_k<3, TX>(up_k, X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
        case 4: return launch_through_k<4, TX>(up_k, X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
        case 5: return launch_through_k<5, TX>(up_k, X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
        default: return launch_through_k<6, TX>(up_k, X, w_in, B, conn, theta, w, gi, node, dtheta, dY_out, st);
    }
}

// Host checks shared by the entry points (before any CUDA call).
int check_common(const void* X, int32_t w_in, int64_t B, const int32_t* conn, const float* theta, int32_t w,
                 int32_t k, int32_t node, const float* dtheta) {
    if (!conn || !theta || !dtheta) return BITLOGIC_ERR_NULL;
    if (w_in <= 0 || w <= 0 || B < 0) return BITLOGIC_ERR_SHAPE;
    if (k < 1 || k > 6 || k > w_in) return BITLOGIC_ERR_FANIN;
    if ((int64_t)w * k > 0x7fffffffLL) return BITLOGIC_ERR_SHAPE;
    if (node != BITLOGIC_NODE_SOFT && node != BITLOGIC_NODE_ST) return BITLOGIC_ERR_NODE;
    if (B > 0 && !X) return BITLOGIC_ERR_NULL;
    return BITLOGIC_OK;
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(lut_through)

// The through form for either input type.
template <typename TX>
static int backward_through(const TX* X, int32_t w_in, int64_t B, const int32_t* conn, const float* theta,
                            int32_t w, int32_t k, int32_t node, const float* Y, const int32_t* up_conn,
                            const float* up_theta, int32_t up_w, int32_t up_k, const float* up_dY, int32_t up_group,
                            const int32_t* up_off, const int32_t* up_edge, float* dtheta, float* dY_out,
                            cudaStream_t stream) {
    int st = check_common(X, w_in, B, conn, theta, w, k, node, dtheta);
    if (st) return st;
    if (!up_conn || !up_theta || !up_off) return BITLOGIC_ERR_NULL;
    if (up_w <= 0) return BITLOGIC_ERR_SHAPE;
    if (up_k < 1 || up_k > 3 || up_k > w) return BITLOGIC_ERR_FANIN;
    if ((int64_t)up_w * up_k > 0x7fffffffLL) return BITLOGIC_ERR_SHAPE;
    if (up_group < 1 || up_group > up_w || up_w % up_group != 0) return BITLOGIC_ERR_SHAPE;
    if (B == 0) {
        if (cudaMemsetAsync(dtheta, 0, sizeof(float) * (size_t)w * ((size_t)1 << k), stream) != cudaSuccess)
            return BITLOGIC_ERR_CUDA;
        return BITLOGIC_OK;
    }
    if (!Y || !up_dY) return BITLOGIC_ERR_NULL;
    if (B % 4 != 0 || !aligned16(X) || !aligned16(Y) || !aligned16(up_dY) || (dY_out && !aligned16(dY_out)))
        return BITLOGIC_ERR_ALIGN;
    GradIn gi{};
    gi.off = up_off;
    gi.edge = up_edge;
    gi.Y = Y;
    gi.up_conn = up_conn;
    gi.up_theta = up_theta;
    gi.up_w = up_w;
    gi.up_dY = up_dY;
    gi.up_group = up_group;
    return run_through<TX>(up_k, X, w_in, B, conn, theta, w, k, gi, node, dtheta, dY_out, stream);
}

extern "C" int bitlogic_lut_backward_through(const float* X, int32_t w_in, int64_t B, const int32_t* conn,
                                             const float* theta, int32_t w, int32_t k, int32_t node,
                                             const float* Y, const int32_t* up_conn, const float* up_theta,
                                             int32_t up_w, int32_t up_k, const float* up_dY, int32_t up_group,
                                             const int32_t* up_off, const int32_t* up_edge, float* dtheta,
                                             float* dY_out, cudaStream_t stream) {
    return backward_through<float>(X, w_in, B, conn, theta, w, k, node, Y, up_conn, up_theta, up_w, up_k, up_dY,
                                   up_group, up_off, up_edge, dtheta, dY_out, stream);
}

extern "C" int bitlogic_lut_backward_through_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                                                const float* theta, int32_t w, int32_t k, int32_t node,
                                                const float* Y, const int32_t* up_conn, const float* up_theta,
                                                int32_t up_w, int32_t up_k, const float* up_dY, int32_t up_group,
                                                const int32_t* up_off, const int32_t* up_edge, float* dtheta,
                                                float* dY_out, cudaStream_t stream) {
    return backward_through<uint8_t>(X, w_in, B, conn, theta, w, k, node, Y, up_conn, up_theta, up_w, up_k, up_dY,
                                     up_group, up_off, up_edge, dtheta, dY_out, stream);
}

namespace {
int backward_bytes(const void* X, int32_t w_in, int64_t B, const int32_t* conn, const float* theta, int32_t w,
                   int32_t k, int32_t node, const float* dY, int32_t dy_group, const float* up_terms,
                   const int32_t* up_off, const int32_t* up_edge, int32_t up_edges, float* dtheta, float* dY_out,
                   bool bits, const int32_t* order, cudaStream_t stream) {
    int st = check_common(X, w_in, B, conn, theta, w, k, node, dtheta);
    if (st) return st;
    const bool terms = up_terms != nullptr;
    if (B > 0 && terms == (dY != nullptr)) return BITLOGIC_ERR_NULL;   // exactly one source
    if (terms) {
        if (!up_off) return BITLOGIC_ERR_NULL;
        if (up_edges < 0) return BITLOGIC_ERR_SHAPE;
    } else if (dy_group < 1 || dy_group > w || w % dy_group != 0) {
        return BITLOGIC_ERR_SHAPE;
    }
    if (B == 0) {
        if (cudaMemsetAsync(dtheta, 0, sizeof(float) * (size_t)w * ((size_t)1 << k), stream) != cudaSuccess)
            return BITLOGIC_ERR_CUDA;
        return BITLOGIC_OK;
    }
    if (B % 4 != 0 || !aligned16(X) || !aligned16(terms ? up_terms : dY) || (dY_out && !aligned16(dY_out)))
        return BITLOGIC_ERR_ALIGN;
    GradIn gi{};
    gi.dY = dY;
    gi.group = dy_group;
    gi.terms = up_terms;
    gi.n_terms = up_edges;
    gi.off = up_off;
    gi.edge = up_edge;
#define BITLOGIC_BYTES_K(K)                                                                           \
    return bits ? launch_bytes<K, true>(terms, X, w_in, B, conn, theta, w, gi, dtheta, dY_out, order, stream) \
                : launch_bytes<K, false>(terms, X, w_in, B, conn, theta, w, gi, dtheta, dY_out, order, stream)
    switch (k) {
        case 1: BITLOGIC_BYTES_K(1);
        case 2: BITLOGIC_BYTES_K(2);
        case 3: BITLOGIC_BYTES_K(3);
        case 4: BITLOGIC_BYTES_K(4);
        case 5: BITLOGIC_BYTES_K(5);
        default: BITLOGIC_BYTES_K(6);
    }
#undef BITLOGIC_BYTES_K
}
}  // namespace

extern "C" int bitlogic_lut_backward_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                                        const float* theta, int32_t w, int32_t k, int32_t node,
                                        const float* dY, int32_t dy_group, const float* up_terms,
                                        const int32_t* up_off, const int32_t* up_edge, int32_t up_edges,
                                        float* dtheta, float* dY_out, cudaStream_t stream) {
    return backward_bytes(X, w_in, B, conn, theta, w, k, node, dY, dy_group, up_terms, up_off, up_edge, up_edges,
                          dtheta, dY_out, false, nullptr, stream);
}

extern "C" int bitlogic_lut_backward_bitrows(const uint32_t* X, int32_t w_in, int64_t B, const int32_t* conn,
                                             const float* theta, int32_t w, int32_t k, int32_t node,
                                             const float* dY, int32_t dy_group, const float* up_terms,
                                             const int32_t* up_off, const int32_t* up_edge, int32_t up_edges,
                                             const int32_t* order, float* dtheta, float* dY_out,
                                             cudaStream_t stream) {
    return backward_bytes(X, w_in, B, conn, theta, w, k, node, dY, dy_group, up_terms, up_off, up_edge, up_edges,
                          dtheta, dY_out, true, order, stream);
}
