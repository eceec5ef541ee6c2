// Learnable routing (paper §3, the paragraph on connectivity: each node
// slot selects its input from a candidate pool through a
// selection that is differentiable in training and snapped to a sparse
// mapping at discretization; App. A "Initialization": pools drawn uniformly,
// routing logits zero).
//
// Slot e = j*k + i of a layer has Kc candidates cand[e][m] and logits
// r[e][m]; its input is the expected selection
//   p_e = softmax(r_e),   Xr[e][s] = sum_m p_e[m] X[cand[e][m]][s],
// written as rows [w*k][B] that the LUT kernels then read through the
// identity connectivity (node j's slot i is row j*k + i).  The backward
// takes the slot inputs' gradient G = dL/dXr (the per-edge terms of the LUT
// backward over those rows):
//   dr[e][m] = p_e[m] (A_m - sum_m' p_e[m'] A_m'),   A_m = sum_s G[e][s] X[cand[e][m]][s]
//   dX[c][s] = sum over candidate edges (e, m) with cand[e][m] == c, in
//              increasing e*Kc + m, of p_e[m] G[e][s]   (CSR, no atomics).
//
// Layer inputs are fp32 rows or byte rows (the encoder's 0/1 wires); the
// forward reads byte rows 16 samples per lane and load (the dr kernel keeps
// 4: at 16 it needs twice the registers and measured slower).
//
// Kernels: the slot's softmax is computed by its warp (candidate m on lane
// m, Kc <= 32) and held in registers; the gathers stream KC 16-byte loads per
// lane and step (KC = Kc rounded up to a power of two, the padding having
// weight 0 on the slot's first candidate).  The pools of a layer read a few
// thousand distinct rows, which stay in L2.
#include <type_traits>

#include "common.cuh"

namespace bitlogic {
namespace {

constexpr int kRouteWarps = 8;

__device__ __forceinline__ float4 ldg4r(const float* p) { return __ldg(reinterpret_cast<const float4*>(p)); }

// Layer inputs come as fp32 rows or as byte rows (the encoder's 0/1 wires,
// a quarter of the bytes to gather): one value and four consecutive values
// of a row, as floats.
__device__ __forceinline__ float in_value(const float* p) { return __ldg(p); }
__device__ __forceinline__ float in_value(const uint8_t* p) { return (float)__ldg(p); }
__device__ __forceinline__ float4 in_quad(const float* p) { return ldg4r(p); }
__device__ __forceinline__ float4 in_quad(const uint8_t* p) {
    const uint32_t w = __ldg(reinterpret_cast<const uint32_t*>(p));
    return make_float4((float)(w & 0xffu), (float)((w >> 8) & 0xffu), (float)((w >> 16) & 0xffu), (float)(w >> 24));
}

// Softmax of the slot's logits on lanes m < Kc (other lanes 0), the lane's
// candidate row (range-checked; a bad index is read as row 0 and flagged).
__device__ __forceinline__ void slot_softmax(const int* __restrict__ cand, const float* __restrict__ r,
                                             long long e, int Kc, int w_in, int lane, float& p, int& c) {
    float z = -INFINITY;
    c = 0;
    if (lane < Kc) {
        z = __ldg(r + e * Kc + lane);
        c = __ldg(cand + e * Kc + lane);
        if ((unsigned)c >= (unsigned)w_in) {
            flag_index_error();
            c = 0;
        }
    }
    float mx = z;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) mx = fmaxf(mx, __shfl_xor_sync(0xffffffffu, mx, o));
    const float ez = lane < Kc ? expf(z - mx) : 0.f;
    float sum = ez;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
    p = ez / sum;
}

// Forward, vector path (B % 4 == 0, 16-byte aligned X and Xr): one warp per
// (slot, batch chunk), 4 consecutive samples per lane and step.
template <int KC, typename T>
__global__ void __launch_bounds__(kRouteWarps * 32)
route_forward_vec_kernel(const T* __restrict__ X, int w_in, long long B, const int* __restrict__ cand,
                         const float* __restrict__ r, long long slots, int Kc, float* __restrict__ Xr,
                         float* __restrict__ prob, long long chunk) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long e = (long long)blockIdx.x * kRouteWarps + warp;
    if (e >= slots) return;
    float p;
    int c;
    slot_softmax(cand, r, e, Kc, w_in, lane, p, c);
    if (prob && blockIdx.y == 0 && lane < Kc) prob[e * Kc + lane] = p;
    float pm[KC];
    const T* row[KC];
    const int c0 = __shfl_sync(0xffffffffu, c, 0);
#pragma unroll
    for (int m = 0; m < KC; ++m) {
        pm[m] = __shfl_sync(0xffffffffu, p, m & 31);
        const int cm = __shfl_sync(0xffffffffu, c, m & 31);
        row[m] = X + (long long)(m < Kc ? cm : c0) * B;
        if (m >= Kc) pm[m] = 0.f;
    }
    const long long s0 = (long long)blockIdx.y * chunk;
    const long long s1 = min(B, s0 + chunk);
    float* out = Xr + e * B;
    for (long long s = s0 + 4 * lane; s < s1; s += 128) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        constexpr int G = KC < 8 ? KC : 8;   // loads issued together
#pragma unroll
        for (int m0 = 0; m0 < KC; m0 += G) {
            float4 v[G];
#pragma unroll
            for (int u = 0; u < G; ++u) v[u] = in_quad(row[m0 + u] + s);
#pragma unroll
            for (int u = 0; u < G; ++u) {
                const float q = pm[m0 + u];
                acc.x = fmaf(q, v[u].x, acc.x);
                acc.y = fmaf(q, v[u].y, acc.y);
                acc.z = fmaf(q, v[u].z, acc.z);
                acc.w = fmaf(q, v[u].w, acc.w);
            }
        }
        *reinterpret_cast<float4*>(out + s) = acc;
    }
}

// Forward over byte rows, 16 consecutive samples per lane and step (one
// 16-byte load per candidate row: a quarter of the load instructions of the
// 4-sample form).  Needs B % 16 == 0 and 16-byte aligned X and Xr.
template <int KC>
__global__ void __launch_bounds__(kRouteWarps * 32)
route_forward_bytes16_kernel(const uint8_t* __restrict__ X, int w_in, long long B, const int* __restrict__ cand,
                             const float* __restrict__ r, long long slots, int Kc, float* __restrict__ Xr,
                             float* __restrict__ prob, long long chunk) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long e = (long long)blockIdx.x * kRouteWarps + warp;
    if (e >= slots) return;
    float p;
    int c;
    slot_softmax(cand, r, e, Kc, w_in, lane, p, c);
    if (prob && blockIdx.y == 0 && lane < Kc) prob[e * Kc + lane] = p;
    float pm[KC];
    const uint8_t* row[KC];
    const int c0 = __shfl_sync(0xffffffffu, c, 0);
#pragma unroll
    for (int m = 0; m < KC; ++m) {
        pm[m] = __shfl_sync(0xffffffffu, p, m & 31);
        const int cm = __shfl_sync(0xffffffffu, c, m & 31);
        row[m] = X + (long long)(m < Kc ? cm : c0) * B;
        if (m >= Kc) pm[m] = 0.f;
    }
    const long long s0 = (long long)blockIdx.y * chunk;
    const long long s1 = min(B, s0 + chunk);
    float* out = Xr + e * B;
    for (long long s = s0 + 16 * lane; s < s1; s += 512) {
        float acc[16];
#pragma unroll
        for (int t = 0; t < 16; ++t) acc[t] = 0.f;
        constexpr int G = KC < 4 ? KC : 4;   // loads issued together
#pragma unroll
        for (int m0 = 0; m0 < KC; m0 += G) {
            uint4 v[G];
#pragma unroll
            for (int u = 0; u < G; ++u) v[u] = __ldg(reinterpret_cast<const uint4*>(row[m0 + u] + s));
#pragma unroll
            for (int u = 0; u < G; ++u) {
                const float q = pm[m0 + u];
                const uint32_t w[4] = {v[u].x, v[u].y, v[u].z, v[u].w};
#pragma unroll
                for (int t = 0; t < 16; ++t)
                    acc[t] = fmaf(q, (float)((w[t >> 2] >> (8 * (t & 3))) & 0xffu), acc[t]);
            }
        }
#pragma unroll
        for (int t = 0; t < 16; t += 4)
            *reinterpret_cast<float4*>(out + s + t) = make_float4(acc[t], acc[t + 1], acc[t + 2], acc[t + 3]);
    }
}

// Forward, scalar path (any B and alignment): one sample per lane and step.
template <typename T>
__global__ void __launch_bounds__(kRouteWarps * 32)
route_forward_kernel(const T* __restrict__ X, int w_in, long long B, const int* __restrict__ cand,
                     const float* __restrict__ r, long long slots, int Kc, float* __restrict__ Xr,
                     float* __restrict__ prob, long long chunk) {
    __shared__ float sp[kRouteWarps][32];
    __shared__ int sc[kRouteWarps][32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long e = (long long)blockIdx.x * kRouteWarps + warp;
    if (e >= slots) return;
    float p;
    int c;
    slot_softmax(cand, r, e, Kc, w_in, lane, p, c);
    if (prob && blockIdx.y == 0 && lane < Kc) prob[e * Kc + lane] = p;
    sp[warp][lane] = p;
    sc[warp][lane] = c;
    __syncwarp();
    const long long s0 = (long long)blockIdx.y * chunk;
    const long long s1 = min(B, s0 + chunk);
    for (long long s = s0 + lane; s < s1; s += 32) {
        float acc = 0.f;
        for (int m = 0; m < Kc; ++m) acc = fmaf(sp[warp][m], in_value(X + (long long)sc[warp][m] * B + s), acc);
        Xr[e * B + s] = acc;
    }
}

// dr: one warp per slot over the whole batch.  Each lane accumulates its
// samples' A_m (m < KC), then the warp sums every A_m with a fixed butterfly.
// The vector path holds the candidate rows as 32-bit offsets in units of 4
// samples (needs w_in B / 4 < 2^32) and is held to 64 registers (four blocks
// per SM; two for 32 candidates), so that more warps keep gathers in flight.
template <int KC, bool VEC, typename T>
__global__ void __launch_bounds__(kRouteWarps * 32, VEC ? (KC <= 16 ? 4 : 2) : 1)
route_dr_kernel(const T* __restrict__ X, int w_in, long long B, const int* __restrict__ cand,
                const float* __restrict__ r, long long slots, int Kc, const float* __restrict__ G,
                float* __restrict__ dr) {
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long e = (long long)blockIdx.x * kRouteWarps + warp;
    if (e >= slots) return;
    float p;
    int c;
    slot_softmax(cand, r, e, Kc, w_in, lane, p, c);
    const int c0 = __shfl_sync(0xffffffffu, c, 0);
    float A[KC];
#pragma unroll
    for (int m = 0; m < KC; ++m) A[m] = 0.f;
    const float* g = G + e * B;
    if constexpr (VEC) {
        const unsigned B4 = (unsigned)(B / 4);
        unsigned row[KC];
#pragma unroll
        for (int m = 0; m < KC; ++m) {
            const int cm = __shfl_sync(0xffffffffu, c, m & 31);
            row[m] = (unsigned)(m < Kc ? cm : c0) * B4 + (unsigned)lane;
        }
        for (unsigned s4 = 0; s4 < B4; s4 += 32) {
            if (s4 + lane >= B4) break;
            const float4 gv = ldg4r(g + 4 * (long long)(s4 + lane));
            constexpr int GR = KC < 8 ? KC : 8;
#pragma unroll
            for (int m0 = 0; m0 < KC; m0 += GR) {
                float4 v[GR];
#pragma unroll
                for (int u = 0; u < GR; ++u) v[u] = in_quad(X + 4 * (size_t)(row[m0 + u] + s4));
#pragma unroll
                for (int u = 0; u < GR; ++u) {
                    float a = A[m0 + u];
                    a = fmaf(gv.x, v[u].x, a);
                    a = fmaf(gv.y, v[u].y, a);
                    a = fmaf(gv.z, v[u].z, a);
                    a = fmaf(gv.w, v[u].w, a);
                    A[m0 + u] = a;
                }
            }
        }
    } else {
        const T* row[KC];
#pragma unroll
        for (int m = 0; m < KC; ++m) {
            const int cm = __shfl_sync(0xffffffffu, c, m & 31);
            row[m] = X + (long long)(m < Kc ? cm : c0) * B;
        }
        for (long long s = lane; s < B; s += 32) {
            const float gv = __ldg(g + s);
#pragma unroll
            for (int m = 0; m < KC; ++m) A[m] = fmaf(gv, in_value(row[m] + s), A[m]);
        }
    }
#pragma unroll
    for (int m = 0; m < KC; ++m) {
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) A[m] += __shfl_xor_sync(0xffffffffu, A[m], o);
    }
    // every lane now holds every A_m; S = sum_m p_m A_m in increasing m
    float S = 0.f, mine = 0.f;
#pragma unroll
    for (int m = 0; m < KC; ++m) {
        const float pm = __shfl_sync(0xffffffffu, p, m & 31);
        if (m < Kc) S = fmaf(pm, A[m], S);
        if (m == lane) mine = A[m];
    }
    if (lane < Kc) dr[e * Kc + lane] = p * (mine - S);
}

// dX[c][s] = sum over the CSR positions q of input c (increasing q) of
// prob[id_q] G[id_q / Kc][s], id_q = csr_edge[q] (candidate edge e*Kc + m).
// Warp w of a block owns input row 8 blockIdx.x + w and the block's batch
// slice (128 samples on the vector path, 32 otherwise); the grid runs the
// rows fastest, so the blocks in flight share one slice of G, which stays
// in L2 while every G row is read by about Kc input rows.  The row's first
// 32 edge ids and weights are held one per lane.
constexpr int kRdxWarps = 8;

template <bool VEC>
__global__ void __launch_bounds__(kRdxWarps * 32)
route_dx_kernel(const float* __restrict__ G, long long B, const float* __restrict__ prob, int Kc,
                const int* __restrict__ off, const int* __restrict__ edge, int w_in, int nE,
                float* __restrict__ dX) {
    constexpr int SPW = VEC ? 128 : 32;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int i = blockIdx.x * kRdxWarps + warp;
    if (i >= w_in) return;
    int e0 = __ldg(off + i), e1 = __ldg(off + i + 1);
    if (e0 < 0 || e1 < e0 || e1 > nE) {
        if (lane == 0) flag_index_error();
        e0 = e1 = 0;
    }
    const int deg = e1 - e0;
    const long long s = (long long)blockIdx.y * SPW + (VEC ? 4 : 1) * lane;
    const bool in = s < B;
    // the row's positions in chunks of 32: lane u holds the G row (slot) and
    // weight of position q0 + u (slot -1: out of range, read as zero)
    constexpr int kBatch = 8;
    auto accumulate = [&](auto& acc) {
        for (int c0 = 0; c0 < deg; c0 += 32) {
            int my_slot = -1;
            float my_w = 0.f;
            if (c0 + lane < deg) {
                const int id = __ldg(edge + e0 + c0 + lane);
                if ((unsigned)id >= (unsigned)nE) {
                    flag_index_error();
                } else {
                    my_slot = id / Kc;
                    my_w = __ldg(prob + id);
                }
            }
            const int n = min(32, deg - c0);
            for (int q0 = 0; q0 < n; q0 += kBatch) {
                int slot[kBatch];
                float wt[kBatch];
#pragma unroll
                for (int u = 0; u < kBatch; ++u) {
                    slot[u] = __shfl_sync(0xffffffffu, my_slot, (q0 + u) & 31);
                    wt[u] = __shfl_sync(0xffffffffu, my_w, (q0 + u) & 31);
                    if (q0 + u >= n) slot[u] = -1;
                }
                if constexpr (VEC) {
                    float4 v[kBatch];
#pragma unroll
                    for (int u = 0; u < kBatch; ++u)
                        v[u] = (in && slot[u] >= 0) ? ldg4r(G + (long long)slot[u] * B + s)
                                                    : make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                    for (int u = 0; u < kBatch; ++u) {
                        if (q0 + u < n) {
                            acc.x = fmaf(wt[u], v[u].x, acc.x);
                            acc.y = fmaf(wt[u], v[u].y, acc.y);
                            acc.z = fmaf(wt[u], v[u].z, acc.z);
                            acc.w = fmaf(wt[u], v[u].w, acc.w);
                        }
                    }
                } else {
                    float v[kBatch];
#pragma unroll
                    for (int u = 0; u < kBatch; ++u)
                        v[u] = (in && slot[u] >= 0) ? __ldg(G + (long long)slot[u] * B + s) : 0.f;
#pragma unroll
                    for (int u = 0; u < kBatch; ++u)
                        if (q0 + u < n) acc = fmaf(wt[u], v[u], acc);
                }
            }
        }
    };
    if constexpr (VEC) {
        float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
        accumulate(acc);
        if (in) *reinterpret_cast<float4*>(dX + (long long)i * B + s) = acc;
    } else {
        float acc = 0.f;
        accumulate(acc);
        if (in) dX[(long long)i * B + s] = acc;
    }
}

__global__ void route_snap_kernel(const int* __restrict__ cand, const float* __restrict__ r, long long slots,
                                  int Kc, int* __restrict__ conn) {
    const long long e = (long long)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= slots) return;
    int best = 0;
    float bv = __ldg(r + e * Kc);
    for (int m = 1; m < Kc; ++m) {
        const float v = __ldg(r + e * Kc + m);
        if (v > bv) {
            bv = v;
            best = m;
        }
    }
    conn[e] = __ldg(cand + e * Kc + best);
}

int check_route(const void* X, int32_t w_in, int64_t B, const void* cand, const void* r, int32_t slots,
                int32_t Kc) {
    if (!cand || !r) return BITLOGIC_ERR_NULL;
    if (B > 0 && !X) return BITLOGIC_ERR_NULL;
    if (w_in <= 0 || slots <= 0 || B < 0) return BITLOGIC_ERR_SHAPE;
    if (Kc < 1 || Kc > 32 || Kc > w_in) return BITLOGIC_ERR_FANIN;
    if ((int64_t)slots * Kc > 0x7fffffffLL) return BITLOGIC_ERR_SHAPE;
    return BITLOGIC_OK;
}

template <int KC, typename T>
int launch_route_forward(const T* X, int w_in, long long B, const int* cand, const float* r, long long slots,
                         int Kc, float* Xr, float* prob, bool vec, cudaStream_t st) {
    // batch chunks of 1024 samples (8 steps per warp)
    const long long chunk = 1024;
    const long long gy = (B + chunk - 1) / chunk;
    if (gy > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((slots + kRouteWarps - 1) / kRouteWarps), (unsigned)gy);
    if (vec)
        route_forward_vec_kernel<KC, T><<<grid, kRouteWarps * 32, 0, st>>>(X, w_in, B, cand, r, slots, Kc, Xr,
                                                                           prob, chunk);
    else
        route_forward_kernel<T><<<grid, kRouteWarps * 32, 0, st>>>(X, w_in, B, cand, r, slots, Kc, Xr, prob, chunk);
    return launch_status();
}

template <int KC, typename T>
int launch_route_dr(const T* X, int w_in, long long B, const int* cand, const float* r, long long slots, int Kc,
                    const float* G, float* dr, bool vec, cudaStream_t st) {
    const unsigned blocks = (unsigned)((slots + kRouteWarps - 1) / kRouteWarps);
    if (vec)
        route_dr_kernel<KC, true, T><<<blocks, kRouteWarps * 32, 0, st>>>(X, w_in, B, cand, r, slots, Kc, G, dr);
    else
        route_dr_kernel<KC, false, T><<<blocks, kRouteWarps * 32, 0, st>>>(X, w_in, B, cand, r, slots, Kc, G, dr);
    return launch_status();
}

// Entry-point bodies shared by the fp32 and byte-row inputs.
template <int KC>
int launch_route_forward_bytes16(const uint8_t* X, int w_in, long long B, const int* cand, const float* r,
                                 long long slots, int Kc, float* Xr, float* prob, cudaStream_t st) {
    const long long chunk = 1024;
    const long long gy = (B + chunk - 1) / chunk;
    if (gy > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((slots + kRouteWarps - 1) / kRouteWarps), (unsigned)gy);
    route_forward_bytes16_kernel<KC><<<grid, kRouteWarps * 32, 0, st>>>(X, w_in, B, cand, r, slots, Kc, Xr, prob,
                                                                        chunk);
    return launch_status();
}

template <typename T>
int route_forward_impl(const T* X, int32_t w_in, int64_t B, const int32_t* cand, const float* r, int32_t slots,
                       int32_t Kc, float* Xr, float* prob, cudaStream_t stream) {
    int st = check_route(X, w_in, B, cand, r, slots, Kc);
    if (st) return st;
    if (B == 0 && !prob) return BITLOGIC_OK;
    if (B > 0 && !Xr) return BITLOGIC_ERR_NULL;
    const bool vec = (B % 4 == 0) && aligned16(X) && aligned16(Xr);
    if constexpr (std::is_same<T, uint8_t>::value) {
        if (B > 0 && B % 16 == 0 && vec) {   // byte rows: 16 samples per lane and load
            if (Kc <= 4) return launch_route_forward_bytes16<4>(X, w_in, B, cand, r, slots, Kc, Xr, prob, stream);
            if (Kc <= 8) return launch_route_forward_bytes16<8>(X, w_in, B, cand, r, slots, Kc, Xr, prob, stream);
            if (Kc <= 16)
                return launch_route_forward_bytes16<16>(X, w_in, B, cand, r, slots, Kc, Xr, prob, stream);
            return launch_route_forward_bytes16<32>(X, w_in, B, cand, r, slots, Kc, Xr, prob, stream);
        }
    }
    if (B == 0) {   // probabilities only
        route_forward_kernel<T><<<(unsigned)((slots + kRouteWarps - 1) / kRouteWarps), kRouteWarps * 32, 0,
                                  stream>>>(X, w_in, 0, cand, r, slots, Kc, Xr, prob, 1);
        return launch_status();
    }
    if (Kc <= 4) return launch_route_forward<4, T>(X, w_in, B, cand, r, slots, Kc, Xr, prob, vec, stream);
    if (Kc <= 8) return launch_route_forward<8, T>(X, w_in, B, cand, r, slots, Kc, Xr, prob, vec, stream);
    if (Kc <= 16) return launch_route_forward<16, T>(X, w_in, B, cand, r, slots, Kc, Xr, prob, vec, stream);
    return launch_route_forward<32, T>(X, w_in, B, cand, r, slots, Kc, Xr, prob, vec, stream);
}

template <typename T>
int route_dr_impl(const T* X, int32_t w_in, int64_t B, const int32_t* cand, const float* r, int32_t slots,
                  int32_t Kc, const float* G, float* dr, cudaStream_t stream) {
    const bool vec = (B % 4 == 0) && aligned16(X) && aligned16(G) &&
                     (unsigned long long)w_in * (unsigned long long)(B / 4) < (1ull << 32);
    if (Kc <= 4) return launch_route_dr<4, T>(X, w_in, B, cand, r, slots, Kc, G, dr, vec, stream);
    if (Kc <= 8) return launch_route_dr<8, T>(X, w_in, B, cand, r, slots, Kc, G, dr, vec, stream);
    if (Kc <= 16) return launch_route_dr<16, T>(X, w_in, B, cand, r, slots, Kc, G, dr, vec, stream);
    return launch_route_dr<32, T>(X, w_in, B, cand, r, slots, Kc, G, dr, vec, stream);
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(route)

extern "C" int bitlogic_route_forward(const float* X, int32_t w_in, int64_t B, const int32_t* cand, const float* r,
                                      int32_t slots, int32_t Kc, float* Xr, float* prob, cudaStream_t stream) {
    return route_forward_impl(X, w_in, B, cand, r, slots, Kc, Xr, prob, stream);
}

extern "C" int bitlogic_route_forward_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* cand,
                                         const float* r, int32_t slots, int32_t Kc, float* Xr, float* prob,
                                         cudaStream_t stream) {
    return route_forward_impl(X, w_in, B, cand, r, slots, Kc, Xr, prob, stream);
}

extern "C" int bitlogic_route_backward(const float* X, int32_t w_in, int64_t B, const int32_t* cand, const float* r,
                                       int32_t slots, int32_t Kc, const float* G, float* dr, const float* prob,
                                       const int32_t* csr_off, const int32_t* csr_edge, float* dX,
                                       cudaStream_t stream) {
    int st = check_route(X, w_in, B, cand, r, slots, Kc);
    if (st) return st;
    if (!dr) return BITLOGIC_ERR_NULL;
    if (B > 0 && !G) return BITLOGIC_ERR_NULL;
    if (dX && B > 0 && (!prob || !csr_off || !csr_edge)) return BITLOGIC_ERR_NULL;
    if (B == 0) {   // empty batch: the batch sums are zero
        if (cudaMemsetAsync(dr, 0, sizeof(float) * (size_t)slots * (size_t)Kc, stream) != cudaSuccess)
            return BITLOGIC_ERR_CUDA;
        return BITLOGIC_OK;
    }
    st = route_dr_impl(X, w_in, B, cand, r, slots, Kc, G, dr, stream);
    if (st || !dX) return st;
    const int nE = slots * Kc;
    const bool vx = (B % 4 == 0) && aligned16(G) && aligned16(dX);
    const long long per_block = vx ? 128 : 32;
    const long long gy = (B + per_block - 1) / per_block;
    if (gy > 65535) return BITLOGIC_ERR_SHAPE;
    dim3 grid((unsigned)((w_in + kRdxWarps - 1) / kRdxWarps), (unsigned)gy);
    if (vx)
        route_dx_kernel<true><<<grid, kRdxWarps * 32, 0, stream>>>(G, B, prob, Kc, csr_off, csr_edge, w_in, nE, dX);
    else
        route_dx_kernel<false><<<grid, kRdxWarps * 32, 0, stream>>>(G, B, prob, Kc, csr_off, csr_edge, w_in, nE, dX);
    return launch_status();
}

extern "C" int bitlogic_route_backward_u8(const uint8_t* X, int32_t w_in, int64_t B, const int32_t* cand,
                                          const float* r, int32_t slots, int32_t Kc, const float* G, float* dr,
                                          cudaStream_t stream) {
    int st = check_route(X, w_in, B, cand, r, slots, Kc);
    if (st) return st;
    if (!dr) return BITLOGIC_ERR_NULL;
    if (B > 0 && !G) return BITLOGIC_ERR_NULL;
    if (B == 0) {
        if (cudaMemsetAsync(dr, 0, sizeof(float) * (size_t)slots * (size_t)Kc, stream) != cudaSuccess)
            return BITLOGIC_ERR_CUDA;
        return BITLOGIC_OK;
    }
    return route_dr_impl(X, w_in, B, cand, r, slots, Kc, G, dr, stream);
}

extern "C" int bitlogic_route_snap(const int32_t* cand, const float* r, int32_t slots, int32_t Kc, int32_t* conn,
                                   cudaStream_t stream) {
    if (!cand || !r || !conn) return BITLOGIC_ERR_NULL;
    if (slots <= 0) return BITLOGIC_ERR_SHAPE;
    if (Kc < 1 || Kc > 32) return BITLOGIC_ERR_FANIN;
    route_snap_kernel<<<(unsigned)((slots + 255) / 256), 256, 0, stream>>>(cand, r, slots, Kc, conn);
    return launch_status();
}
