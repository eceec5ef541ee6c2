// Group-sum head with temperature and softmax cross-entropy (paper §3
// "Encoders and heads": popcount GroupSum; §4 "Training": cross-entropy on
// the raw head logits, averaged over the batch).
//
//   logits[s][c] = (sum_{j in group c} Y[j][s]) / tau,  group c = [c*g, (c+1)*g)
//   loss         = mean_s (logsumexp(logits[s]) - logits[s][label_s])
//   dY[j][s]     = ((softmax(logits[s])[c(j)] - [c(j) == label_s]) / B) / tau
//
// Two short kernels (three when the per-node dY is requested): group sums
// (lanes over samples, warps over the rows of a group), per-sample softmax
// (one warp per sample) whose last block to finish also takes the batch mean,
// and the broadcast of dlogit/tau over each group's rows.  Each kernel after
// the first is a programmatic dependent launch, so it is scheduled while the
// one before it drains.  Every reduction runs in a fixed order.
#include <cfloat>
#include <mutex>
#include <vector>

#include <cuda.h>

#include "common.cuh"

namespace bitlogic {
namespace {

constexpr int kSumWarps = 8;

__global__ void __launch_bounds__(kSumWarps * 32)
head_group_sum_kernel(const float* __restrict__ Y, long long B, int C, int g, float tau,
                      float* __restrict__ logits, unsigned int* __restrict__ done) {
    __shared__ float part[kSumWarps][32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    dependent_kernel_start();
    if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) *done = 0u;   // the softmax's block count
    const int c = blockIdx.x;
    const long long s = (long long)blockIdx.y * 32 + lane;
    float acc = 0.f;
    if (s < B) {
        const long long j0 = (long long)c * g;
        int r = warp;
#pragma unroll 4
        for (; r < g; r += kSumWarps) acc += __ldg(Y + (j0 + r) * B + s);
    }
    part[warp][lane] = acc;
    __syncthreads();
    if (warp == 0 && s < B) {
        float t = 0.f;
#pragma unroll
        for (int q = 0; q < kSumWarps; ++q) t += part[q][lane];
        logits[s * C + c] = t / tau;
    }
}

// Vector form (B % 4 == 0, 16-byte aligned Y): one block of 32 warps per
// (class, row split, 128 samples), lane = 4 consecutive samples, warp r sums
// rows r, r + 32, ... of the split with 16-byte loads, then thread t adds the
// 32 warps' partial sums of sample t in order.  With one split the block
// writes the logits; with several (so that enough blocks pull from HBM) it
// writes the split's sum, and the softmax kernel adds the splits in order.
#ifndef BITLOGIC_SUM_VEC_WARPS
#define BITLOGIC_SUM_VEC_WARPS 16
#endif
constexpr int kSumVecWarps = BITLOGIC_SUM_VEC_WARPS;
constexpr int kMaxRowSplits = 4;

__global__ void __launch_bounds__(kSumVecWarps * 32)
head_group_sum_vec_kernel(const float* __restrict__ Y, long long B, int C, int g, float tau,
                          float* __restrict__ logits, float* __restrict__ split_sums, int splits,
                          int rows_per_split, unsigned int* __restrict__ done) {
    __shared__ __align__(16) float part[kSumVecWarps][128];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    dependent_kernel_start();
    if (blockIdx.x == 0 && blockIdx.y == 0 && threadIdx.x == 0) *done = 0u;   // the softmax's block count
    const int c = blockIdx.x / splits, rs = blockIdx.x - c * splits;
    const int r0 = rs * rows_per_split, r1 = min(g, r0 + rows_per_split);
    const long long s4 = (long long)blockIdx.y * 128 + 4 * lane;
    float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
    if (s4 < B) {   // B % 4 == 0: all four samples are in range
        const float* base = Y + (long long)c * g * B + s4;
#pragma unroll 4
        for (int r = r0 + warp; r < r1; r += kSumVecWarps) {
            const float4 v = __ldg(reinterpret_cast<const float4*>(base + (long long)r * B));
            acc.x += v.x;
            acc.y += v.y;
            acc.z += v.z;
            acc.w += v.w;
        }
    }
    *reinterpret_cast<float4*>(&part[warp][4 * lane]) = acc;
    __syncthreads();
    if (threadIdx.x < 128) {
        const long long s = (long long)blockIdx.y * 128 + threadIdx.x;
        float t = 0.f;
#pragma unroll 8
        for (int q = 0; q < kSumVecWarps; ++q) t += part[q][threadIdx.x];
        if (s < B) {
            if (splits == 1) logits[s * C + c] = t / tau;
            else split_sums[((long long)rs * B + s) * C + c] = t;
        }
    }
}

__device__ __forceinline__ float warp_max(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmaxf(v, __shfl_xor_sync(0xffffffffu, v, o));
    return v;
}

__device__ __forceinline__ float warp_sum(float v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

constexpr int kSoftWarps = 8;
constexpr int kSoftRegs = 4;   // classes per lane held in registers (C <= 128)

// One warp per sample.  The block adds its samples' losses in warp order and
// publishes the sum in block_sums; the last block to finish (a device-wide
// count in `done`, zeroed by the group-sum kernel that runs before) adds the
// blocks' sums in index order and writes the batch mean: one pass, no
// separate reduction launch, and a fixed summation order.  Up to 128 classes
// a lane keeps its classes' logits (c = lane + 32 j) in registers; wider heads
// read them back from memory.  Data of the group-sum kernel is read past L1.
__global__ void __launch_bounds__(kSoftWarps * 32)
head_softmax_kernel(float* __restrict__ logits, long long B, int C,
                    const int* __restrict__ labels, float* __restrict__ dlogit,
                    float* __restrict__ block_sums, unsigned int* __restrict__ done, float* __restrict__ loss,
                    float tau, float* __restrict__ dYg, const float* __restrict__ split_sums, int splits) {
    __shared__ float part[kSoftWarps];
    __shared__ bool last;
    __shared__ float red[kSoftWarps * 32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const long long s = (long long)blockIdx.x * kSoftWarps + warp;
    dependent_kernel_start();
    float li = 0.f;
    if (s < B) {
        int lab = __ldg(labels + s);
        if (lab < 0 || lab >= C) {
            if (lane == 0) flag_index_error();
            lab = 0;
        }
        const float invB = 1.0f / (float)B;
        float* l = logits + s * C;
        if (C <= 32 * kSoftRegs) {
            float v[kSoftRegs];
#pragma unroll
            for (int q = 0; q < kSoftRegs; ++q) {
                const int c = lane + 32 * q;
                v[q] = -FLT_MAX;
                if (c < C) {
                    if (split_sums) {   // logits from the row splits' sums, added in split order
                        float t = 0.f;
                        for (int rs = 0; rs < splits; ++rs) t += __ldcg(split_sums + ((long long)rs * B + s) * C + c);
                        v[q] = t / tau;
                        l[c] = v[q];
                    } else {
                        v[q] = __ldcg(l + c);
                    }
                }
            }
            float m = -FLT_MAX;
#pragma unroll
            for (int q = 0; q < kSoftRegs; ++q)
                if (lane + 32 * q < C) m = fmaxf(m, v[q]);
            m = warp_max(m);
            float z = 0.f;
#pragma unroll
            for (int q = 0; q < kSoftRegs; ++q)
                if (lane + 32 * q < C) z += expf(v[q] - m);
            z = warp_sum(z);
            const float lse = m + logf(z);
            float vl = 0.f;
#pragma unroll
            for (int q = 0; q < kSoftRegs; ++q)
                if (q == (lab >> 5)) vl = v[q];
            li = lse - __shfl_sync(0xffffffffu, vl, lab & 31);
#pragma unroll
            for (int q = 0; q < kSoftRegs; ++q) {
                const int c = lane + 32 * q;
                if (c < C) {
                    const float p = expf(v[q] - lse);
                    const float dl = (p - (c == lab ? 1.0f : 0.0f)) * invB;
                    dlogit[s * C + c] = dl;
                    if (dYg) dYg[(long long)c * B + s] = dl / tau;   // the gradient of every node of class c
                }
            }
        } else {
            if (split_sums) {
                for (int c = lane; c < C; c += 32) {
                    float t = 0.f;
                    for (int rs = 0; rs < splits; ++rs) t += __ldcg(split_sums + ((long long)rs * B + s) * C + c);
                    l[c] = t / tau;
                }
                __syncwarp();
            }
            float m = -FLT_MAX;
            for (int c = lane; c < C; c += 32) m = fmaxf(m, __ldcg(l + c));
            m = warp_max(m);
            float z = 0.f;
            for (int c = lane; c < C; c += 32) z += expf(__ldcg(l + c) - m);
            z = warp_sum(z);
            const float lse = m + logf(z);
            li = lse - __ldcg(l + lab);
            for (int c = lane; c < C; c += 32) {
                const float p = expf(__ldcg(l + c) - lse);
                const float dl = (p - (c == lab ? 1.0f : 0.0f)) * invB;
                dlogit[s * C + c] = dl;
                if (dYg) dYg[(long long)c * B + s] = dl / tau;
            }
        }
    }
    if (lane == 0) part[warp] = li;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
#pragma unroll
        for (int q = 0; q < kSoftWarps; ++q) t += part[q];
        block_sums[blockIdx.x] = t;
        __threadfence();   // the sum is visible before the count says so
        last = atomicAdd(done, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (!last) return;
    // last block: the batch mean from every block's sum (read past L1)
    float acc = 0.f;
    for (unsigned i = threadIdx.x; i < gridDim.x; i += kSoftWarps * 32) acc += __ldcg(block_sums + i);
    red[threadIdx.x] = acc;
    __syncthreads();
    for (int o = kSoftWarps * 16; o > 0; o >>= 1) {
        if (threadIdx.x < o) red[threadIdx.x] += red[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0) {
        loss[0] = red[0] / (float)B;
        *done = 0u;
    }
}

// dY[j][s] = dlogit[s][j / g] / tau: thread per sample, each block a run of
// kRows rows, so stores along the batch are coalesced.
constexpr int kDyThreads = 128;
constexpr int kDyRows = 32;

__global__ void __launch_bounds__(kDyThreads)
head_dy_kernel(const float* __restrict__ dlogit, long long B, int C, int g, int w, float tau,
               float* __restrict__ dY) {
    dependent_kernel_start();
    const long long s = (long long)blockIdx.y * kDyThreads + threadIdx.x;
    if (s >= B) return;
    const int j0 = blockIdx.x * kDyRows;
    const int j1 = min(w, j0 + kDyRows);
    int c = j0 / g;
    int cend = (c + 1) * g;
    float v = __ldg(dlogit + s * C + c) / tau;
    for (int j = j0; j < j1; ++j) {
        if (j >= cend) {
            ++c;
            cend += g;
            v = __ldg(dlogit + s * C + c) / tau;
        }
        dY[(long long)j * B + s] = v;
    }
}

size_t align_up(size_t v) { return (v + 255) & ~(size_t)255; }

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(head)

extern "C" size_t bitlogic_head_loss_workspace(int64_t B, int32_t C) {
    if (B <= 0 || C <= 0) return 0;
    const size_t bc = (size_t)B * (size_t)C * sizeof(float);
    // dlogit [B][C], the softmax blocks' loss sums [<= B], logits [B][C]
    // (used when the caller passes no logits buffer), the row splits' sums
    // [splits][B][C], the softmax's block count
    return align_up(bc) + align_up((size_t)B * sizeof(float)) + align_up(bc) + align_up(kMaxRowSplits * bc) +
           align_up(sizeof(unsigned int));
}

extern "C" int bitlogic_head_loss_ex(const float* Y, int32_t w, int64_t B, int32_t C, float tau,
                                     const int32_t* labels, float* logits, float* loss, float* dY,
                                     float* dY_grouped, void* workspace, size_t ws_bytes,
                                     cudaStream_t stream) {
    if (!Y || !labels || !loss || !workspace) return BITLOGIC_ERR_NULL;
    if (w <= 0 || B <= 0 || C <= 0 || w % C != 0 || !(tau > 0.f)) return BITLOGIC_ERR_SHAPE;
    if (B > 0x7fffffffLL / (C > 0 ? C : 1)) return BITLOGIC_ERR_SHAPE;
    if (!aligned16(workspace)) return BITLOGIC_ERR_ALIGN;
    if (ws_bytes < bitlogic_head_loss_workspace(B, C)) return BITLOGIC_ERR_WORKSPACE;
    const long long sb = (B + 31) / 32;
    const long long gy = (B + kDyThreads - 1) / kDyThreads;
    if (sb > 65535 || gy > 65535) return BITLOGIC_ERR_SHAPE;
    const int g = w / C;
    char* ws = static_cast<char*>(workspace);
    const size_t bc = (size_t)B * (size_t)C * sizeof(float);
    float* dlogit = reinterpret_cast<float*>(ws);
    float* block_sums = reinterpret_cast<float*>(ws + align_up(bc));
    float* lg = logits ? logits : reinterpret_cast<float*>(ws + align_up(bc) + align_up((size_t)B * 4));
    float* split_sums = reinterpret_cast<float*>(ws + align_up(bc) + align_up((size_t)B * 4) + align_up(bc));
    unsigned int* done = reinterpret_cast<unsigned int*>(ws + align_up(bc) + align_up((size_t)B * 4) + align_up(bc) +
                                                         align_up(kMaxRowSplits * bc));
    int splits = 1;

    if (B % 4 == 0 && aligned16(Y)) {
        // split the rows of a class while the doubled grid still fits one
        // wave of resident blocks, keeping at least 4 rows per warp
        const long long nsb = (B + 127) / 128;
        const long long resident = (long long)(2048 / (kSumVecWarps * 32)) * sm_count();
        while (splits < kMaxRowSplits && (long long)C * (2 * splits) * nsb <= resident &&
               g / (2 * splits) >= 4 * kSumVecWarps)
            splits *= 2;
        const int rows_per_split = (g + splits - 1) / splits;
        if ((long long)C * splits > 0x7fffffffll || nsb > 65535) return BITLOGIC_ERR_SHAPE;
        (void)launch_dependent(head_group_sum_vec_kernel, dim3((unsigned)(C * splits), (unsigned)nsb),
                               kSumVecWarps * 32, 0, stream, Y, B, C, g, tau, lg, split_sums, splits,
                               rows_per_split, done);
    } else
        (void)launch_dependent(head_group_sum_kernel, dim3((unsigned)C, (unsigned)sb), kSumWarps * 32, 0, stream, Y,
                               B, C, g, tau, lg, done);
    if (launch_status()) return BITLOGIC_ERR_CUDA;
    if (launch_dependent(head_softmax_kernel, (unsigned)((B + kSoftWarps - 1) / kSoftWarps), kSoftWarps * 32, 0,
                         stream, lg, B, C, labels, dlogit, block_sums, done, loss, tau,
                         dY_grouped, splits > 1 ? split_sums : nullptr, splits) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    if (dY && launch_dependent(head_dy_kernel, dim3((unsigned)((w + kDyRows - 1) / kDyRows), (unsigned)gy),
                               kDyThreads, 0, stream, dlogit, B, C, g, w, tau, dY) != cudaSuccess)
        return BITLOGIC_ERR_CUDA;
    return launch_status();
}

extern "C" int bitlogic_head_loss(const float* Y, int32_t w, int64_t B, int32_t C, float tau,
                                  const int32_t* labels, float* logits, float* loss, float* dY,
                                  void* workspace, size_t ws_bytes, cudaStream_t stream) {
    return bitlogic_head_loss_ex(Y, w, B, C, tau, labels, logits, loss, dY, nullptr, workspace,
                                 ws_bytes, stream);
}

// ------------------------------------- allocation-free variant of the head --
//
// For callers that cannot allocate device memory themselves (see the header):
// the head's workspace lives in a fixed file-scope device array instead of a
// caller buffer.  Every GPU that loads the library reserves the array until
// the process exits; all calls share it.

namespace {

constexpr size_t kNoAllocScratchBytes = (size_t)8 << 20;   // 8 MiB
static __device__ __align__(256) unsigned char g_head_scratch[kNoAllocScratchBytes];

// The array is a global of the library's module, and a module is loaded once
// per CUDA context, so its device address belongs to a context: a device
// reset or a context other than the primary one loads the module again,
// possibly at another address.  The address is therefore looked up once per
// context (with the calling thread's context current) and cached under the
// context's unique id.  The host-side name g_head_scratch is only a stand-in
// and is never passed to a kernel.
using CtxGetCurrentFn = CUresult (*)(CUcontext*);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long*);

struct ScratchAddr {
    unsigned long long ctx_id;
    void* addr;
};

std::mutex g_scratch_mutex;
std::vector<ScratchAddr> g_scratch_addr;
CtxGetCurrentFn g_ctx_get_current = nullptr;
CtxGetIdFn g_ctx_get_id = nullptr;
bool g_ctx_fns_looked_up = false;

// Unique id of the calling thread's current context (0 if there is none, or
// the driver entry points cannot be found: then nothing is cached).
unsigned long long current_context_id() {
    if (!g_ctx_fns_looked_up) {
        g_ctx_fns_looked_up = true;
        void* f1 = nullptr;
        void* f2 = nullptr;
        cudaDriverEntryPointQueryResult q1 = cudaDriverEntryPointSymbolNotFound, q2 = q1;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &f1, 12000, cudaEnableDefault, &q1) ==
                cudaSuccess && q1 == cudaDriverEntryPointSuccess &&
            cudaGetDriverEntryPointByVersion("cuCtxGetId", &f2, 12000, cudaEnableDefault, &q2) ==
                cudaSuccess && q2 == cudaDriverEntryPointSuccess) {
            g_ctx_get_current = reinterpret_cast<CtxGetCurrentFn>(f1);
            g_ctx_get_id = reinterpret_cast<CtxGetIdFn>(f2);
        }
    }
    if (!g_ctx_get_current || !g_ctx_get_id) return 0;
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (g_ctx_get_current(&ctx) != CUDA_SUCCESS || !ctx) return 0;
    if (g_ctx_get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of the scratch array in the current context.
int noalloc_scratch(void** out) {
    std::lock_guard<std::mutex> lock(g_scratch_mutex);
    unsigned long long id = current_context_id();
    if (id) {
        for (const ScratchAddr& e : g_scratch_addr)
            if (e.ctx_id == id) {
                *out = e.addr;
                return BITLOGIC_OK;
            }
    }
    // the lookup makes the device's primary context current if no context is
    void* p = nullptr;
    if (cudaGetSymbolAddress(&p, g_head_scratch) != cudaSuccess || !p) return BITLOGIC_ERR_CUDA;
    if (!id) id = current_context_id();
    if (id) g_scratch_addr.push_back({id, p});
    *out = p;
    return BITLOGIC_OK;
}

}  // namespace

extern "C" int bitlogic_head_loss_noalloc(const float* Y, int32_t w, int64_t B, int32_t C, float tau,
                                          const int32_t* labels, float* logits, float* loss,
                                          float* dY, cudaStream_t stream) {
    if (B <= 0 || C <= 0 || B > 0x7fffffffLL / C) return BITLOGIC_ERR_SHAPE;
    if (bitlogic_head_loss_workspace(B, C) > kNoAllocScratchBytes) return BITLOGIC_ERR_TOO_LARGE;
    void* ws = nullptr;
    const int st = noalloc_scratch(&ws);
    if (st) return st;
    // every byte of the workspace that the kernels read is written first in
    // the same call, so nothing has to be cleared between calls
    return bitlogic_head_loss_ex(Y, w, B, C, tau, labels, logits, loss, dY, nullptr, ws,
                                 kNoAllocScratchBytes, stream);
}
