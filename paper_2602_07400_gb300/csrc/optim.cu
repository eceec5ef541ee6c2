// AdamW update of the table logits (paper §4 "Training": AdamW with beta1
// 0.9, beta2 0.999, eps 1e-8, constant learning rate 0.01, weight decay 0;
// the decay, when used, is decoupled).  Elementwise and bound by HBM: per
// parameter 16 bytes read (theta, m, v, grad) and 12 written; the vector
// path moves 16 bytes per load and store, in a grid-stride loop sized to the
// SMs.  The bias corrections 1 / (1 - beta^step) are formed on the host in
// double precision.
#include <cmath>

#include "common.cuh"

namespace bitlogic {
namespace {

struct AdamW {
    float lr, b1, b2, eps, wd;
    float c1, c2;   // 1 / (1 - beta1^step), 1 / (1 - beta2^step)
};

__device__ __forceinline__ void adamw_one(float& th, float& m, float& v, float g, const AdamW& a) {
    m = a.b1 * m + (1.0f - a.b1) * g;
    v = a.b2 * v + (1.0f - a.b2) * (g * g);
    const float mhat = m * a.c1;
    const float vhat = v * a.c2;
    th = th - a.lr * (mhat / (sqrtf(vhat) + a.eps) + a.wd * th);
}

__global__ void __launch_bounds__(256)
adamw_vec_kernel(float4* __restrict__ theta, float4* __restrict__ m, float4* __restrict__ v,
                 const float4* __restrict__ g, long long n4, AdamW a) {
    for (long long i = (long long)blockIdx.x * 256 + threadIdx.x; i < n4; i += (long long)gridDim.x * 256) {
        float4 th = theta[i], mm = m[i], vv = v[i];
        const float4 gg = __ldg(g + i);
        adamw_one(th.x, mm.x, vv.x, gg.x, a);
        adamw_one(th.y, mm.y, vv.y, gg.y, a);
        adamw_one(th.z, mm.z, vv.z, gg.z, a);
        adamw_one(th.w, mm.w, vv.w, gg.w, a);
        theta[i] = th;
        m[i] = mm;
        v[i] = vv;
    }
}

__global__ void __launch_bounds__(256)
adamw_kernel(float* __restrict__ theta, float* __restrict__ m, float* __restrict__ v,
             const float* __restrict__ g, long long n, AdamW a) {
    for (long long i = (long long)blockIdx.x * 256 + threadIdx.x; i < n; i += (long long)gridDim.x * 256) {
        float th = theta[i], mm = m[i], vv = v[i];
        adamw_one(th, mm, vv, __ldg(g + i), a);
        theta[i] = th;
        m[i] = mm;
        v[i] = vv;
    }
}

}  // namespace
}  // namespace bitlogic

using namespace bitlogic;

BITLOGIC_ERROR_READER(optim)

extern "C" int bitlogic_adamw_update(float* theta, float* m, float* v, const float* grad, int64_t n,
                                     int64_t step, float lr, float beta1, float beta2, float eps,
                                     float weight_decay, cudaStream_t stream) {
    if (n < 0) return BITLOGIC_ERR_SHAPE;
    if (step < 1) return BITLOGIC_ERR_HYPER;
    if (!(beta1 >= 0.f && beta1 < 1.f && beta2 >= 0.f && beta2 < 1.f && eps > 0.f && lr >= 0.f &&
          weight_decay >= 0.f))
        return BITLOGIC_ERR_HYPER;
    if (n == 0) return BITLOGIC_OK;
    if (!theta || !m || !v || !grad) return BITLOGIC_ERR_NULL;
    AdamW a;
    a.lr = lr;
    a.b1 = beta1;
    a.b2 = beta2;
    a.eps = eps;
    a.wd = weight_decay;
    a.c1 = (float)(1.0 / (1.0 - std::pow((double)beta1, (double)step)));
    a.c2 = (float)(1.0 / (1.0 - std::pow((double)beta2, (double)step)));
    const long long cap = (long long)sm_count() * 8;
    if (n % 4 == 0 && aligned16(theta) && aligned16(m) && aligned16(v) && aligned16(grad)) {
        const long long n4 = n / 4;
        long long blocks = (n4 + 255) / 256;
        if (blocks > cap) blocks = cap;
        adamw_vec_kernel<<<(unsigned)blocks, 256, 0, stream>>>(
            reinterpret_cast<float4*>(theta), reinterpret_cast<float4*>(m), reinterpret_cast<float4*>(v),
            reinterpret_cast<const float4*>(grad), n4, a);
    } else {
        long long blocks = (n + 255) / 256;
        if (blocks > cap) blocks = cap;
        adamw_kernel<<<(unsigned)blocks, 256, 0, stream>>>(theta, m, v, grad, n, a);
    }
    return launch_status();
}
