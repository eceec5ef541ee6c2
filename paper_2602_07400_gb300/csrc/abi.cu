// Host-side parts of the C ABI that launch no kernels: status strings, the
// inverse-connectivity (CSR) builder, and the device-side index flag reader.
#include <algorithm>
#include <atomic>
#include <vector>

#include "common.cuh"

namespace bitlogic {

int sm_count() {
    constexpr int kMaxDevices = 64;
    static std::atomic<int> cache[kMaxDevices];   // 0: not queried yet
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 152;
    if (dev < kMaxDevices) {
        const int c = cache[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) n = 152;
    if (dev < kMaxDevices) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

}  // namespace bitlogic

extern "C" int bitlogic_internal_index_error_lut_soft(cudaStream_t);
extern "C" int bitlogic_internal_index_error_head(cudaStream_t);
extern "C" int bitlogic_internal_index_error_encode(cudaStream_t);
extern "C" int bitlogic_internal_index_error_hard(cudaStream_t);
extern "C" int bitlogic_internal_index_error_optim(cudaStream_t);
extern "C" int bitlogic_internal_index_error_route(cudaStream_t);
extern "C" int bitlogic_internal_index_error_lut_through(cudaStream_t);
extern "C" int bitlogic_internal_index_error_lut_bytes(cudaStream_t);

extern "C" const char* bitlogic_status_string(int code) {
    switch (code) {
        case BITLOGIC_OK: return "ok";
        case BITLOGIC_ERR_NULL: return "a required pointer is NULL";
        case BITLOGIC_ERR_SHAPE: return "invalid shape (size <= 0, overflow, grid limit, or w % C != 0)";
        case BITLOGIC_ERR_FANIN: return "unsupported fan-in (k must be 1..6 and <= w_in)";
        case BITLOGIC_ERR_ALIGN: return "workspace is not 16-byte aligned";
        case BITLOGIC_ERR_WORKSPACE: return "workspace too small";
        case BITLOGIC_ERR_CUDA: return "CUDA launch or copy failed";
        case BITLOGIC_ERR_INDEX: return "index out of range";
        case BITLOGIC_ERR_DEVICE: return "a kernel met an out-of-range index (read as 0)";
        case BITLOGIC_ERR_THRESH: return "number of thresholds must be 1..32";
        case BITLOGIC_ERR_TOO_LARGE: return "sizes exceed the fixed scratch of the allocation-free entry point";
        case BITLOGIC_ERR_HYPER: return "optimizer hyperparameter out of range";
        case BITLOGIC_ERR_NODE: return "unknown node form";
        default: return "unknown status";
    }
}

extern "C" int bitlogic_version(void) { return 100; }

// Counting sort of the edges e = j*k + slot by their input index; within an
// input the edges keep increasing e, which fixes the summation order of the
// input gradient.
extern "C" int bitlogic_build_csr(const int32_t* conn_host, int32_t w, int32_t k, int32_t w_in,
                                  int32_t* off_host, int32_t* edge_host) {
    if (!conn_host || !off_host || !edge_host) return BITLOGIC_ERR_NULL;
    if (w <= 0 || k <= 0 || w_in <= 0) return BITLOGIC_ERR_SHAPE;
    const long long nE = (long long)w * k;
    if (nE > 0x7fffffffLL) return BITLOGIC_ERR_SHAPE;
    for (long long e = 0; e < nE; ++e)
        if (conn_host[e] < 0 || conn_host[e] >= w_in) return BITLOGIC_ERR_INDEX;
    for (int32_t i = 0; i <= w_in; ++i) off_host[i] = 0;
    for (long long e = 0; e < nE; ++e) ++off_host[conn_host[e] + 1];
    for (int32_t i = 0; i < w_in; ++i) off_host[i + 1] += off_host[i];
    std::vector<int32_t> fill(off_host, off_host + w_in);
    for (long long e = 0; e < nE; ++e) edge_host[fill[conn_host[e]]++] = (int32_t)e;
    return BITLOGIC_OK;
}

extern "C" int bitlogic_csr_positions(const int32_t* edge_host, int32_t n_edges, int32_t* pos_host) {
    if (!edge_host || !pos_host) return BITLOGIC_ERR_NULL;
    if (n_edges < 0) return BITLOGIC_ERR_SHAPE;
    for (int32_t e = 0; e < n_edges; ++e) pos_host[e] = -1;
    for (int32_t p = 0; p < n_edges; ++p) {
        const int32_t e = edge_host[p];
        if (e < 0 || e >= n_edges || pos_host[e] != -1) return BITLOGIC_ERR_INDEX;
        pos_host[e] = p;
    }
    return BITLOGIC_OK;
}

extern "C" int bitlogic_degree_order(const int32_t* off_host, int32_t n, int32_t* order_host) {
    if (!off_host || !order_host) return BITLOGIC_ERR_NULL;
    if (n <= 0) return BITLOGIC_ERR_SHAPE;
    if (off_host[0] != 0) return BITLOGIC_ERR_INDEX;
    for (int32_t i = 0; i < n; ++i)
        if (off_host[i + 1] < off_host[i]) return BITLOGIC_ERR_INDEX;
    // stable sort by decreasing degree: ties keep increasing index
    for (int32_t i = 0; i < n; ++i) order_host[i] = i;
    std::stable_sort(order_host, order_host + n, [off_host](int32_t a, int32_t b) {
        return off_host[a + 1] - off_host[a] > off_host[b + 1] - off_host[b];
    });
    return BITLOGIC_OK;
}

extern "C" int bitlogic_device_error(cudaStream_t stream) {
    int worst = BITLOGIC_OK;
    const int r[8] = {bitlogic_internal_index_error_lut_soft(stream),
                      bitlogic_internal_index_error_head(stream),
                      bitlogic_internal_index_error_encode(stream),
                      bitlogic_internal_index_error_hard(stream),
                      bitlogic_internal_index_error_optim(stream),
                      bitlogic_internal_index_error_route(stream),
                      bitlogic_internal_index_error_lut_through(stream),
                      bitlogic_internal_index_error_lut_bytes(stream)};
    for (int v : r) {
        if (v == BITLOGIC_ERR_CUDA) return v;
        if (v != BITLOGIC_OK) worst = v;
    }
    return worst;
}
