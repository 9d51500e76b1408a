// Error reporting, version and device queries of the C ABI.
#include <cstdarg>
#include <cstdio>
#include <map>
#include <mutex>
#include <tuple>

#include "pldp_internal.cuh"

namespace pldp {

static thread_local char g_last_error[512] = "";

pldp_status fail(pldp_status code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof g_last_error, fmt, ap);
    va_end(ap);
    return code;
}

pldp_status check_launch(const char* what) {
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess)
        return fail(PLDP_ERR_CUDA, "%s: launch failed: %s", what, cudaGetErrorString(e));
    return PLDP_OK;
}

int sm_count() {
    int dev = 0, n = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 1;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 1;
    return n > 0 ? n : 1;
}

int resident_blocks(const void* kernel, int threads, size_t smem) {
    static std::mutex mu;
    static std::map<std::tuple<int, const void*, int, size_t>, int> cache;
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return sm_count();
    const auto key = std::make_tuple(dev, kernel, threads, smem);
    {
        std::lock_guard<std::mutex> lock(mu);
        auto it = cache.find(key);
        if (it != cache.end()) return it->second;
    }
    int per_sm = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, kernel, threads, smem) != cudaSuccess ||
        per_sm < 1)
        per_sm = 1;
    const int n = per_sm * sm_count();
    std::lock_guard<std::mutex> lock(mu);
    cache[key] = n;
    return n;
}

}  // namespace pldp

extern "C" {

PLDP_API const char* pldp_last_error(void) { return pldp::g_last_error; }

PLDP_API int pldp_version(void) { return 200; }  // 0.2.0: attention key stride, fused sampling call

}  // extern "C"
