// rs3_api.cu -- small host-side pieces of the C ABI: defaults, k_max, status
// strings, device queries.
#include "rs3_internal.cuh"

#include <cmath>
#include <mutex>
#include <utility>
#include <vector>

extern "C" void rs3_default_params(rs3_params *p)
{
    if (!p) return;
    p->rho = 0.3;          // Algorithm 1 hyper-parameters
    p->r_s = 4;
    p->c = 14;
    p->D_w = 24;           // SAM2 default of Sec. 5.3
    p->union_mode = 1;     // Eq. 2: P(t) is the union over the stream's objects
    p->fall_lo = 0.05;     // Sec. 3.2 fall-through bounds
    p->fall_hi = 0.95;
    p->fall_through = 1;
    p->bbox_mode = 0;
}

extern "C" int64_t rs3_kmax(double rho, int64_t mn)
{
    if (!(rho >= 0.0 && rho <= 1.0) || mn < 0) return -1;
    return (int64_t)std::floor(rho * (double)mn);
}

extern "C" const char *rs3_status_string(int code)
{
    switch (code) {
    case RS3_OK: return "ok";
    case RS3_EINVAL: return "invalid argument";
    case RS3_ECAPACITY: return "capacity exceeded";
    case RS3_EUNSUPPORTED: return "unsupported size or dtype";
    case RS3_ECUDA: return "CUDA error";
    case RS3_EINTERNAL: return "inconsistent bank metadata";
    case RS3_ETIMEOUT: return "device wait timed out";
    default: return "unknown status";
    }
}

extern "C" int rs3_version(void) { return RS3_VERSION; }

int rs3_sm_count()
{
    static int cached[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 64) return 148;
    if (cached[dev] == 0) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0)
            n = 148;
        cached[dev] = n;
    }
    return cached[dev];
}

bool rs3_aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

rs3_status rs3_kernel_smem(const void *kernel, size_t bytes)
{
    if (bytes <= 48 * 1024) return RS3_OK;     // the default limit
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return RS3_ECUDA;
    static std::mutex mu;
    static std::vector<std::pair<std::pair<const void *, int>, size_t>> done;   // (kernel, device) -> bytes
    std::lock_guard<std::mutex> lock(mu);
    for (auto &e : done)
        if (e.first.first == kernel && e.first.second == dev) {
            if (e.second >= bytes) return RS3_OK;
            if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes) !=
                cudaSuccess)
                return RS3_ECUDA;
            e.second = bytes;
            return RS3_OK;
        }
    if (cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes) != cudaSuccess)
        return RS3_ECUDA;
    done.push_back({{kernel, dev}, bytes});
    return RS3_OK;
}
