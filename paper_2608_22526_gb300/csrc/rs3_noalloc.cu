// rs3_noalloc.cu -- keep-set selection for callers that cannot allocate
// device memory.
//
// rs3_select_queries needs a caller-provided scratch workspace.  Some callers
// have no way to obtain one: code that runs where cudaMalloc is not allowed
// (for example while a stream is being captured into a graph in the global
// capture mode), serving loops that must not allocate once they are running,
// or hosts that embed the library behind an interface that hands over only
// the input and output buffers.  This file gives them one entry point whose
// scratch lives in a fixed device array compiled into the library.
#include "rs3_internal.cuh"

#include <cuda.h>

#include <mutex>

// 8 MiB of scratch, held by every GPU that loads the library until the process
// exits.  Enough for G = U = 64 on the largest grid (mn = 16384).
#define RS3_NOALLOC_SCRATCH_BYTES (8u << 20)

static __device__ __align__(256) uint8_t rs3_noalloc_scratch[RS3_NOALLOC_SCRATCH_BYTES];

namespace {

std::mutex g_setup_mutex;
void *g_scratch_ptr[64] = {nullptr};
unsigned long long g_scratch_ctx[64] = {0};   // id of the context the address belongs to

typedef CUresult (*ctx_get_current_fn)(CUcontext *);
typedef CUresult (*ctx_get_id_fn)(CUcontext, unsigned long long *);

// Id of the calling thread's current context (0 when it cannot be asked).  A
// device reset, or a new primary context, gives the array a new address; the
// id tells the cached address from the current one.
unsigned long long current_context_id()
{
    static ctx_get_current_fn get_cur = nullptr;
    static ctx_get_id_fn get_id = nullptr;
    static bool looked = false;
    if (!looked) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetCurrent", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_cur = reinterpret_cast<ctx_get_current_fn>(p);
        p = nullptr;
        if (cudaGetDriverEntryPointByVersion("cuCtxGetId", &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            get_id = reinterpret_cast<ctx_get_id_fn>(p);
        looked = true;
    }
    CUcontext ctx = nullptr;
    unsigned long long id = 0;
    if (!get_cur || !get_id || get_cur(&ctx) != CUDA_SUCCESS || !ctx || get_id(ctx, &id) != CUDA_SUCCESS) return 0;
    return id;
}

// Device address of the scratch array on the current device.  In host code
// the array's name is only a host-side stand-in, so the address is asked from
// the runtime with the device current, and cached per device together with
// the id of the context it belongs to (asked again when that id changes).
rs3_status scratch_for_current_device(void **out)
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return RS3_ECUDA;
    if (dev < 0 || dev >= 64) return RS3_EUNSUPPORTED;
    std::lock_guard<std::mutex> lock(g_setup_mutex);
    const unsigned long long ctx = current_context_id();
    if (g_scratch_ptr[dev] == nullptr || (ctx != 0 && ctx != g_scratch_ctx[dev])) {
        void *p = nullptr;
        if (cudaGetSymbolAddress(&p, rs3_noalloc_scratch) != cudaSuccess || p == nullptr)
            return RS3_ECUDA;
        g_scratch_ptr[dev] = p;
        g_scratch_ctx[dev] = current_context_id();
    }
    *out = g_scratch_ptr[dev];
    return RS3_OK;
}

}  // namespace

extern "C" rs3_status rs3_select_queries_noalloc(const void *z, rs3_dtype dtype, int G, int m, int n,
                                                 int C, const uint8_t *prev_masks,
                                                 const int32_t *unit_group, int U, rs3_track *track,
                                                 const rs3_params *p, int32_t *idx, int32_t *count,
                                                 int32_t *status, rs3_stream_t stream)
{
    const size_t need = rs3_select_workspace_bytes(G, U, m, n);
    if (need == 0) return RS3_EINVAL;
    if (need > RS3_NOALLOC_SCRATCH_BYTES) return RS3_ECAPACITY;
    void *scratch = nullptr;
    const rs3_status s = scratch_for_current_device(&scratch);
    if (s != RS3_OK) return s;
    // The scratch keeps whatever the previous call left; the selection clears
    // the part that must start at zero (the group bitmap) on `stream` itself.
    return rs3_select_queries(z, dtype, G, m, n, C, prev_masks, unit_group, U, track, p, idx, count,
                              scratch, RS3_NOALLOC_SCRATCH_BYTES, status, stream);
}
