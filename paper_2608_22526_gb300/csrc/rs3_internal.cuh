// rs3_internal.cuh -- device helpers and internal layouts shared by the
// librs3 translation units (not part of the public ABI).
#pragma once

#include <cuda_runtime.h>
#include <cuda_bf16.h>
#include <stdint.h>

#include "../../include/rs3.h"

#define RS3_VERSION 100
#define RS3_BANK_MAGIC 0x52533342u   // "RS3B"
#define RS3_MAX_MN 16384

// ---------------------------------------------------------------------------
// Bank metadata layout (device, int64 words per unit)
// ---------------------------------------------------------------------------
// header words
enum {
    BM_HEAD = 0,        // ring logical position of the oldest live row
    BM_TAIL = 1,        // ring logical position one past the newest row
    BM_COND_LEN = 2,    // rows in the pinned region
    BM_NFRAMES = 3,     // ring frames held
    BM_OLDEST = 4,      // frame-table slot of the oldest ring frame
    BM_NCOND = 5,       // pinned frames held
    BM_PTRLEN = 6,      // pointer rows held
    BM_ARRIVE = 8,      // CTAs of the running commit that have read the old counters
    BM_HEADER_WORDS = 16
};
// after the header: int64 foff[max_frames], int64 flen[max_frames]

__host__ __device__ inline int64_t bank_meta_words(int max_frames)
{
    return (int64_t)BM_HEADER_WORDS + 2 * (int64_t)max_frames;
}

// ---------------------------------------------------------------------------
// Readout work list (in the caller's workspace)
// ---------------------------------------------------------------------------
struct RangeSet {           // a unit's bank as <= 4 contiguous row ranges
    int64_t start[4];       // first physical row (within the unit's storage)
    int32_t len[4];
    int32_t tiles[4];       // ceil(len / BN)
    int32_t n_tiles;        // total tiles
    int32_t nq;             // query tiles of BM rows
    int32_t cnt;            // kept queries (clamped to k_max)
    int32_t splits;         // KV splits per (head, query tile)
    int32_t slot_base;      // first partial slot of the unit (-1 if no splits)
    int32_t pad[3];
};

struct WorkItem {
    int32_t u, h, qt, split;
    int32_t tile_begin, tile_end;
    int32_t slot;           // partial slot, -1 = write the output directly
    int32_t pad;
};

struct CombineItem {
    int32_t u, h, qt, slot0;
    int32_t nsplit, pad[3];
};

struct ReadoutHeader {
    int32_t n_items;
    int32_t n_combine;
    int32_t pad[30];
};

struct ReadoutLayout {      // byte offsets inside the workspace
    size_t header, cta_items, ranges, items, combine, part_o, part_ml, total;
    int64_t max_items, max_combine, max_slots;
};


// ---------------------------------------------------------------------------
// Device helpers
// ---------------------------------------------------------------------------
__device__ __forceinline__ void latch_status(int32_t *status, int32_t code)
{
    if (status) atomicCAS(status, 0, code);
}

__device__ __forceinline__ float bf16_bits_to_float(uint16_t b)
{
    return __uint_as_float(((uint32_t)b) << 16);
}

__device__ __forceinline__ uint16_t float_to_bf16_bits(float f)
{
    __nv_bfloat16 h = __float2bfloat16_rn(f);
    return *reinterpret_cast<uint16_t *>(&h);
}

template <typename T>
__device__ __forceinline__ T warp_sum(T v)
{
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xffffffffu, v, o);
    return v;
}

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// ---------------------------------------------------------------------------
// Programmatic dependent launch.  Every kernel of the library is launched with
// programmatic stream serialisation, so its launch is processed while the
// previous kernel of its stream runs; pdl_wait() returns once that kernel has
// completed and its writes are visible (at once when there is none), and every
// kernel calls it before its first global-memory access.  No kernel triggers
// its dependents early: they are scheduled when it completes, so kernels
// waiting for their predecessor never hold SMs that the selection running on
// another stream could use.
// ---------------------------------------------------------------------------
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kernel)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t st,
                              Args &&...args)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = st;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kernel, static_cast<Args &&>(args)...);
}

// Host helpers implemented in rs3_api.cu
int rs3_sm_count();
bool rs3_aligned16(const void *p);
// Raises `kernel`'s dynamic shared-memory limit on the current device to at
// least `bytes` (once per kernel and device; safe to call from several host
// threads).  RS3_ECUDA when the runtime refuses.
rs3_status rs3_kernel_smem(const void *kernel, size_t bytes);
