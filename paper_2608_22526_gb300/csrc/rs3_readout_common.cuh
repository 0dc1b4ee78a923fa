// rs3_readout_common.cuh -- argument block and helpers shared by the readout
// kernels (CUDA-core and tensor-core paths).
#pragma once

#include "rs3_internal.cuh"

#define RS3_MAX_UNITS 4096  // units per readout call

struct ReadoutArgs {
    const void *q;
    const void *k_store;
    const void *v_store;
    const int64_t *meta;
    int64_t meta_stride_words;
    int64_t pinned_cap, ring_cap, rows_per_unit;
    int64_t n_ptr;
    const int32_t *unit_group;
    const int32_t *idx;
    const int32_t *count;
    const float *rope;
    const void *residual;
    void *out;
    int32_t *status;
    int U, G, mn, H, d, D, k_max;
    int BM, BN, n_sm, min_chunk;
    int plan_ov;            // leading plan slots per group: a piece's start-up cost in tiles
    int64_t max_slots;
    int64_t max_items;
    int grid_ctas;          // CTAs of the readout launch (the plan's slice count bound)
    int32_t *cta_items;     // [grid_ctas][2]: CTA b runs items [cta_items[2b], cta_items[2b+1])
    float scale_log2;       // softmax scale * log2(e)
    uint64_t wait_ns;       // limit of each device-side wait (global-timer ns)
    ReadoutHeader *header;
    RangeSet *ranges;
    WorkItem *items;
    CombineItem *combine;
    float *part_o;          // [slot][BM][d]
    float *part_ml;         // [slot][BM] (m, l) pairs, m in the log2 domain
};

struct ReadoutPath {
    int kind;   // 0 = CUDA-core, 1 = tensor-core (tcgen05)
    int BM, BN;
    int grid;   // CTAs of the readout launch
};

ReadoutPath choose_readout_path(rs3_dtype dtype, int d);
bool rs3_tc_supported(int d);
int rs3_tc_block_n(int d);
rs3_status rs3_launch_tc_readout(const ReadoutArgs &a, cudaStream_t st);
rs3_status rs3_readout_prepare(const void *q, rs3_dtype dtype, int G, int mn, int H, int d,
                               const int32_t *unit_group, const int32_t *idx, const int32_t *count,
                               int k_max, const rs3_bank *bank, const float *rope,
                               const void *residual, void *out, float scale, void *workspace,
                               size_t workspace_bytes, int32_t *status, ReadoutArgs *a,
                               ReadoutPath *path, int64_t *grid_items, int64_t *grid_combine);
// phases of a readout: the attention over the bank (pass-through, plan,
// readout kernel) and the merge of split-KV partials
enum { RS3_PHASE_PLAN = 1, RS3_PHASE_RUN = 4, RS3_PHASE_ATTEND = 1 | 4, RS3_PHASE_MERGE = 2 };
rs3_status rs3_readout_launch(const ReadoutArgs &a, const ReadoutPath &p, int64_t max_items,
                              int64_t max_combine, rs3_dtype dtype, cudaStream_t st, int phases);

// Tile t of a unit's bank (tiles of BN rows, never crossing a range end) ->
// first physical row and the number of valid rows.
__device__ __forceinline__ void tile_rows(const RangeSet &rs, int t, int BN, int64_t &row0, int &nvalid)
{
    row0 = 0;
    nvalid = 0;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        if (t < rs.tiles[r]) {
            row0 = rs.start[r] + (int64_t)t * BN;
            nvalid = min(BN, rs.len[r] - t * BN);
            return;
        }
        t -= rs.tiles[r];
    }
}

// Same, reading the range set in place (global memory) instead of a local copy.
__device__ __forceinline__ void tile_rows(const RangeSet *rs, int t, int BN, int64_t &row0, int &nvalid)
{
    row0 = 0;
    nvalid = 0;
#pragma unroll
    for (int r = 0; r < 4; ++r) {
        const int tiles = __ldg(&rs->tiles[r]);
        if (t < tiles) {
            row0 = __ldg(&rs->start[r]) + (int64_t)t * BN;
            nvalid = min(BN, __ldg(&rs->len[r]) - t * BN);
            return;
        }
        t -= tiles;
    }
}

__device__ __forceinline__ float4 load4(const float *p) { return __ldg(reinterpret_cast<const float4 *>(p)); }
__device__ __forceinline__ float4 load4(const uint16_t *p)
{
    const uint2 w = __ldg(reinterpret_cast<const uint2 *>(p));
    return make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u),
                       __uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
}

__device__ __forceinline__ void load16(const float *p, float *o)
{
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const float4 v = __ldg(reinterpret_cast<const float4 *>(p) + k);
        o[4 * k] = v.x; o[4 * k + 1] = v.y; o[4 * k + 2] = v.z; o[4 * k + 3] = v.w;
    }
}
__device__ __forceinline__ void load16(const uint16_t *p, float *o)
{
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const uint4 v = __ldg(reinterpret_cast<const uint4 *>(p) + k);
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            o[8 * k + 2 * e] = __uint_as_float(w[e] << 16);
            o[8 * k + 2 * e + 1] = __uint_as_float(w[e] & 0xffff0000u);
        }
    }
}

// Two fp32 values to a bf16 pair (round to nearest even), `lo` in the low half;
// one cvt instruction (the per-value conversions cost about three times more).
__device__ __forceinline__ uint32_t pack_bf16x2(float lo, float hi)
{
    uint32_t r;
    asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(hi), "f"(lo));
    return r;
}

// out[u][cell][c0 .. c0+15] = residual[...] + o (one rounding to T)
template <typename T>
__device__ __forceinline__ void store_out16(const ReadoutArgs &a, int u, int cell, int c0, const float *o);

template <>
__device__ __forceinline__ void store_out16<float>(const ReadoutArgs &a, int u, int cell, int c0, const float *o)
{
    const int64_t off = ((int64_t)u * a.mn + cell) * a.D + c0;
    float r[16];
    if (a.residual) load16(static_cast<const float *>(a.residual) + off, r);
    else {
#pragma unroll
        for (int k = 0; k < 16; ++k) r[k] = 0.f;
    }
    float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(a.out) + off);
#pragma unroll
    for (int k = 0; k < 4; ++k)
        dst[k] = make_float4(r[4 * k] + o[4 * k], r[4 * k + 1] + o[4 * k + 1], r[4 * k + 2] + o[4 * k + 2],
                             r[4 * k + 3] + o[4 * k + 3]);
}

template <>
__device__ __forceinline__ void store_out16<uint16_t>(const ReadoutArgs &a, int u, int cell, int c0, const float *o)
{
    const int64_t off = ((int64_t)u * a.mn + cell) * a.D + c0;
    float r[16];
    if (a.residual) load16(static_cast<const uint16_t *>(a.residual) + off, r);
    else {
#pragma unroll
        for (int k = 0; k < 16; ++k) r[k] = 0.f;
    }
    uint4 *dst = reinterpret_cast<uint4 *>(static_cast<uint16_t *>(a.out) + off);
#pragma unroll
    for (int k = 0; k < 2; ++k)
        dst[k] = make_uint4(pack_bf16x2(r[8 * k] + o[8 * k], r[8 * k + 1] + o[8 * k + 1]),
                            pack_bf16x2(r[8 * k + 2] + o[8 * k + 2], r[8 * k + 3] + o[8 * k + 3]),
                            pack_bf16x2(r[8 * k + 4] + o[8 * k + 4], r[8 * k + 5] + o[8 * k + 5]),
                            pack_bf16x2(r[8 * k + 6] + o[8 * k + 6], r[8 * k + 7] + o[8 * k + 7]));
}

template <typename T>
__device__ __forceinline__ void store_out4(const ReadoutArgs &a, int u, int cell, int c, const float *o);

template <>
__device__ __forceinline__ void store_out4<float>(const ReadoutArgs &a, int u, int cell, int c, const float *o)
{
    const int64_t off = ((int64_t)u * a.mn + cell) * a.D + c;
    float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
    if (a.residual) r = load4(static_cast<const float *>(a.residual) + off);
    *reinterpret_cast<float4 *>(static_cast<float *>(a.out) + off) =
        make_float4(r.x + o[0], r.y + o[1], r.z + o[2], r.w + o[3]);
}

template <>
__device__ __forceinline__ void store_out4<uint16_t>(const ReadoutArgs &a, int u, int cell, int c, const float *o)
{
    const int64_t off = ((int64_t)u * a.mn + cell) * a.D + c;
    float4 r = make_float4(0.f, 0.f, 0.f, 0.f);
    if (a.residual) r = load4(static_cast<const uint16_t *>(a.residual) + off);
    *reinterpret_cast<uint2 *>(static_cast<uint16_t *>(a.out) + off) =
        make_uint2(pack_bf16x2(r.x + o[0], r.y + o[1]), pack_bf16x2(r.z + o[2], r.w + o[3]));
}
