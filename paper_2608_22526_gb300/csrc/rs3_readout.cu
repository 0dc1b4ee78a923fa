// rs3_readout.cu -- pruned memory readout (Sec. 3.1: Eq. 6 gather / attention /
// scatter, Eq. 7 RoPE by the gathered index), host entry and the shared
// pieces of both kernel paths.
//
// Launch sequence (no host synchronisation).  Attend phase:
//   k_passthrough  out-of-place only: out = residual (or zeros) on every cell
//   k_plan         one CTA: per unit, the bank's row ranges (pinned, ring
//                  pieces, pointers) and a balanced work list of
//                  (unit, head, query tile, KV tile range) items; long banks
//                  are split along the keys so every SM gets work
//   k_readout_*    flash attention per item: gather the kept query rows (and
//                  rotate them), stream the bank tiles, online softmax in the
//                  log2 domain, fp32 accumulation; an unsplit item writes
//                  out = residual + A directly at the kept cells, a split item
//                  writes (O, m, l) partials
// Merge phase (reads no bank, so it may run beside a commit):
//   k_combine      log-sum-exp merge of the partials and the scatter
// rs3_memory_readout issues both phases on one stream;
// rs3_memory_readout_attend / _merge issue one each.
#include "rs3_internal.cuh"

#include <atomic>
#include <cmath>

#include "rs3_readout_common.cuh"

namespace {

// ---------------------------------------------------------------------------
// k_passthrough: unselected cells equal the residual bit for bit (Eq. 6 S_K)
// ---------------------------------------------------------------------------
__global__ void k_passthrough(const uint4 *__restrict__ res, uint4 *__restrict__ out, int64_t nvec)
{
    pdl_wait();
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nvec;
         i += (int64_t)gridDim.x * blockDim.x)
        out[i] = res ? __ldcs(res + i) : make_uint4(0, 0, 0, 0);
}

// ---------------------------------------------------------------------------
// k_plan: ranges and the work list
// ---------------------------------------------------------------------------
__device__ RangeSet unit_ranges(const ReadoutArgs &a, int u, int cnt)
{
    RangeSet rs;
    const int64_t *mu = a.meta + (int64_t)u * a.meta_stride_words;
    const int64_t cond = mu[BM_COND_LEN];
    const int64_t head = mu[BM_HEAD], tail = mu[BM_TAIL], ptr = mu[BM_PTRLEN];
    for (int r = 0; r < 4; ++r) { rs.start[r] = 0; rs.len[r] = 0; rs.tiles[r] = 0; }
    rs.start[0] = 0;
    rs.len[0] = (int32_t)cond;
    const int64_t live = tail - head;
    if (live > 0 && a.ring_cap > 0) {
        const int64_t p0 = head % a.ring_cap;
        const int64_t first = min(live, a.ring_cap - p0);
        rs.start[1] = a.pinned_cap + p0;
        rs.len[1] = (int32_t)first;
        rs.start[2] = a.pinned_cap;
        rs.len[2] = (int32_t)(live - first);
    }
    rs.start[3] = a.pinned_cap + a.ring_cap;
    rs.len[3] = (int32_t)ptr;
    int nt = 0;
    for (int r = 0; r < 4; ++r) {
        rs.tiles[r] = (rs.len[r] + a.BN - 1) / a.BN;
        nt += rs.tiles[r];
    }
    rs.n_tiles = nt;
    rs.cnt = cnt;
    rs.nq = (cnt + a.BM - 1) / a.BM;
    rs.splits = 1;
    rs.slot_base = -1;
    return rs;
}

// Exclusive block scan of an (int64, int32) pair per thread; returns the
// offsets and writes the block totals.
__device__ void block_scan_pair(int64_t v, int32_t g, int64_t &off_v, int32_t &off_g, int64_t &tot_v,
                                int32_t &tot_g)
{
    __shared__ int64_t s_pv[32];
    __shared__ int32_t s_pg[32];
    __shared__ int64_t s_tv;
    __shared__ int32_t s_tg;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int64_t iv = v;
    int32_t ig = g;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int64_t tv = __shfl_up_sync(0xffffffffu, iv, o);
        const int32_t tg = __shfl_up_sync(0xffffffffu, ig, o);
        if (lane >= o) { iv += tv; ig += tg; }
    }
    if (lane == 31) { s_pv[warp] = iv; s_pg[warp] = ig; }
    __syncthreads();
    if (threadIdx.x == 0) {
        int64_t rv = 0;
        int32_t rg = 0;
        for (int w = 0; w < nw; ++w) {
            const int64_t tv = s_pv[w];
            const int32_t tg = s_pg[w];
            s_pv[w] = rv;
            s_pg[w] = rg;
            rv += tv;
            rg += tg;
        }
        s_tv = rv;
        s_tg = rg;
    }
    __syncthreads();
    off_v = s_pv[warp] + iv - v;
    off_g = s_pg[warp] + ig - g;
    tot_v = s_tv;
    tot_g = s_tg;
    __syncthreads();
}

// Stream-K plan.  Group g = (unit u, query tile qt, head h) owns
// wg_u = OV + T_u consecutive slots of a linear work axis (T_u = key tiles of
// the unit's bank): OV leading slots stand for the fixed cost of starting a
// piece of work (loading the query rows, the epilogue), so a CTA whose slice
// starts groups gets fewer tiles, and the T_u tile slots follow.  CTA b of P
// takes slots [sb(b), sb(b+1)) with sb(b) = b W / P; its slice is cut at group
// boundaries into items, each the tiles of the group its part covers.  A group
// with no tiles (empty bank) is one item with no tiles, emitted where its first
// slot lies, so its rows are still written.
//
// Indexing without a scan over the slices: the piece of group G (linear index
// over all units' groups) in slice b is item G + b.  Each group's pieces lie in
// consecutive slices and the groups follow each other along the axis, so the
// indices are unique and a slice's items are consecutive.  Only a slice's first
// item can be cut at its start and only its last at its end, so a split piece
// takes partial slot 2b (the slice's first item) or 2b + 1 (its last); a split
// group's later pieces are each the first item of their slice.  The slice that
// holds a split group's first tile emits the group's merge entry (the entries
// are packed in any order).
struct PlanView {
    const int64_t *tb;   // [U+1] first linear slot of each unit
    const int64_t *wg;   // [U]   slots per group of each unit
    const int32_t *nt;   // [U]   key tiles of each unit
    const int32_t *gb;   // [U+1] first linear group of each unit
    const int32_t *cnt;  // [U]   kept queries of each unit
    int U, H;
    int64_t W;
    int P;
    int ov;              // leading slots of a group (the start-up cost)
};

// b W / P; in 32 bits when b W cannot reach 2^32 (W < 2^22, b < 1024)
__device__ __forceinline__ int64_t slice_start(const PlanView &v, int b)
{
    if (v.P <= 0) return 0;
    if (v.W < ((int64_t)1 << 22) && b < 1024) return (int64_t)((uint32_t)b * (uint32_t)v.W / (uint32_t)v.P);
    return (int64_t)b * v.W / v.P;
}

__device__ __forceinline__ void locate(const PlanView &v, int64_t x, int &u, int &gl, int64_t &off)
{
    int lo = 0, hi = v.U;                          // largest u with tb[u] <= x
    while (hi - lo > 1) {
        const int mid = (lo + hi) >> 1;
        if (v.tb[mid] <= x) lo = mid; else hi = mid;
    }
    u = lo;
    const int64_t rel = x - v.tb[u];
    if (v.W < ((int64_t)1 << 22)) {
        gl = (int)((uint32_t)rel / (uint32_t)v.wg[u]);
    } else {
        gl = (int)(rel / v.wg[u]);
    }
    off = rel - (int64_t)gl * v.wg[u];
}

// Writes slice b's items and its item range; returns its merge entry in c
// (nsplit 0: none) and its partial pieces in n_part.
__device__ void plan_slice(const ReadoutArgs &a, const PlanView &v, int b, int &n_part, CombineItem &c)
{
    const int64_t lo = slice_start(v, b), hi = slice_start(v, b + 1);
    int64_t first = -1, last = -1;
    c.u = c.h = c.qt = c.slot0 = c.nsplit = 0;
    c.pad[0] = b;
    c.pad[1] = c.pad[2] = 0;                      // pad[1]: the unit's kept queries
    n_part = 0;
    for (int64_t x = lo; x < hi;) {
        int u, gl;
        int64_t off;
        locate(v, x, u, gl, off);
        const int64_t wg = v.wg[u];
        const int64_t len = min(hi - x, wg - off);
        const int64_t nt = v.nt[u];
        // the tiles this part covers, and whether it holds all or the first
        const int64_t t0 = min(max(off - v.ov, (int64_t)0), nt);
        const int64_t t1 = min(max(off + len - v.ov, (int64_t)0), nt);
        const bool emit = nt > 0 ? t1 > t0 : off == 0;
        if (emit) {
            const bool whole = t0 == 0 && t1 == nt;
            const int64_t idx = (int64_t)v.gb[u] + gl + b;
            WorkItem w;
            w.u = u; w.qt = gl / v.H; w.h = gl % v.H; w.split = 0;
            w.tile_begin = (int32_t)t0;
            w.tile_end = (int32_t)t1;
            w.slot = whole ? -1 : 2 * b + (first < 0 ? 0 : 1);
            w.pad = 0;
            a.items[idx] = w;
            if (first < 0) first = idx;
            last = idx;
            if (!whole) ++n_part;
            if (!whole && t0 == 0) {
                // first piece of a split group: the last slice its last slot
                // reaches is the largest e with sb(e) <= gend
                const int64_t gend = x - off + wg - 1;
                int64_t e = ((gend + 1) * v.P - 1) / v.W;
                if (e > v.P - 1) e = v.P - 1;
                c.u = u; c.h = w.h; c.qt = w.qt;
                c.slot0 = w.slot;
                c.nsplit = (int32_t)(e - b + 1);
                c.pad[1] = v.cnt[u];
            }
        }
        x += len;
    }
    a.cta_items[2 * b] = (int32_t)(first < 0 ? 0 : first);
    a.cta_items[2 * b + 1] = (int32_t)(first < 0 ? 0 : last + 1);
}

constexpr int PLAN_THREADS = 256;

__global__ void __launch_bounds__(PLAN_THREADS) k_plan(ReadoutArgs a)
{
    pdl_wait();
    ReadoutHeader *hdr = a.header;
    // [U+1] tb, [U] wg (int64); [U+1] gb, [U] nt (int32)
    extern __shared__ int64_t s_plan[];
    int64_t *s_tb = s_plan, *s_wg = s_tb + (a.U + 1);
    int32_t *s_gb = reinterpret_cast<int32_t *>(s_wg + a.U), *s_nt = s_gb + (a.U + 1), *s_cnt = s_nt + a.U;
    __shared__ int s_np, s_nc;
    if (threadIdx.x == 0) { s_np = 0; s_nc = 0; }
    // per unit: the bank's ranges, its groups and their width, scanned into
    // slot and group bases (rounds of blockDim units)
    int64_t run = 0;
    int32_t grun = 0;
    for (int u0 = 0; u0 < a.U; u0 += blockDim.x) {
        const int u = u0 + threadIdx.x;
        int64_t slots = 0;
        int32_t groups = 0;
        if (u < a.U) {
            // every load first (none depends on another), then the checks
            const int64_t *mu = a.meta + (int64_t)u * a.meta_stride_words;
            int cnt = a.count[u];
            const int g = a.unit_group[u];
            const int64_t head = mu[BM_HEAD], tail = mu[BM_TAIL], cond = mu[BM_COND_LEN], ptr = mu[BM_PTRLEN];
            if (cnt < 0 || cnt > a.k_max) {
                latch_status(a.status, RS3_EINVAL);
                cnt = cnt < 0 ? 0 : a.k_max;
            }
            if (g < 0 || g >= a.G) {                // no work for a unit without a valid grid
                latch_status(a.status, RS3_EINVAL);
                cnt = 0;
            }
            const bool sane = head >= 0 && tail >= head && tail - head <= a.ring_cap && cond >= 0 &&
                              cond <= a.pinned_cap && ptr >= 0 && ptr <= a.n_ptr;
            RangeSet rs;
            if (!sane) {
                latch_status(a.status, RS3_EINTERNAL);
                for (int r = 0; r < 4; ++r) { rs.start[r] = 0; rs.len[r] = 0; rs.tiles[r] = 0; }
                rs.n_tiles = 0; rs.cnt = 0; rs.nq = 0; rs.splits = 1; rs.slot_base = -1;
            } else {
                rs = unit_ranges(a, u, cnt);
            }
            a.ranges[u] = rs;
            s_wg[u] = (int64_t)a.plan_ov + rs.n_tiles;
            s_nt[u] = rs.n_tiles;
            s_cnt[u] = rs.cnt;
            groups = rs.nq * a.H;
            slots = (int64_t)groups * s_wg[u];
        }
        int64_t off, tot;
        int32_t goff, gtot;
        block_scan_pair(slots, groups, off, goff, tot, gtot);
        if (u < a.U) {
            s_tb[u] = off + run;
            s_gb[u] = goff + grun;
        }
        run += tot;
        grun += gtot;
    }
    if (threadIdx.x == 0) {
        s_tb[a.U] = run;
        s_gb[a.U] = grun;
    }
    int64_t P = (run + a.min_chunk - 1) / a.min_chunk;
    if (P > a.grid_ctas) P = a.grid_ctas;
    __syncthreads();
    PlanView v;
    v.tb = s_tb; v.wg = s_wg; v.nt = s_nt; v.gb = s_gb; v.cnt = s_cnt; v.U = a.U; v.H = a.H; v.W = run;
    v.ov = a.plan_ov;
    v.P = (int)P;
    // every CTA of the launch gets its item range (empty past the P slices);
    // merge entries are packed through a shared counter
    for (int b = threadIdx.x; b < a.grid_ctas; b += blockDim.x) {
        if (b < v.P) {
            int np;
            CombineItem c;
            plan_slice(a, v, b, np, c);
            if (np) atomicAdd(&s_np, np);
            if (c.nsplit > 0) a.combine[atomicAdd(&s_nc, 1)] = c;
        } else {
            a.cta_items[2 * b] = 0;
            a.cta_items[2 * b + 1] = 0;
        }
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        hdr->n_items = (int32_t)(grun + v.P);       // bound on the item indices
        hdr->n_combine = s_nc;
        hdr->pad[0] = v.P;
        hdr->pad[1] = s_np;                         // partial pieces of all split groups
    }
}

// ---------------------------------------------------------------------------
// k_readout_simt: CUDA-core flash readout (fp32 path; any dtype)
// ---------------------------------------------------------------------------
// One CTA per work item of BM = 32 query rows.  A row is owned by TPR = d/16
// threads, each holding 16 dimensions of q~ and of the output accumulator.
// Keys are staged 32 at a time in shared memory as fp32.
constexpr int SIMT_BM = 32;
constexpr int SIMT_BN = 32;

template <typename T>
__global__ void __launch_bounds__(512) k_readout_simt(ReadoutArgs a)
{
    pdl_wait();
    extern __shared__ __align__(16) float sm[];
    const int d = a.d;
    const int TPR = d / 16;
    float *sK = sm;                      // [SIMT_BN][d]
    float *sV = sm + SIMT_BN * d;        // [SIMT_BN][d]
    const int it_end = a.cta_items[2 * blockIdx.x + 1];
    for (int it = a.cta_items[2 * blockIdx.x]; it < it_end; ++it) {
        const WorkItem w = a.items[it];
        const RangeSet rs = a.ranges[w.u];
        const int r = threadIdx.x / TPR;
        const int part = threadIdx.x % TPR;
        const int j = w.qt * SIMT_BM + r;
        const bool valid = j < rs.cnt;
        const int g = a.unit_group[w.u];
        if (g < 0 || g >= a.G) {                 // uniform over the CTA
            if (threadIdx.x == 0) latch_status(a.status, RS3_EINVAL);
            continue;
        }
        int cell = 0;
        if (valid) cell = a.idx[(int64_t)w.u * a.k_max + j];
        if (cell < 0 || cell >= a.mn) cell = 0;
        const int c0 = w.h * d + part * 16;
        float qv[16];
        {
            const T *qr = static_cast<const T *>(a.q) + ((int64_t)g * a.mn + cell) * a.D + c0;
            load16(qr, qv);
            if (a.rope) {
                const float *f = a.rope + ((int64_t)cell * (d / 2) + part * 8) * 2;
#pragma unroll
                for (int p = 0; p < 8; ++p) {
                    const float cs = f[2 * p], sn = f[2 * p + 1];
                    const float x0 = qv[2 * p], x1 = qv[2 * p + 1];
                    qv[2 * p] = x0 * cs - x1 * sn;
                    qv[2 * p + 1] = x0 * sn + x1 * cs;
                }
            }
#pragma unroll
            for (int k = 0; k < 16; ++k) qv[k] *= a.scale_log2;
        }
        float o[16];
#pragma unroll
        for (int k = 0; k < 16; ++k) o[k] = 0.f;
        float mrun = -INFINITY, lrun = 0.f;
        const T *Kb = static_cast<const T *>(a.k_store) + (int64_t)w.u * a.rows_per_unit * a.D;
        const T *Vb = static_cast<const T *>(a.v_store) + (int64_t)w.u * a.rows_per_unit * a.D;
        for (int t = w.tile_begin; t < w.tile_end; ++t) {
            int64_t row0;
            int nvalid;
            tile_rows(rs, t, SIMT_BN, row0, nvalid);
            if (nvalid <= 0) continue;           // uniform over the CTA
            __syncthreads();
            // stage keys / values of this head as fp32
            const int vec_per_row = d / 4;
            for (int e = threadIdx.x; e < SIMT_BN * vec_per_row; e += blockDim.x) {
                const int kk = e / vec_per_row, c4 = (e % vec_per_row) * 4;
                float4 kv = make_float4(0.f, 0.f, 0.f, 0.f), vv = kv;
                if (kk < nvalid) {
                    kv = load4(Kb + (row0 + kk) * a.D + w.h * d + c4);
                    vv = load4(Vb + (row0 + kk) * a.D + w.h * d + c4);
                }
                *reinterpret_cast<float4 *>(sK + kk * d + c4) = kv;
                *reinterpret_cast<float4 *>(sV + kk * d + c4) = vv;
            }
            __syncthreads();
            float s[SIMT_BN];
#pragma unroll
            for (int kk = 0; kk < SIMT_BN; ++kk) {
                const float *kr = sK + kk * d + part * 16;
                float acc = 0.f;
#pragma unroll
                for (int k = 0; k < 16; ++k) acc = fmaf(qv[k], kr[k], acc);
                s[kk] = acc;
            }
            for (int off = TPR >> 1; off >= 1; off >>= 1) {
#pragma unroll
                for (int kk = 0; kk < SIMT_BN; ++kk) s[kk] += __shfl_xor_sync(0xffffffffu, s[kk], off);
            }
            float mt = -INFINITY;
#pragma unroll
            for (int kk = 0; kk < SIMT_BN; ++kk) {
                if (kk >= nvalid) s[kk] = -INFINITY;
                mt = fmaxf(mt, s[kk]);
            }
            const float mnew = fmaxf(mrun, mt);
            const float alpha = exp2f(mrun - mnew);
            lrun *= alpha;
#pragma unroll
            for (int k = 0; k < 16; ++k) o[k] *= alpha;
#pragma unroll
            for (int kk = 0; kk < SIMT_BN; ++kk) {
                const float p = exp2f(s[kk] - mnew);
                lrun += p;
                const float *vr = sV + kk * d + part * 16;
#pragma unroll
                for (int k = 0; k < 16; ++k) o[k] = fmaf(p, vr[k], o[k]);
            }
            mrun = mnew;
        }
        if (valid) {
            if (w.slot < 0) {
                const float inv = lrun > 0.f ? 1.f / lrun : 0.f;
#pragma unroll
                for (int k = 0; k < 16; ++k) o[k] *= inv;
                store_out16<T>(a, w.u, cell, c0, o);
            } else {
                float *po = a.part_o + ((int64_t)w.slot * a.BM + r) * d + part * 16;
#pragma unroll
                for (int k = 0; k < 16; k += 4)
                    *reinterpret_cast<float4 *>(po + k) = make_float4(o[k], o[k + 1], o[k + 2], o[k + 3]);
                if (part == 0) {
                    float2 *pm = reinterpret_cast<float2 *>(a.part_ml) + (int64_t)w.slot * a.BM + r;
                    *pm = make_float2(mrun, lrun);
                }
            }
        }
    }
}

// ---------------------------------------------------------------------------
// k_combine: log-sum-exp merge of split-KV partials, then the scatter
// ---------------------------------------------------------------------------
// A warp takes one output row: the row's splits' (m, l) pairs give M = max m
// and L = sum 2^(m - M) l; each lane accumulates E columns per CW-column chunk
// over the splits with weight 2^(m_s - M) (eight splits' loads in flight at a
// time) and stores residual + sum / L.  When the groups are split many ways
// (small frames spread over all SMs) a row is shared by one warp per chunk;
// otherwise one warp does the whole row (lanes striding the columns four at a
// time), so the loads of the row's entry, cell and (m, l) pairs are not
// repeated per chunk.
template <typename T, int E>
__device__ __forceinline__ void store_out_e(const ReadoutArgs &a, int u, int cell, int c, const float *o);

template <>
__device__ __forceinline__ void store_out_e<float, 1>(const ReadoutArgs &a, int u, int cell, int c, const float *o)
{
    const int64_t off = ((int64_t)u * a.mn + cell) * a.D + c;
    const float r = a.residual ? static_cast<const float *>(a.residual)[off] : 0.f;
    static_cast<float *>(a.out)[off] = r + o[0];
}

template <>
__device__ __forceinline__ void store_out_e<float, 2>(const ReadoutArgs &a, int u, int cell, int c, const float *o)
{
    const int64_t off = ((int64_t)u * a.mn + cell) * a.D + c;
    float2 r = make_float2(0.f, 0.f);
    if (a.residual) r = *reinterpret_cast<const float2 *>(static_cast<const float *>(a.residual) + off);
    *reinterpret_cast<float2 *>(static_cast<float *>(a.out) + off) = make_float2(r.x + o[0], r.y + o[1]);
}

template <>
__device__ __forceinline__ void store_out_e<uint16_t, 1>(const ReadoutArgs &a, int u, int cell, int c, const float *o)
{
    const int64_t off = ((int64_t)u * a.mn + cell) * a.D + c;
    const float r = a.residual ? bf16_bits_to_float(static_cast<const uint16_t *>(a.residual)[off]) : 0.f;
    static_cast<uint16_t *>(a.out)[off] = float_to_bf16_bits(r + o[0]);
}

template <>
__device__ __forceinline__ void store_out_e<uint16_t, 2>(const ReadoutArgs &a, int u, int cell, int c, const float *o)
{
    const int64_t off = ((int64_t)u * a.mn + cell) * a.D + c;
    float r0 = 0.f, r1 = 0.f;
    if (a.residual) {
        const uint32_t x = *reinterpret_cast<const uint32_t *>(static_cast<const uint16_t *>(a.residual) + off);
        r0 = __uint_as_float(x << 16);
        r1 = __uint_as_float(x & 0xffff0000u);
    }
    *reinterpret_cast<uint32_t *>(static_cast<uint16_t *>(a.out) + off) = pack_bf16x2(r0 + o[0], r1 + o[1]);
}

template <typename T, int E>
__global__ void __launch_bounds__(256) k_combine(ReadoutArgs a)
{
    pdl_wait();
    constexpr int CW = 32 * E;                      // columns per warp
    const int d = a.d;
    // chunked tasks only when the groups are split more than four ways on
    // average (one decision for the launch, so no task is spent idle)
    const int n_comb = a.header->n_combine;
    const bool chunked = a.header->pad[1] > 4 * n_comb;
    const int chunks = chunked ? (d + CW - 1) / CW : 1;   // tasks per row
    const int64_t n_tasks = (int64_t)n_comb * a.BM * chunks;
    const int lane = threadIdx.x & 31;
    const float2 *pm = reinterpret_cast<const float2 *>(a.part_ml);
    for (int64_t task = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; task < n_tasks;
         task += ((int64_t)gridDim.x * blockDim.x) >> 5) {
        const int64_t gr = task / chunks;
        const int chunk = (int)(task % chunks);
        const int ci = (int)(gr / a.BM), r = (int)(gr % a.BM);
        const CombineItem c = a.combine[ci];
        if (c.nsplit <= 0) continue;                   // warp-uniform
        const int j = c.qt * a.BM + r;
        if (j >= c.pad[1]) continue;                   // the unit's kept queries (warp-uniform)
        // piece 0 of the group is at slot0; piece s >= 1 is the first item of
        // slice b0 + s, partial slot 2 (b0 + s).  slot(s) = 2 (b0 + s) + d0 [s = 0]
        // with d0 = slot0 - 2 b0: a select, no branch, so every piece's loads
        // can be in flight together
        const int64_t b0 = c.pad[0], d0 = (int64_t)c.slot0 - 2 * b0;
        const float2 *ml = pm + 2 * b0 * a.BM + r;                 // piece s at ml[slot_rel(s) BM]
        const int64_t sstride = (int64_t)a.BM * d;                 // one slot
#define SLOT_REL(s_) (2 * (int64_t)(s_) + ((s_) == 0 ? d0 : 0))
        if (!chunked) {
            // One round trip for the row's cell, the pieces' (m, l) pairs (lane
            // s holds piece s) and the first MP pieces' partial columns (lanes
            // stride the row four columns at a time); the weights follow.
            constexpr int MP = 4;
            int cell = a.idx[(int64_t)c.u * a.k_max + j];
            const float2 mv = lane < c.nsplit ? ml[SLOT_REL(lane) * a.BM] : make_float2(-INFINITY, 0.f);
            const float *base = a.part_o + (2 * b0 * a.BM + r) * d;
            float4 pf[MP][2];
#pragma unroll
            for (int q = 0; q < MP; ++q)
#pragma unroll
                for (int cb = 0; cb < 2; ++cb) {
                    const int c4 = lane * 4 + 128 * cb;
                    pf[q][cb] = (q < c.nsplit && c4 < d)
                                    ? __ldcs(reinterpret_cast<const float4 *>(base + SLOT_REL(q) * sstride + c4))
                                    : make_float4(0.f, 0.f, 0.f, 0.f);
                }
            float M = mv.x;
            for (int s = lane + 32; s < c.nsplit; s += 32) M = fmaxf(M, ml[SLOT_REL(s) * a.BM].x);
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
            float L = 0.f;
            if (M != -INFINITY) {
                if (lane < c.nsplit) L = exp2f(mv.x - M) * mv.y;
                for (int s = lane + 32; s < c.nsplit; s += 32) {
                    const float2 v = ml[SLOT_REL(s) * a.BM];
                    L += exp2f(v.x - M) * v.y;
                }
            }
            L = warp_sum(L);
            const float inv = L > 0.f ? 1.f / L : 0.f;
            float wq[MP];
#pragma unroll
            for (int q = 0; q < MP; ++q) {
                const float mq = __shfl_sync(0xffffffffu, mv.x, q);
                wq[q] = (q < c.nsplit && M != -INFINITY) ? exp2f(mq - M) : 0.f;
            }
            if (cell < 0 || cell >= a.mn) cell = 0;
#pragma unroll
            for (int cb = 0; cb < 2; ++cb) {
                const int c4 = lane * 4 + 128 * cb;
                if (c4 >= d) continue;
                float4 acc = make_float4(0.f, 0.f, 0.f, 0.f);
#pragma unroll
                for (int q = 0; q < MP; ++q) {
                    acc.x = fmaf(wq[q], pf[q][cb].x, acc.x);
                    acc.y = fmaf(wq[q], pf[q][cb].y, acc.y);
                    acc.z = fmaf(wq[q], pf[q][cb].z, acc.z);
                    acc.w = fmaf(wq[q], pf[q][cb].w, acc.w);
                }
                for (int s = MP; s < c.nsplit; ++s) {
                    const float ws = M == -INFINITY ? 0.f : exp2f(ml[SLOT_REL(s) * a.BM].x - M);
                    const float4 po = __ldcs(reinterpret_cast<const float4 *>(base + SLOT_REL(s) * sstride + c4));
                    acc.x = fmaf(ws, po.x, acc.x);
                    acc.y = fmaf(ws, po.y, acc.y);
                    acc.z = fmaf(ws, po.z, acc.z);
                    acc.w = fmaf(ws, po.w, acc.w);
                }
                const float o4[4] = {acc.x * inv, acc.y * inv, acc.z * inv, acc.w * inv};
                store_out4<T>(a, c.u, cell, c.h * d + c4, o4);
            }
            continue;
        }
        int cell = a.idx[(int64_t)c.u * a.k_max + j];
        if (cell < 0 || cell >= a.mn) cell = 0;
        float M = -INFINITY;
        for (int s = lane; s < c.nsplit; s += 32) M = fmaxf(M, ml[SLOT_REL(s) * a.BM].x);
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) M = fmaxf(M, __shfl_xor_sync(0xffffffffu, M, o));
        float L = 0.f;
        if (M != -INFINITY)
            for (int s = lane; s < c.nsplit; s += 32) {
                const float2 v = ml[SLOT_REL(s) * a.BM];
                L += exp2f(v.x - M) * v.y;
            }
        L = warp_sum(L);
        const float inv = L > 0.f ? 1.f / L : 0.f;
        const int col = chunk * CW + lane * E;
        if (col >= d) continue;                          // d < 32 only; no collectives below
        const float *base = a.part_o + (2 * b0 * a.BM + r) * d + col;
        float acc[E];
#pragma unroll
        for (int e = 0; e < E; ++e) acc[e] = 0.f;
#pragma unroll 8
        for (int s = 0; s < c.nsplit; ++s) {
            const float ws = M == -INFINITY ? 0.f : exp2f(ml[SLOT_REL(s) * a.BM].x - M);
            if constexpr (E == 2) {
                const float2 po = __ldcs(reinterpret_cast<const float2 *>(base + SLOT_REL(s) * sstride));
                acc[0] = fmaf(ws, po.x, acc[0]);
                acc[1] = fmaf(ws, po.y, acc[1]);
            } else {
                acc[0] = fmaf(ws, __ldcs(base + SLOT_REL(s) * sstride), acc[0]);
            }
        }
#undef SLOT_REL
#pragma unroll
        for (int e = 0; e < E; ++e) acc[e] *= inv;
        store_out_e<T, E>(a, c.u, cell, c.h * d + col, acc);
    }
}

}  // namespace

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
namespace {

// Bounds of the stream-K plan: item indices < groups + CTAs (group + slice);
// a CTA has at most two partial items (slots 2b, 2b + 1); at most one merge
// entry per CTA and per group.
ReadoutLayout readout_layout(int U, int H, int d, int k_max, int BM, int grid)
{
    ReadoutLayout L;
    const int64_t nq = k_max > 0 ? (k_max + BM - 1) / BM : 1;
    const int64_t groups = (int64_t)U * H * nq;
    L.max_slots = 2 * (int64_t)grid;
    L.max_combine = groups < grid ? groups : grid;   // at most one per CTA slice and per group
    L.max_items = groups + grid;
    size_t off = 0;
    L.header = off;
    off = align_up(off + sizeof(ReadoutHeader), 256);
    L.cta_items = off;
    off = align_up(off + (size_t)grid * 2 * 4, 256);   // [begin, end) per CTA
    L.ranges = off;
    off = align_up(off + (size_t)U * sizeof(RangeSet), 256);
    L.items = off;
    off = align_up(off + (size_t)L.max_items * sizeof(WorkItem), 256);
    L.combine = off;
    off = align_up(off + (size_t)L.max_combine * sizeof(CombineItem), 256);
    L.part_o = off;
    off = align_up(off + (size_t)L.max_slots * BM * d * 4, 256);
    L.part_ml = off;
    off = align_up(off + (size_t)L.max_slots * BM * 8, 256);
    L.total = off;
    return L;
}

}  // namespace

namespace {
std::atomic<uint64_t> g_wait_ns{1000000000ull};
}

extern "C" void rs3_set_wait_limit_ns(uint64_t ns) { g_wait_ns.store(ns); }
extern "C" uint64_t rs3_get_wait_limit_ns(void) { return g_wait_ns.load(); }

ReadoutPath choose_readout_path(rs3_dtype dtype, int d)
{
    ReadoutPath p;
    const int n_sm = rs3_sm_count();
    if (dtype == RS3_BF16 && rs3_tc_supported(d)) {
        p.kind = 1;
        p.BM = 128;
        p.BN = rs3_tc_block_n(d);
        p.grid = n_sm;                 // one persistent CTA per SM
    } else {
        p.kind = 0;
        p.BM = SIMT_BM;
        p.BN = SIMT_BN;
        p.grid = 4 * n_sm;
    }
    return p;
}

extern "C" size_t rs3_readout_workspace_bytes(int U, int H, int d, int k_max, rs3_dtype dtype)
{
    if (U < 1 || H < 1 || d < 1 || k_max < 0) return 0;
    const ReadoutPath p = choose_readout_path(dtype, d);
    return readout_layout(U, H, d, k_max, p.BM, p.grid).total;
}

rs3_status rs3_readout_prepare(const void *q, rs3_dtype dtype, int G, int mn, int H, int d,
                               const int32_t *unit_group, const int32_t *idx, const int32_t *count,
                               int k_max, const rs3_bank *bank, const float *rope,
                               const void *residual, void *out, float scale, void *workspace,
                               size_t workspace_bytes, int32_t *status, ReadoutArgs *a,
                               ReadoutPath *path, int64_t *grid_items, int64_t *grid_combine)
{
    if (!q || !unit_group || !idx || !count || !bank || !out || !workspace || !status)
        return RS3_EINVAL;
    if (bank->magic != RS3_BANK_MAGIC || !bank->meta || !bank->k_store || !bank->v_store)
        return RS3_EINVAL;
    if (dtype != RS3_F32 && dtype != RS3_BF16) return RS3_EINVAL;
    if ((int)dtype != bank->dtype || H != bank->H || d != bank->d) return RS3_EINVAL;
    if (G < 1 || mn < 1 || H < 1 || d < 1 || k_max < 0) return RS3_EINVAL;
    if (mn > RS3_MAX_MN || bank->U > RS3_MAX_UNITS) return RS3_EUNSUPPORTED;
    if (d < 16 || d > 256 || (d & (d - 1)) != 0) return RS3_EUNSUPPORTED;
    if (!rs3_aligned16(q) || !rs3_aligned16(out) || !rs3_aligned16(workspace) ||
        (residual && !rs3_aligned16(residual)) || (rope && !rs3_aligned16(rope)))
        return RS3_EINVAL;
    const ReadoutPath p = choose_readout_path(dtype, d);
    const ReadoutLayout L = readout_layout(bank->U, H, d, k_max, p.BM, p.grid);
    // work-item indices (group + slice) and item ranges are 32-bit
    if (L.max_items >= ((int64_t)1 << 30) || L.max_slots >= ((int64_t)1 << 30)) return RS3_EUNSUPPORTED;
    if (workspace_bytes < L.total) return RS3_ECAPACITY;
    uint8_t *ws = static_cast<uint8_t *>(workspace);
    a->q = q;
    a->k_store = bank->k_store;
    a->v_store = bank->v_store;
    a->meta = static_cast<const int64_t *>(bank->meta);
    a->meta_stride_words = bank->meta_stride / 8;
    a->pinned_cap = bank->pinned_cap;
    a->ring_cap = bank->ring_cap;
    a->rows_per_unit = bank->rows_per_unit;
    a->n_ptr = bank->n_ptr;
    a->unit_group = unit_group;
    a->idx = idx;
    a->count = count;
    a->rope = rope;
    a->residual = residual;
    a->out = out;
    a->status = status;
    a->U = bank->U;
    a->G = G;
    a->mn = mn;
    a->H = H;
    a->d = d;
    a->D = H * d;
    a->k_max = k_max;
    a->BM = p.BM;
    a->BN = p.BN;
    a->n_sm = rs3_sm_count();
    a->min_chunk = p.kind == 1 ? 2 : 4;
    // start-up cost of a piece in tile slots: on the tensor-core path a
    // sweep of 4..32 over the 1- and 8-object sequences was best at 8..16
    a->plan_ov = p.kind == 1 ? 12 : 1;
    a->max_slots = L.max_slots;
    a->max_items = L.max_items;
    a->grid_ctas = p.grid;
    a->cta_items = reinterpret_cast<int32_t *>(ws + L.cta_items);
    const float sc = scale > 0.f ? scale : 1.0f / sqrtf((float)d);
    a->scale_log2 = sc * 1.4426950408889634f;
    a->wait_ns = g_wait_ns.load();
    a->header = reinterpret_cast<ReadoutHeader *>(ws + L.header);
    a->ranges = reinterpret_cast<RangeSet *>(ws + L.ranges);
    a->items = reinterpret_cast<WorkItem *>(ws + L.items);
    a->combine = reinterpret_cast<CombineItem *>(ws + L.combine);
    a->part_o = reinterpret_cast<float *>(ws + L.part_o);
    a->part_ml = reinterpret_cast<float *>(ws + L.part_ml);
    *path = p;
    *grid_items = L.max_items;
    *grid_combine = L.max_combine;
    return RS3_OK;
}

namespace {

// pass-through of the unselected cells (out of place only) and the plan
rs3_status launch_plan(const ReadoutArgs &a, cudaStream_t st, rs3_dtype dtype)
{
    if (a.residual != a.out) {
        const int64_t nvec = (int64_t)a.U * a.mn * a.D * (dtype == RS3_BF16 ? 2 : 4) / 16;
        int64_t blocks = (nvec + 255) / 256;
        const int64_t cap = (int64_t)a.n_sm * 8;
        if (blocks > cap) blocks = cap;
        launch_pdl(k_passthrough, dim3((unsigned)blocks), dim3(256), 0, st,
                   static_cast<const uint4 *>(a.residual), static_cast<uint4 *>(a.out), nvec);
        if (cudaGetLastError() != cudaSuccess) return RS3_ECUDA;
    }
    // plan shared memory: unit slot bases and widths (int64), group bases, tiles, kept queries (int32)
    const size_t plan_smem = (size_t)(2 * a.U + 1) * 8 + (size_t)(3 * a.U + 1) * 4;
    if (rs3_kernel_smem((const void *)k_plan, plan_smem) != RS3_OK) return RS3_EUNSUPPORTED;
    launch_pdl(k_plan, dim3(1), dim3(PLAN_THREADS), plan_smem, st, a);
    return cudaGetLastError() != cudaSuccess ? RS3_ECUDA : RS3_OK;
}

// the attention kernel over the plan in the workspace
rs3_status launch_run(const ReadoutArgs &a, const ReadoutPath &p, rs3_dtype dtype, cudaStream_t st)
{
    if (p.kind == 1) return rs3_launch_tc_readout(a, st);
    const size_t smem = (size_t)2 * SIMT_BN * a.d * sizeof(float);
    const int threads = 2 * a.d;
    const int64_t blocks = a.grid_ctas;
    if (rs3_kernel_smem(dtype == RS3_BF16 ? (const void *)k_readout_simt<uint16_t>
                                          : (const void *)k_readout_simt<float>, smem) != RS3_OK)
        return RS3_ECUDA;
    if (dtype == RS3_BF16)
        launch_pdl(k_readout_simt<uint16_t>, dim3((unsigned)blocks), dim3(threads), smem, st, a);
    else
        launch_pdl(k_readout_simt<float>, dim3((unsigned)blocks), dim3(threads), smem, st, a);
    return cudaGetLastError() == cudaSuccess ? RS3_OK : RS3_ECUDA;
}

// merge of the split-KV partials and their scatter
rs3_status launch_merge(const ReadoutArgs &a, int64_t max_combine, rs3_dtype dtype, cudaStream_t st)
{
    // one warp per (partial row, 64-column chunk; 32 for d < 64)
    const int ce = a.d >= 64 ? 2 : 1;
    const int64_t chunks = (a.d + 32 * ce - 1) / (32 * ce);
    int64_t cblocks = (max_combine * a.BM * chunks + 7) / 8;
    const int64_t ccap = (int64_t)a.n_sm * 16;
    if (cblocks > ccap) cblocks = ccap;
    if (cblocks < 1) cblocks = 1;
    if (dtype == RS3_BF16) {
        if (ce == 2) launch_pdl(k_combine<uint16_t, 2>, dim3((unsigned)cblocks), dim3(256), 0, st, a);
        else launch_pdl(k_combine<uint16_t, 1>, dim3((unsigned)cblocks), dim3(256), 0, st, a);
    } else {
        if (ce == 2) launch_pdl(k_combine<float, 2>, dim3((unsigned)cblocks), dim3(256), 0, st, a);
        else launch_pdl(k_combine<float, 1>, dim3((unsigned)cblocks), dim3(256), 0, st, a);
    }
    return cudaGetLastError() == cudaSuccess ? RS3_OK : RS3_ECUDA;
}

}  // namespace

rs3_status rs3_readout_launch(const ReadoutArgs &a, const ReadoutPath &p, int64_t max_items,
                              int64_t max_combine, rs3_dtype dtype, cudaStream_t st, int phases)
{
    (void)max_items;
    if (phases & RS3_PHASE_PLAN) {
        const rs3_status s = launch_plan(a, st, dtype);
        if (s != RS3_OK) return s;
    }
    if (phases & RS3_PHASE_RUN) {
        const rs3_status s = launch_run(a, p, dtype, st);
        if (s != RS3_OK) return s;
    }
    if (phases & RS3_PHASE_MERGE) return launch_merge(a, max_combine, dtype, st);
    return RS3_OK;
}

namespace {

rs3_status readout_call(const void *q, rs3_dtype dtype, int G, int mn, int H, int d, const int32_t *unit_group,
                        const int32_t *idx, const int32_t *count, int k_max, const rs3_bank *bank,
                        const float *rope, const void *residual, void *out, float scale, void *workspace,
                        size_t workspace_bytes, int32_t *status, rs3_stream_t stream, int phases)
{
    ReadoutArgs a;
    ReadoutPath p;
    int64_t gi, gc;
    const rs3_status s = rs3_readout_prepare(q, dtype, G, mn, H, d, unit_group, idx, count, k_max,
                                             bank, rope, residual, out, scale, workspace,
                                             workspace_bytes, status, &a, &p, &gi, &gc);
    if (s != RS3_OK) return s;
    return rs3_readout_launch(a, p, gi, gc, dtype, reinterpret_cast<cudaStream_t>(stream), phases);
}

}  // namespace

extern "C" rs3_status rs3_memory_readout(const void *q, rs3_dtype dtype, int G, int mn, int H,
                                         int d, const int32_t *unit_group, const int32_t *idx,
                                         const int32_t *count, int k_max, const rs3_bank *bank,
                                         const float *rope, const void *residual, void *out,
                                         float scale, void *workspace, size_t workspace_bytes,
                                         int32_t *status, rs3_stream_t stream)
{
    return readout_call(q, dtype, G, mn, H, d, unit_group, idx, count, k_max, bank, rope, residual, out, scale,
                        workspace, workspace_bytes, status, stream, RS3_PHASE_ATTEND | RS3_PHASE_MERGE);
}

extern "C" rs3_status rs3_memory_readout_attend(const void *q, rs3_dtype dtype, int G, int mn, int H,
                                                int d, const int32_t *unit_group, const int32_t *idx,
                                                const int32_t *count, int k_max, const rs3_bank *bank,
                                                const float *rope, const void *residual, void *out,
                                                float scale, void *workspace, size_t workspace_bytes,
                                                int32_t *status, rs3_stream_t stream)
{
    return readout_call(q, dtype, G, mn, H, d, unit_group, idx, count, k_max, bank, rope, residual, out, scale,
                        workspace, workspace_bytes, status, stream, RS3_PHASE_ATTEND);
}

extern "C" rs3_status rs3_memory_readout_plan(const void *q, rs3_dtype dtype, int G, int mn, int H,
                                              int d, const int32_t *unit_group, const int32_t *idx,
                                              const int32_t *count, int k_max, const rs3_bank *bank,
                                              const float *rope, const void *residual, void *out,
                                              float scale, void *workspace, size_t workspace_bytes,
                                              int32_t *status, rs3_stream_t stream)
{
    return readout_call(q, dtype, G, mn, H, d, unit_group, idx, count, k_max, bank, rope, residual, out, scale,
                        workspace, workspace_bytes, status, stream, RS3_PHASE_PLAN);
}

extern "C" rs3_status rs3_memory_readout_run(const void *q, rs3_dtype dtype, int G, int mn, int H,
                                             int d, const int32_t *unit_group, const int32_t *idx,
                                             const int32_t *count, int k_max, const rs3_bank *bank,
                                             const float *rope, const void *residual, void *out,
                                             float scale, void *workspace, size_t workspace_bytes,
                                             int32_t *status, rs3_stream_t stream)
{
    return readout_call(q, dtype, G, mn, H, d, unit_group, idx, count, k_max, bank, rope, residual, out, scale,
                        workspace, workspace_bytes, status, stream, RS3_PHASE_RUN);
}

extern "C" rs3_status rs3_memory_readout_merge(const void *q, rs3_dtype dtype, int G, int mn, int H,
                                               int d, const int32_t *unit_group, const int32_t *idx,
                                               const int32_t *count, int k_max, const rs3_bank *bank,
                                               const float *rope, const void *residual, void *out,
                                               float scale, void *workspace, size_t workspace_bytes,
                                               int32_t *status, rs3_stream_t stream)
{
    return readout_call(q, dtype, G, mn, H, d, unit_group, idx, count, k_max, bank, rope, residual, out, scale,
                        workspace, workspace_bytes, status, stream, RS3_PHASE_MERGE);
}
