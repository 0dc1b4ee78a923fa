// rs3_select.cu -- read-side keep-set K_r (Sec. 3.1: Eq. 1, 2, 4, 5) and the
// write keep-set K_w (Sec. 3.2: Eq. 8).
//
// Three launches per frame, all integer-exact:
//   k_prior   one CTA per unit: bbox + tracker update (Eq. 4 state), prior as
//             a separable Chebyshev dilation in shared memory, written as a
//             byte mask and OR-ed (ballot + atomicOr) into a per-group bitmap
//             of the cells that need an energy.
//   k_energy  warp-per-row ||z||^2 over the needed rows only, in the canonical
//             fp32 order (16-byte loads, fmaf chain, xor-shuffle tree).
//   k_select  one CTA per unit: 4-pass 8-bit radix select of the k-th largest
//             energy key in shared memory, then a ballot/popc stream compaction
//             that emits the keep-set in ascending cell order.
#include "rs3_internal.cuh"

#include <climits>
#include <cmath>

namespace {

constexpr uint32_t KEY_NONE = 0xFFFFFFFFu;   // not in the prior (never a finite energy's bits)

enum { PMODE_EMPTY = 0, PMODE_MASK = 1, PMODE_BOX = 2, PMODE_BAD = 3 };

__device__ __forceinline__ uint32_t lanemask_lt()
{
    uint32_t m;
    asm("mov.u32 %0, %%lanemask_lt;" : "=r"(m));
    return m;
}

// Block-wide min/max reduction of four ints (y0, x0 by min; y1, x1 by max).
__device__ void block_bbox(int &y0, int &x0, int &y1, int &x1)
{
    __shared__ int red[4][32];
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        y0 = min(y0, __shfl_xor_sync(0xffffffffu, y0, o));
        x0 = min(x0, __shfl_xor_sync(0xffffffffu, x0, o));
        y1 = max(y1, __shfl_xor_sync(0xffffffffu, y1, o));
        x1 = max(x1, __shfl_xor_sync(0xffffffffu, x1, o));
    }
    if (lane == 0) {
        red[0][warp] = y0; red[1][warp] = x0; red[2][warp] = y1; red[3][warp] = x1;
    }
    __syncthreads();
    const int nw = blockDim.x >> 5;
    if (warp == 0) {
        y0 = lane < nw ? red[0][lane] : INT_MAX;
        x0 = lane < nw ? red[1][lane] : INT_MAX;
        y1 = lane < nw ? red[2][lane] : -1;
        x1 = lane < nw ? red[3][lane] : -1;
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            y0 = min(y0, __shfl_xor_sync(0xffffffffu, y0, o));
            x0 = min(x0, __shfl_xor_sync(0xffffffffu, x0, o));
            y1 = max(y1, __shfl_xor_sync(0xffffffffu, y1, o));
            x1 = max(x1, __shfl_xor_sync(0xffffffffu, x1, o));
        }
        if (lane == 0) {
            red[0][0] = y0; red[1][0] = x0; red[2][0] = y1; red[3][0] = x1;
        }
    }
    __syncthreads();
    y0 = red[0][0]; x0 = red[1][0]; y1 = red[2][0]; x1 = red[3][0];
    __syncthreads();
}

// Chebyshev dilation of sIn by r into out(i) (called per cell after the row
// pass).  Row pass: sTmp[y][x] = OR sIn[y][x-r .. x+r].
__device__ void row_pass(const uint8_t *sIn, uint8_t *sTmp, int m, int n, int r)
{
    const int mn = m * n;
    for (int i = threadIdx.x; i < mn; i += blockDim.x) {
        const int y = i / n, x = i - y * n;
        const int xa = max(0, x - r), xb = min(n - 1, x + r);
        uint8_t v = 0;
        for (int xx = xa; xx <= xb && !v; ++xx) v |= sIn[y * n + xx];
        sTmp[i] = v;
    }
}

__device__ __forceinline__ uint8_t col_value(const uint8_t *sTmp, int m, int n, int r, int i)
{
    const int y = i / n, x = i - y * n;
    const int ya = max(0, y - r), yb = min(m - 1, y + r);
    uint8_t v = 0;
    for (int yy = ya; yy <= yb && !v; ++yy) v |= sTmp[yy * n + x];
    return v;
}

// ---------------------------------------------------------------------------
// k_prior: Eq. 1 / Eq. 2 / Eq. 4 and the tracker update of Algorithm 1
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024)
k_prior(const uint8_t *__restrict__ masks, int m, int n, const int32_t *__restrict__ unit_group,
        int G, rs3_track *__restrict__ track, int r_s, int c, int bbox_mode,
        uint8_t *__restrict__ prior, uint32_t *__restrict__ need, int32_t *status)
{
    pdl_wait();
    extern __shared__ __align__(16) uint8_t smem[];
    const int mn = m * n;
    const int u = blockIdx.x;
    uint8_t *sM = smem;
    uint8_t *sT = smem + ((mn + 15) & ~15);
    __shared__ int s_mode, s_r, s_g, s_box[4];

    // the unit's group and tracker state load beside the mask (thread 0
    // decides the prior's mode once the mask's box is known)
    int g0 = 0;
    rs3_track t0 = {};
    if (threadIdx.x == 0) {
        g0 = unit_group[u];
        t0 = track[u];
    }
    const uint8_t *Mu = masks + (size_t)u * mn;
    int y0 = INT_MAX, x0 = INT_MAX, y1 = -1, x1 = -1;
#pragma unroll 4
    for (int i = threadIdx.x; i < mn; i += blockDim.x) {
        const uint8_t v = Mu[i] != 0;
        sM[i] = v;
        if (v) {
            const int y = i / n, x = i - y * n;
            y0 = min(y0, y); y1 = max(y1, y);
            x0 = min(x0, x); x1 = max(x1, x);
        }
    }
    block_bbox(y0, x0, y1, x1);   // contains __syncthreads

    if (threadIdx.x == 0) {
        const int g = g0;
        rs3_track t = t0;
        int mode, r = 0;
        if (g < 0 || g >= G) {
            latch_status(status, RS3_EINVAL);
            mode = PMODE_BAD;
        } else if (y1 >= 0) {                       // non-empty mask
            t.y0 = y0; t.x0 = x0; t.y1 = y1; t.x1 = x1;
            t.valid = 1;
            t.streak = 0;
            mode = bbox_mode ? PMODE_BOX : PMODE_MASK;
            r = r_s;
        } else {                                    // empty: streak-counted fallback
            if (t.streak < 0x3fffffff) t.streak += 1;
            if (t.valid) {
                mode = PMODE_BOX;
                r = r_s + min(t.streak, c);
            } else {
                mode = PMODE_EMPTY;
            }
        }
        if (mode != PMODE_BAD) track[u] = t;
        s_mode = mode;
        s_r = r;
        s_g = g;
        s_box[0] = t.y0; s_box[1] = t.x0; s_box[2] = t.y1; s_box[3] = t.x1;
    }
    __syncthreads();
    const int mode = s_mode, r = s_r, g = s_g;
    if (mode == PMODE_MASK) {
        row_pass(sM, sT, m, n, r);
        __syncthreads();
    }
    const int by0 = s_box[0] - r, bx0 = s_box[1] - r, by1 = s_box[2] + r, bx1 = s_box[3] + r;
    const int nwords = (mn + 31) >> 5;
    uint8_t *Pu = prior + (size_t)u * mn;
    for (int base = 0; base < mn; base += blockDim.x) {
        const int i = base + threadIdx.x;
        uint8_t v = 0;
        if (i < mn) {
            if (mode == PMODE_MASK) {
                v = col_value(sT, m, n, r, i);
            } else if (mode == PMODE_BOX) {
                const int y = i / n, x = i - y * n;
                v = (y >= by0 && y <= by1 && x >= bx0 && x <= bx1) ? 1 : 0;
            }
            Pu[i] = v;
        }
        const uint32_t bal = __ballot_sync(0xffffffffu, v != 0);
        if ((threadIdx.x & 31) == 0 && bal != 0 && mode != PMODE_BAD && i < mn)
            atomicOr(&need[(size_t)g * nwords + (i >> 5)], bal);
    }
}

// ---------------------------------------------------------------------------
// k_energy: canonical fp32 ||z||^2 of the rows some prior needs (Eq. 5)
// ---------------------------------------------------------------------------
template <typename T> struct Chunk8;
template <> struct Chunk8<float> {
    __device__ static __forceinline__ float acc(const float *p, float s)
    {
        const float4 a = __ldg(reinterpret_cast<const float4 *>(p));
        const float4 b = __ldg(reinterpret_cast<const float4 *>(p) + 1);
        s = __fmaf_rn(a.x, a.x, s); s = __fmaf_rn(a.y, a.y, s);
        s = __fmaf_rn(a.z, a.z, s); s = __fmaf_rn(a.w, a.w, s);
        s = __fmaf_rn(b.x, b.x, s); s = __fmaf_rn(b.y, b.y, s);
        s = __fmaf_rn(b.z, b.z, s); s = __fmaf_rn(b.w, b.w, s);
        return s;
    }
};
template <> struct Chunk8<uint16_t> {
    __device__ static __forceinline__ float acc(const uint16_t *p, float s)
    {
        const uint4 w = __ldg(reinterpret_cast<const uint4 *>(p));
        const uint32_t v[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            const float lo = __uint_as_float(v[k] << 16);
            const float hi = __uint_as_float(v[k] & 0xffff0000u);
            s = __fmaf_rn(lo, lo, s);
            s = __fmaf_rn(hi, hi, s);
        }
        return s;
    }
};

template <typename T>
__global__ void __launch_bounds__(256)
k_energy(const T *__restrict__ z, int G, int mn, int C, int lpr, const uint32_t *__restrict__ need,
         float *__restrict__ e)
{
    pdl_wait();
    const int nchunk = C >> 3;
    const int rpw = 32 / lpr;
    const int lane = threadIdx.x & 31;
    const int sub = lane / lpr, l = lane % lpr;
    const int nwords = (mn + 31) >> 5;
    const long total = (long)G * mn;
    const long wid = ((long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const long nwarps = ((long)gridDim.x * blockDim.x) >> 5;
    for (long base = wid * rpw; base < total; base += nwarps * rpw) {
        const long row = base + sub;
        bool needed = false;
        if (row < total) {
            const int g = (int)(row / mn);
            const int i = (int)(row - (long)g * mn);
            needed = (need[(size_t)g * nwords + (i >> 5)] >> (i & 31)) & 1u;
        }
        float s = 0.0f;
        if (needed) {
            const T *zr = z + row * (long)C;
            for (int ch = l; ch < nchunk; ch += 32) s = Chunk8<T>::acc(zr + ch * 8, s);
        }
        for (int w = lpr >> 1; w >= 1; w >>= 1) s = s + __shfl_xor_sync(0xffffffffu, s, w);
        if (needed && l == 0) e[row] = s;
    }
}

// ---------------------------------------------------------------------------
// k_select: top-k by (energy desc, index asc) inside the prior (Eq. 5)
// ---------------------------------------------------------------------------
// Exclusive block scan of one 32-bit value per thread (values sum < 2^32).
__device__ __forceinline__ uint32_t block_excl_scan(uint32_t v, uint32_t &total)
{
    __shared__ uint32_t s_warp[32];
    __shared__ uint32_t s_total;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    uint32_t incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const uint32_t t = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += t;
    }
    if (lane == 31) s_warp[warp] = incl;
    __syncthreads();
    const int nw = blockDim.x >> 5;
    if (warp == 0) {
        uint32_t x = lane < nw ? s_warp[lane] : 0u;
        uint32_t xi = x;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const uint32_t t = __shfl_up_sync(0xffffffffu, xi, o);
            if (lane >= o) xi += t;
        }
        if (lane < nw) s_warp[lane] = xi - x;    // exclusive warp offsets
        if (lane == nw - 1) s_total = xi;
    }
    __syncthreads();
    const uint32_t off = s_warp[warp] + (incl - v);
    total = s_total;
    __syncthreads();
    return off;
}

__global__ void __launch_bounds__(1024)
k_select(const uint8_t *__restrict__ prior, const uint32_t *__restrict__ need,
         const float *__restrict__ e, const int32_t *__restrict__ unit_group, int G, int mn,
         int union_mode, int k, int32_t *__restrict__ idx, int32_t *__restrict__ count)
{
    pdl_wait();
    extern __shared__ __align__(16) uint32_t skey[];
    __shared__ uint32_t hist[256];
    __shared__ uint32_t s_bin, s_rem;
    const int u = blockIdx.x;
    const int g = unit_group[u];
    if (g < 0 || g >= G) {                     // k_prior latched the error
        if (threadIdx.x == 0) count[u] = 0;
        return;
    }
    const int nwords = (mn + 31) >> 5;
    const uint8_t *Pu = prior + (size_t)u * mn;
    const uint32_t *Ng = need + (size_t)g * nwords;
    const float *eg = e + (size_t)g * mn;
    // every load of the loop is independent (the energy is read whether or
    // not the cell is in the prior: the buffer holds mn values per group), so
    // the unrolled iterations share one round trip
    uint32_t np_local = 0;
#pragma unroll 4
    for (int i = threadIdx.x; i < mn; i += blockDim.x) {
        const uint32_t ebits = __float_as_uint(eg[i]);
        const bool inP = union_mode ? ((Ng[i >> 5] >> (i & 31)) & 1u) : (Pu[i] != 0);
        skey[i] = inP ? ebits : KEY_NONE;
        np_local += inP ? 1u : 0u;
    }
    uint32_t nP;
    block_excl_scan(np_local, nP);          // also syncs skey

    const bool keep_all = nP <= (uint32_t)k;
    uint32_t T = 0, rem = 0;
    if (!keep_all) {
        // radix select of the k-th largest key, 8 bits per pass, MSB first
        uint32_t prefix = 0, pmask = 0, want = (uint32_t)k;
        for (int pass = 0; pass < 4; ++pass) {
            const int shift = 24 - 8 * pass;
            for (int b = threadIdx.x; b < 256; b += blockDim.x) hist[b] = 0;
            __syncthreads();
            for (int i = threadIdx.x; i < mn; i += blockDim.x) {
                const uint32_t key = skey[i];
                if (key != KEY_NONE && (key & pmask) == prefix) atomicAdd(&hist[(key >> shift) & 255u], 1u);
            }
            __syncthreads();
            if (threadIdx.x < 32) {
                const int lane = threadIdx.x;
                uint32_t tot = 0;
#pragma unroll
                for (int b = 0; b < 8; ++b) tot += hist[lane * 8 + b];
                // inclusive suffix sum over lanes (lane 31 holds the top bins)
                uint32_t suf = tot;
#pragma unroll
                for (int o = 1; o < 32; o <<= 1) {
                    const uint32_t t = __shfl_down_sync(0xffffffffu, suf, o);
                    if (lane + o < 32) suf += t;
                }
                const uint32_t above = suf - tot;          // keys in bins above this lane
                if (above < want && want <= suf) {
                    uint32_t cum = above;
                    for (int b = lane * 8 + 7; b >= lane * 8; --b) {
                        const uint32_t h = hist[b];
                        if (cum + h >= want) {
                            s_bin = (uint32_t)b;
                            s_rem = want - cum;
                            break;
                        }
                        cum += h;
                    }
                }
            }
            __syncthreads();
            prefix |= s_bin << shift;
            pmask |= 255u << shift;
            want = s_rem;
            __syncthreads();
        }
        T = prefix;
        rem = want;   // how many keys equal to T are kept (lowest indices first)
    }

    // stream compaction in ascending cell order: position = (# greater keys
    // before) + min(# equal keys before, rem)
    uint32_t base_gt = 0, base_eq = 0;
    int32_t *out = idx + (size_t)u * k;
    for (int i0 = 0; i0 < mn; i0 += blockDim.x) {
        const int i = i0 + threadIdx.x;
        const uint32_t key = i < mn ? skey[i] : KEY_NONE;
        const bool inP = key != KEY_NONE;
        const bool gt = keep_all ? inP : (inP && key > T);
        const bool eq = keep_all ? false : (inP && key == T);
        const uint32_t bg = __ballot_sync(0xffffffffu, gt);
        const uint32_t be = __ballot_sync(0xffffffffu, eq);
        const uint32_t lm = lanemask_lt();
        // pack (gt count << 16 | eq count) of this warp for one block scan
        const uint32_t mine = (threadIdx.x & 31) == 0 ? ((uint32_t)__popc(bg) << 16) | (uint32_t)__popc(be) : 0u;
        uint32_t tot;
        const uint32_t woff = block_excl_scan(mine, tot);   // lane 0 of each warp holds its warp offset
        const uint32_t wbase = __shfl_sync(0xffffffffu, woff, 0);
        const uint32_t gt_before = base_gt + (wbase >> 16) + (uint32_t)__popc(bg & lm);
        const uint32_t eq_before = base_eq + (wbase & 0xffffu) + (uint32_t)__popc(be & lm);
        const bool keep = gt || (eq && eq_before < rem);
        const uint32_t pos = gt_before + min(eq_before, rem);
        if (keep && pos < (uint32_t)k) out[pos] = i;
        base_gt += tot >> 16;
        base_eq += tot & 0xffffu;
    }
    if (threadIdx.x == 0) count[u] = (int32_t)min(base_gt + min(base_eq, rem), keep_all ? nP : (uint32_t)k);
}

// ---------------------------------------------------------------------------
// k_write_keepset: Eq. 8 with the 5% / 95% fall-through of Sec. 3.2
// ---------------------------------------------------------------------------
__global__ void __launch_bounds__(1024)
k_write_keepset(const uint8_t *__restrict__ seeds, const int32_t *__restrict__ unit_group, int U,
                int G_unused, int m, int n, int D_w, double fall_lo, double fall_hi,
                int fall_through, int union_mode, uint8_t *__restrict__ kw, int32_t *status)
{
    pdl_wait();
    extern __shared__ __align__(16) uint8_t smem[];
    const int mn = m * n;
    const int u = blockIdx.x;
    uint8_t *sS = smem;
    uint8_t *sT = smem + ((mn + 15) & ~15);
    const int g = unit_group[u];
    for (int i = threadIdx.x; i < mn; i += blockDim.x) sS[i] = seeds[(size_t)u * mn + i] != 0;
    __syncthreads();
    if (union_mode) {
        for (int v = 0; v < U; ++v) {
            if (v == u || unit_group[v] != g) continue;
            for (int i = threadIdx.x; i < mn; i += blockDim.x) sS[i] |= seeds[(size_t)v * mn + i] != 0;
        }
        __syncthreads();
    }
    uint32_t area_local = 0;
    for (int i = threadIdx.x; i < mn; i += blockDim.x) area_local += sS[i];
    uint32_t area;
    block_excl_scan(area_local, area);
    const double frac = (double)area / (double)mn;
    uint8_t *out = kw + (size_t)u * mn;
    if (fall_through && (frac > fall_hi || frac < fall_lo)) {
        for (int i = threadIdx.x; i < mn; i += blockDim.x) out[i] = 1;
        return;
    }
    row_pass(sS, sT, m, n, D_w);
    __syncthreads();
    for (int i = threadIdx.x; i < mn; i += blockDim.x) out[i] = col_value(sT, m, n, D_w, i);
}

inline int next_pow2(int x)
{
    int p = 1;
    while (p < x) p <<= 1;
    return p;
}

struct SelectWs {
    size_t need, prior, energy, total;
};

SelectWs select_ws(int G, int U, int m, int n)
{
    const size_t mn = (size_t)m * n;
    const size_t nwords = (mn + 31) / 32;
    SelectWs w;
    w.need = 0;
    w.prior = align_up(w.need + (size_t)G * nwords * 4, 256);
    w.energy = align_up(w.prior + (size_t)U * mn, 256);
    w.total = align_up(w.energy + (size_t)G * mn * 4, 256);
    return w;
}

}  // namespace

// ---------------------------------------------------------------------------
// host entry points
// ---------------------------------------------------------------------------
extern "C" size_t rs3_select_workspace_bytes(int G, int U, int m, int n)
{
    if (G < 1 || U < 1 || m < 1 || n < 1) return 0;
    return select_ws(G, U, m, n).total;
}

extern "C" rs3_status rs3_select_queries(const void *z, rs3_dtype dtype, int G, int m, int n, int C,
                                         const uint8_t *prev_masks, const int32_t *unit_group,
                                         int U, rs3_track *track, const rs3_params *p,
                                         int32_t *idx, int32_t *count, void *workspace,
                                         size_t workspace_bytes, int32_t *status,
                                         rs3_stream_t stream)
{
    if (!z || !prev_masks || !unit_group || !track || !p || !idx || !count || !workspace || !status)
        return RS3_EINVAL;
    if (dtype != RS3_F32 && dtype != RS3_BF16) return RS3_EINVAL;
    if (G < 1 || U < 1 || m < 1 || n < 1 || C < 8 || (C % 8) != 0) return RS3_EINVAL;
    if ((long)m * n > RS3_MAX_MN || C > 4096) return RS3_EUNSUPPORTED;
    if (!(p->rho >= 0.0 && p->rho <= 1.0) || p->r_s < 0 || p->c < 0) return RS3_EINVAL;
    if (!rs3_aligned16(z) || !rs3_aligned16(workspace)) return RS3_EINVAL;
    const SelectWs ws = select_ws(G, U, m, n);
    if (workspace_bytes < ws.total) return RS3_ECAPACITY;
    const int mn = m * n;
    const int64_t k = rs3_kmax(p->rho, mn);
    if (k < 0) return RS3_EINVAL;

    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    uint8_t *wsb = static_cast<uint8_t *>(workspace);
    uint32_t *need = reinterpret_cast<uint32_t *>(wsb + ws.need);
    uint8_t *prior = wsb + ws.prior;
    float *energy = reinterpret_cast<float *>(wsb + ws.energy);
    const int nwords = (mn + 31) / 32;

    if (cudaMemsetAsync(need, 0, (size_t)G * nwords * 4, st) != cudaSuccess) return RS3_ECUDA;
    const size_t smem_prior = 2 * (size_t)((mn + 15) & ~15);
    launch_pdl(k_prior, dim3(U), dim3(1024), smem_prior, st, prev_masks, m, n, unit_group, G, track, p->r_s, p->c,
                                         p->bbox_mode, prior, need, status);
    if (cudaGetLastError() != cudaSuccess) return RS3_ECUDA;

    const int nchunk = C / 8;
    const int lpr = nchunk >= 32 ? 32 : next_pow2(nchunk);
    const int rpw = 32 / lpr;
    const long rows = (long)G * mn;
    const long warps_needed = (rows + rpw - 1) / rpw;
    long blocks = (warps_needed + 7) / 8;
    const long cap = (long)rs3_sm_count() * 8;
    if (blocks > cap) blocks = cap;
    if (blocks < 1) blocks = 1;
    if (dtype == RS3_BF16)
        launch_pdl(k_energy<uint16_t>, dim3((unsigned)blocks), dim3(256), 0, st, static_cast<const uint16_t *>(z), G, mn, C,
                                                           lpr, need, energy);
    else
        launch_pdl(k_energy<float>, dim3((unsigned)blocks), dim3(256), 0, st, static_cast<const float *>(z), G, mn, C, lpr,
                                                        need, energy);
    if (cudaGetLastError() != cudaSuccess) return RS3_ECUDA;

    const size_t smem_sel = (size_t)mn * 4;
    if (rs3_kernel_smem((const void *)k_select, smem_sel) != RS3_OK) return RS3_ECUDA;
    launch_pdl(k_select, dim3(U), dim3(1024), smem_sel, st, prior, need, energy, unit_group, G, mn, p->union_mode,
                                        (int)k, idx, count);
    if (cudaGetLastError() != cudaSuccess) return RS3_ECUDA;
    return RS3_OK;
}

extern "C" rs3_status rs3_write_keepset(const uint8_t *seed_masks, const int32_t *unit_group, int U,
                                        int m, int n, const rs3_params *p, uint8_t *kw_out,
                                        int32_t *status, rs3_stream_t stream)
{
    if (!seed_masks || !unit_group || !p || !kw_out || !status) return RS3_EINVAL;
    if (U < 1 || m < 1 || n < 1 || p->D_w < 0) return RS3_EINVAL;
    if ((long)m * n > RS3_MAX_MN) return RS3_EUNSUPPORTED;
    const int mn = m * n;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t smem = 2 * (size_t)((mn + 15) & ~15);
    launch_pdl(k_write_keepset, dim3(U), dim3(1024), smem, st, seed_masks, unit_group, U, 0, m, n, p->D_w, p->fall_lo,
                                           p->fall_hi, p->fall_through, p->union_mode, kw_out,
                                           status);
    if (cudaGetLastError() != cudaSuccess) return RS3_ECUDA;
    return RS3_OK;
}
