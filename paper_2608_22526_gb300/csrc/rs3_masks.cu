// rs3_masks.cu -- the decoder side and the pixel-space front end of RS3-Prune.
//
//   rs3_close_argmax     Sec. 3.3: per-object closure of the decoder's binary
//                        masks with a (2R+1)^2 square (9 x 9 in the paper),
//                        then the per-pixel argmax over a stream's objects
//                        (the palette mask); optionally down_s of each closed
//                        mask onto the token grid (Sec. 3.1, Eq. 2's input)
//   rs3_seed_from_masks  Sec. 3.1, Eq. 1: the seed box of each object's pixel
//                        mask projected onto the grid (the tracker state of
//                        Eq. 4), with down_s of the mask and the filled box
//
// Closure.  A CTA of 256 threads owns a tile of BR rows x 256 columns of one
// stream's decoder output; thread t owns column t.  The CTAs of a thread-block
// cluster (up to 8, along the stream's objects) share one tile: rank r closes
// objects r, r + KC, ... of the stream.  For each of its objects a CTA
// thresholds the logits (logit > 0) into bit masks -- a warp ballot over 32
// adjacent columns is one 32-bit word -- for the tile plus a 2R-row halo above
// and below and one word left and right (all of an object's loads issued
// before its first ballot), then runs the four separable passes on words in
// shared memory: horizontal dilation (OR of funnel-shifted words), vertical
// dilation (OR over rows), horizontal and vertical erosion (AND).  The object
// is a set of the unbounded plane with nothing set outside the image: pixels
// outside are zero words, and the dilation is evaluated there too, so the
// erosion never treats the border as set or unset by convention.  With R <= 8
// every bit the tile's result depends on lies within 2R = 16 pixels of the
// tile, i.e. in the loaded window.  Each CTA keeps, per pixel, the largest
// logit among its objects whose closed mask holds the pixel (in shared memory,
// the column's thread alone touching it; equal logits keep the earlier
// object); after a cluster barrier each rank merges a share of the tile's rows
// from all ranks' shared memory (DSMEM), equal logits going to the object
// listed first, and writes those palette rows.  Each logit is read
// from DRAM once; halo re-reads by neighbouring tiles hit L2.
#include "rs3_internal.cuh"

#include <algorithm>
#include <climits>

namespace {

constexpr int CA_TW = 8;            // words (of 32 pixels) per tile row: 256 columns
constexpr int CA_THREADS = 32 * CA_TW;
constexpr int CA_RMAX = 8;

// bits of the row word x (with its left / right neighbour words) ORed over
// horizontal shifts -R..R: bit k of the result covers pixels 32w + k - R ..
// 32w + k + R.  __funnelshift_r(x, nx, d) brings pixel 32w + k + d to bit k,
// __funnelshift_l(pv, x, d) brings pixel 32w + k - d.
__device__ __forceinline__ uint32_t dil_h(uint32_t pv, uint32_t x, uint32_t nx, int R)
{
    uint32_t r = x;
#pragma unroll
    for (int d = 1; d <= R; ++d) r |= __funnelshift_r(x, nx, d) | __funnelshift_l(pv, x, d);
    return r;
}

__device__ __forceinline__ uint32_t ero_h(uint32_t pv, uint32_t x, uint32_t nx, int R)
{
    uint32_t r = x;
#pragma unroll
    for (int d = 1; d <= R; ++d) r &= __funnelshift_r(x, nx, d) & __funnelshift_l(pv, x, d);
    return r;
}

__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// every thread of every CTA of the cluster arrives, then waits (the release /
// acquire pair orders shared-memory writes before the barrier with reads of
// them through DSMEM after it)
__device__ __forceinline__ void cluster_barrier()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\t"
                 "barrier.cluster.wait.acquire.aligned;" ::: "memory");
}

__device__ __forceinline__ uint32_t dsmem_addr(const void *p, uint32_t rank)
{
    const uint32_t a = (uint32_t)__cvta_generic_to_shared(p);
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(a), "r"(rank));
    return r;
}

__device__ __forceinline__ float dsmem_ld_f32(uint32_t a)
{
    float v;
    asm volatile("ld.shared::cluster.f32 %0, [%1];" : "=f"(v) : "r"(a) : "memory");
    return v;
}

__device__ __forceinline__ uint32_t dsmem_ld_u8(uint32_t a)
{
    uint32_t v;
    asm volatile("ld.shared::cluster.u8 %0, [%1];" : "=r"(v) : "r"(a) : "memory");
    return v;
}

constexpr int CA_HB = 16;           // halo rows per load batch
constexpr int CA_SB = 8;            // side-word ballots per warp per load batch

// halo rows j0 .. j0 + CA_HB - 1 of the 4R (the first 2R above the tile, the
// rest below it), column x; rows outside the image read as 0
__device__ __forceinline__ void load_halo_rows(float (&hv)[CA_HB], const float *L, int j0, int R, int BR, int r0,
                                               int h, int w, int x, bool colin)
{
#pragma unroll
    for (int q = 0; q < CA_HB; ++q) {
        const int j = j0 + q;
        const int lr = j < 2 * R ? j : BR + j;           // window row
        const int row = r0 - 2 * R + lr;
        hv[q] = (j < 4 * R && colin && row >= 0 && row < h) ? __ldg(L + (size_t)row * w + x) : 0.f;
    }
}

template <int NW>
__device__ __forceinline__ void store_halo_rows(uint32_t (*sA)[NW], const float (&hv)[CA_HB], int j0, int R,
                                                int BR, int lane, int warp)
{
#pragma unroll
    for (int q = 0; q < CA_HB; ++q) {
        const int j = j0 + q;
        const uint32_t b = __ballot_sync(0xffffffffu, hv[q] > 0.f);
        if (lane == 0 && j < 4 * R) sA[j < 2 * R ? j : BR + j][1 + warp] = b;
    }
}

// side words: pair p = warp + CA_TW * i (i = i0 .. i0 + CA_SB - 1) is window
// row p / 2, the word left of the tile (p even) or right of it (p odd)
__device__ __forceinline__ void load_side_words(float (&hw)[CA_SB], const float *L, int i0, int nwin, int r0,
                                                int R, int h, int w, int w0, int WW, int warp, int lane)
{
#pragma unroll
    for (int q = 0; q < CA_SB; ++q) {
        const int p = warp + CA_TW * (i0 + q);
        const int row = r0 - 2 * R + (p >> 1);
        const int gw = (p & 1) ? w0 + CA_TW : w0 - 1;
        hw[q] = (p < 2 * nwin && row >= 0 && row < h && gw >= 0 && gw < WW)
                    ? __ldg(L + (size_t)row * w + 32 * gw + lane)
                    : 0.f;
    }
}

template <int NW>
__device__ __forceinline__ void store_side_words(uint32_t (*sA)[NW], const float (&hw)[CA_SB], int i0, int nwin,
                                                 int warp, int lane)
{
#pragma unroll
    for (int q = 0; q < CA_SB; ++q) {
        const int p = warp + CA_TW * (i0 + q);
        const uint32_t b = __ballot_sync(0xffffffffu, hw[q] > 0.f);
        if (lane == 0 && p < 2 * nwin) sA[p >> 1][(p & 1) ? CA_TW + 1 : 0] = b;
    }
}

// RC > 0 fixes the radius at compile time (the paper's 9 x 9 element is
// RC = 4), so the shift and row loops unroll; RC = 0 takes it from R_rt.
template <int BR, int RC>
__global__ void __launch_bounds__(CA_THREADS, 2)
k_close_argmax(const float *__restrict__ logits, const int32_t *__restrict__ gstart, int U, int h,
               int w, int R_rt, int s, int KC, uint8_t *__restrict__ palette, uint8_t *__restrict__ closed,
               uint8_t *__restrict__ grid, int32_t *status)
{
    const int R = RC > 0 ? RC : R_rt;
    constexpr int NR = BR + 4 * CA_RMAX;    // window rows [r0 - 2R, r0 + BR + 2R)
    constexpr int NW = CA_TW + 2;           // window words [w0 - 1, w0 + TW + 1)
    __shared__ uint32_t sA[NR][NW];         // thresholded logits
    __shared__ uint32_t sH[NR][NW];         // horizontal dilation
    __shared__ uint32_t sD[NR][NW];         // dilation
    __shared__ uint32_t sE[NR][CA_TW];      // dilation, then horizontal erosion
    __shared__ uint32_t sC[BR][CA_TW];      // closure of the tile's rows
    __shared__ float sV[BR][CA_THREADS];    // the current object's logits of the tile
    __shared__ float sBV[BR][CA_THREADS];   // this CTA's best logit per pixel
    __shared__ uint8_t sBL[BR][CA_THREADS]; // ... and its label (0 = none)
    // (thread t alone touches column t of sV, sBV and sBL until the merge)
    pdl_wait();
    const uint32_t rank = KC > 1 ? cluster_rank() : 0u;
    const int g = blockIdx.z / KC;
    const int r0 = blockIdx.y * BR, w0 = blockIdx.x * CA_TW;
    const int WW = w >> 5;
    const int t = threadIdx.x, warp = t >> 5, lane = t & 31;
    const int brv = min(BR, h - r0);                 // tile rows inside the image
    const bool colin = w0 + warp < WW;               // warp-uniform: the warp's word is inside
    const int x = 32 * w0 + t;                       // this thread's column
    const int u0 = gstart[g], u1 = gstart[g + 1];
    // the same values reach every CTA of the cluster, so all of them leave
    // here together, before any cluster barrier
    if (u0 < 0 || u1 < u0 || u1 > U || u1 - u0 > 255) {
        if (t == 0 && rank == 0) latch_status(status, RS3_EINVAL);
        return;
    }
    const int nwin = BR + 4 * R;                     // window rows in use
    const int m = h / s, n = w / s;
    // down_s without divisions in the pixel loop: the tile rows that are grid
    // rows (a bit per row) and the first one's grid row; this column's grid
    // column, or -1
    const int gi0 = (r0 + s - 1) / s;
    uint32_t growmask = 0u;
    for (int i = gi0; i * s < r0 + brv; ++i) growmask |= 1u << (i * s - r0);
    const int gx = (x % s == 0) ? x / s : -1;
#pragma unroll
    for (int k = 0; k < BR; ++k) {
        sBV[k][t] = 0.f;
        sBL[k][t] = 0;
    }
    for (int u = u0 + (int)rank; u < u1; u += KC) {
        const float *L = logits + (size_t)u * h * w;
        // 1. the object's loads: the tile's rows (thread t reads column x),
        //    the 4R halo rows, and the words left and right of the tile on
        //    every window row (one ballot per (row, side); warp j takes pairs
        //    j, j + 8, ...).  The first batch -- all of it for R <= 4 -- is
        //    issued before its first ballot; larger radii take more batches.
        float v[BR], hv[CA_HB], hw[CA_SB];
#pragma unroll
        for (int k = 0; k < BR; ++k) v[k] = (k < brv && colin) ? __ldg(L + (size_t)(r0 + k) * w + x) : 0.f;
        load_halo_rows(hv, L, 0, R, BR, r0, h, w, x, colin);
        load_side_words(hw, L, 0, nwin, r0, R, h, w, w0, WW, warp, lane);
        // the ballot of warp j over row k is word w0 + j of that row
#pragma unroll
        for (int k = 0; k < BR; ++k) {
            const uint32_t b = __ballot_sync(0xffffffffu, v[k] > 0.f);
            if (lane == 0) sA[2 * R + k][1 + warp] = b;
            sV[k][t] = v[k];
        }
        store_halo_rows<NW>(sA, hv, 0, R, BR, lane, warp);
        store_side_words<NW>(sA, hw, 0, nwin, warp, lane);
        for (int j0 = CA_HB; j0 < 4 * R; j0 += CA_HB) {
            load_halo_rows(hv, L, j0, R, BR, r0, h, w, x, colin);
            store_halo_rows<NW>(sA, hv, j0, R, BR, lane, warp);
        }
        for (int i0 = CA_SB; warp + CA_TW * i0 < 2 * nwin; i0 += CA_SB) {
            load_side_words(hw, L, i0, nwin, r0, R, h, w, w0, WW, warp, lane);
            store_side_words<NW>(sA, hw, i0, nwin, warp, lane);
        }
        __syncthreads();
        // 2. horizontal dilation on every window word (the outermost words'
        //    missing neighbours are read as zero: only their bits next to the
        //    tile are used below, and those do not depend on them)
        for (int p = t; p < nwin * NW; p += CA_THREADS) {
            const int lr = p / NW, lw = p - lr * NW;
            const uint32_t pv = lw > 0 ? sA[lr][lw - 1] : 0u;
            const uint32_t nx = lw < NW - 1 ? sA[lr][lw + 1] : 0u;
            sH[lr][lw] = dil_h(pv, sA[lr][lw], nx, R);
        }
        __syncthreads();
        // 3. vertical dilation, window rows [R, BR + 3R)
        for (int p = t; p < (BR + 2 * R) * NW; p += CA_THREADS) {
            const int lr = R + p / NW, lw = p % NW;
            uint32_t r = 0u;
#pragma unroll
            for (int d = -R; d <= R; ++d) r |= sH[lr + d][lw];
            sD[lr][lw] = r;
        }
        __syncthreads();
        // 4. horizontal erosion of the tile's words, window rows [R, BR + 3R)
        for (int p = t; p < (BR + 2 * R) * CA_TW; p += CA_THREADS) {
            const int lr = R + p / CA_TW, k = p % CA_TW;
            sE[lr][k] = ero_h(sD[lr][k], sD[lr][k + 1], sD[lr][k + 2], R);
        }
        __syncthreads();
        // 5. vertical erosion: the closure of the tile's rows
        for (int p = t; p < BR * CA_TW; p += CA_THREADS) {
            const int k = p / CA_TW, wd = p % CA_TW;
            uint32_t r = 0xffffffffu;
#pragma unroll
            for (int d = -R; d <= R; ++d) r &= sE[2 * R + k + d][wd];
            sC[k][wd] = r;
        }
        __syncthreads();
        // 6. argmax update, closed mask and its down_s onto the grid
        const uint32_t label = (uint32_t)(u - u0 + 1);
#pragma unroll
        for (int k = 0; k < BR; ++k) {
            if (k < brv && colin) {
                const uint32_t bit = (sC[k][warp] >> lane) & 1u;
                const float vk = sV[k][t];
                if (bit && (sBL[k][t] == 0 || vk > sBV[k][t])) {
                    sBV[k][t] = vk;
                    sBL[k][t] = (uint8_t)label;
                }
                if (closed) closed[((size_t)u * h + r0 + k) * w + x] = (uint8_t)bit;
                if (grid && gx >= 0 && ((growmask >> k) & 1u))
                    grid[((size_t)u * m + gi0 + __popc(growmask & ((1u << k) - 1u))) * n + gx] = (uint8_t)bit;
            }
        }
    }
    if (KC > 1) {
        // 7. the ranks' bests are in their shared memory; rank r merges tile rows
        //    r, r + KC, ...: the larger logit, the lower label on equal logits
        //    (each rank's best already holds its lowest label among equal
        //    logits), and writes those palette rows
        cluster_barrier();
        for (int k = (int)rank; k < BR; k += KC) {
            float v2[8];
            uint32_t l2[8];
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                if (q < KC) {
                    v2[q] = dsmem_ld_f32(dsmem_addr(&sBV[k][t], (uint32_t)q));
                    l2[q] = dsmem_ld_u8(dsmem_addr(&sBL[k][t], (uint32_t)q));
                }
            }
            float b = 0.f;
            uint32_t l = 0u;
#pragma unroll
            for (int q = 0; q < 8; ++q) {
                if (q < KC && l2[q] != 0u && (l == 0u || v2[q] > b || (v2[q] == b && l2[q] < l))) {
                    b = v2[q];
                    l = l2[q];
                }
            }
            if (palette && k < brv && colin) palette[((size_t)g * h + r0 + k) * w + x] = (uint8_t)l;
        }
        cluster_barrier();       // no CTA leaves while another reads its shared memory
    } else if (palette) {
#pragma unroll
        for (int k = 0; k < BR; ++k)
            if (k < brv && colin) palette[((size_t)g * h + r0 + k) * w + x] = sBL[k][t];
    }
}

// ---------------------------------------------------------------------------
// Seed box and down_s of pixel masks
// ---------------------------------------------------------------------------

__global__ void k_seed_init(rs3_track *track, int U)
{
    pdl_wait();
    const int u = blockIdx.x * blockDim.x + threadIdx.x;
    if (u < U) track[u] = rs3_track{INT_MAX, INT_MAX, -1, -1, 0, 0};
}

// one CTA per (band of rows, unit): the band's set pixels' extreme rows and
// columns, merged into the unit's track with atomics (16-byte loads; byte j
// of a chunk is column 16c + j)
__global__ void __launch_bounds__(256) k_seed_scan(const uint8_t *__restrict__ masks, int h, int w, int rows,
                                                   rs3_track *track)
{
    pdl_wait();
    const int u = blockIdx.y;
    const int r0 = blockIdx.x * rows;
    const int nr = min(rows, h - r0);
    const int cpr = w >> 4;                                   // chunks per row
    const uint4 *base = reinterpret_cast<const uint4 *>(masks + ((size_t)u * h + r0) * w);
    int y0 = INT_MAX, x0 = INT_MAX, y1 = -1, x1 = -1;
    for (int c = threadIdx.x; c < nr * cpr; c += blockDim.x) {
        const uint4 q = __ldg(base + c);
        if ((q.x | q.y | q.z | q.w) == 0u) continue;
        const int row = r0 + c / cpr, xb = 16 * (c % cpr);
        const uint32_t wd[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            const uint32_t nz = __vcmpne4(wd[j], 0u);          // 0xff in every non-zero byte
            if (nz) {
                x0 = min(x0, xb + 4 * j + ((__ffs(nz) - 1) >> 3));
                x1 = max(x1, xb + 4 * j + ((31 - __clz(nz)) >> 3));
            }
        }
        y0 = min(y0, row);
        y1 = max(y1, row);
    }
    y0 = __reduce_min_sync(0xffffffffu, y0);
    x0 = __reduce_min_sync(0xffffffffu, x0);
    y1 = __reduce_max_sync(0xffffffffu, y1);
    x1 = __reduce_max_sync(0xffffffffu, x1);
    if ((threadIdx.x & 31) == 0 && y1 >= 0) {
        atomicMin(&track[u].y0, y0);
        atomicMin(&track[u].x0, x0);
        atomicMax(&track[u].y1, y1);
        atomicMax(&track[u].x1, x1);
    }
}

// one CTA per unit: the pixel box divided by s (rounding down) becomes the
// tracker state; down_s of the mask and the filled grid box are written
__global__ void __launch_bounds__(256) k_seed_finish(const uint8_t *__restrict__ masks, int h, int w, int s,
                                                     rs3_track *track, uint8_t *grid, uint8_t *box)
{
    pdl_wait();
    const int u = blockIdx.x;
    __shared__ rs3_track sb;
    if (threadIdx.x == 0) {
        rs3_track tr = track[u];
        if (tr.y1 >= 0)
            tr = rs3_track{tr.y0 / s, tr.x0 / s, tr.y1 / s, tr.x1 / s, 1, 0};
        else
            tr = rs3_track{0, 0, 0, 0, 0, 0};
        track[u] = tr;
        sb = tr;
    }
    __syncthreads();
    const int m = h / s, n = w / s;
    for (int c = threadIdx.x; c < m * n; c += blockDim.x) {
        const int i = c / n, j = c - i * n;
        if (grid) grid[(size_t)u * m * n + c] = masks[((size_t)u * h + (size_t)i * s) * w + (size_t)j * s] != 0;
        if (box)
            box[(size_t)u * m * n + c] = sb.valid && i >= sb.y0 && i <= sb.y1 && j >= sb.x0 && j <= sb.x1;
    }
}

}  // namespace

template <int BR, int RC>
static cudaError_t launch_close(int tiles_x, int h, int G, int KC, cudaStream_t st, const float *logits,
                                const int32_t *gstart, int U, int w, int R, int s, uint8_t *palette,
                                uint8_t *closed, uint8_t *grid, int32_t *status)
{
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(tiles_x, (h + BR - 1) / BR, G * KC);
    cfg.blockDim = dim3(CA_THREADS);
    cfg.dynamicSmemBytes = 0;
    cfg.stream = st;
    cudaLaunchAttribute attr[2];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    attr[1].id = cudaLaunchAttributeClusterDimension;
    attr[1].val.clusterDim.x = 1;
    attr[1].val.clusterDim.y = 1;
    attr[1].val.clusterDim.z = KC;
    cfg.attrs = attr;
    cfg.numAttrs = 2;
    return cudaLaunchKernelEx(&cfg, k_close_argmax<BR, RC>, logits, gstart, U, h, w, R, s, KC, palette, closed,
                              grid, status);
}

extern "C" rs3_status rs3_close_argmax(const float *logits, const int32_t *group_start, int G, int U, int h,
                                       int w, int radius, int s, uint8_t *palette, uint8_t *closed,
                                       uint8_t *grid_masks, int32_t *status, rs3_stream_t stream)
{
    if (!logits || !group_start || !status) return RS3_EINVAL;
    if (G < 1 || U < 0 || h < 1 || w < 32 || radius < 0 || s < 1) return RS3_EINVAL;
    if (w % 32 != 0 || radius > CA_RMAX) return RS3_EUNSUPPORTED;
    if (grid_masks && (h % s != 0 || w % s != 0)) return RS3_EINVAL;
    if ((long long)h * w > (1ll << 31)) return RS3_EUNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    // cluster size: the mean number of objects per stream, at most 8 (the
    // portable cluster size); ranks past a stream's object count idle
    const int KC = std::min(8, std::max(1, (U + G - 1) / G));
    if ((long long)G * KC > 65535) return RS3_EUNSUPPORTED;
    const int tiles_x = (w / 32 + CA_TW - 1) / CA_TW;
    // the taller tile (fewer halo rows per tile row) when it still gives two
    // CTAs per SM
    const long long ctas16 = (long long)tiles_x * ((h + 15) / 16) * G * KC;
    const bool tall = ctas16 >= 2ll * rs3_sm_count();
    cudaError_t e;
    if (radius == 4)        // the paper's 9 x 9 element, unrolled
        e = tall ? launch_close<16, 4>(tiles_x, h, G, KC, st, logits, group_start, U, w, radius, s, palette,
                                       closed, grid_masks, status)
                 : launch_close<8, 4>(tiles_x, h, G, KC, st, logits, group_start, U, w, radius, s, palette,
                                      closed, grid_masks, status);
    else
        e = tall ? launch_close<16, 0>(tiles_x, h, G, KC, st, logits, group_start, U, w, radius, s, palette,
                                       closed, grid_masks, status)
                 : launch_close<8, 0>(tiles_x, h, G, KC, st, logits, group_start, U, w, radius, s, palette,
                                      closed, grid_masks, status);
    return e == cudaSuccess ? RS3_OK : RS3_ECUDA;
}

extern "C" rs3_status rs3_seed_from_masks(const uint8_t *masks, int U, int h, int w, int s, rs3_track *track,
                                          uint8_t *grid_masks, uint8_t *box_masks, rs3_stream_t stream)
{
    if (!masks || !track) return RS3_EINVAL;
    if (U < 1 || h < 1 || w < 16 || s < 1) return RS3_EINVAL;
    if (w % 16 != 0 || !rs3_aligned16(masks)) return RS3_EINVAL;
    if (h % s != 0 || w % s != 0) return RS3_EINVAL;
    if (U > 65535) return RS3_EUNSUPPORTED;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const int rows = w >= 16384 ? 1 : 16384 / w;              // ~1024 chunks of 16 bytes per CTA
    cudaError_t e = launch_pdl(k_seed_init, dim3((U + 255) / 256), dim3(256), 0, st, track, U);
    if (e == cudaSuccess)
        e = launch_pdl(k_seed_scan, dim3((h + rows - 1) / rows, U), dim3(256), 0, st, masks, h, w, rows, track);
    if (e == cudaSuccess)
        e = launch_pdl(k_seed_finish, dim3(U), dim3(256), 0, st, masks, h, w, s, track, grid_masks, box_masks);
    return e == cudaSuccess ? RS3_OK : RS3_ECUDA;
}
