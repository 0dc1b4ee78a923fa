/*
 * rs3_oracle.c -- plain, slow CPU oracle for the RS3-Prune hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline leg may load this library.  It shares no code,
 * header, table or helper with the CUDA library; the product path never calls
 * it.
 *
 * Every routine is the paper's definition written out with explicit loops
 * (fp64 wherever the paper fixes no precision):
 *   bbox / dilate / prior   Sec. 3.1, Eq. 1, Eq. 2, Eq. 4, Algorithm 1
 *   energy + top-k          Sec. 3.1, Eq. 5 (ranking by ||z||^2)
 *   readout                 Sec. 3.1, Eq. 6 (gather, softmax(qK^T/sqrt(C_k))V,
 *                           scatter) and Eq. 7 (RoPE by the gathered index)
 *   commit                  Sec. 3.2, Eq. 8 and Algorithm 1 (sparse write)
 *   write keep-set          Sec. 3.2, Eq. 8 and the 5%/95% fall-through
 *   closure + palette       Sec. 3.3 (9 x 9 closure per object, then argmax)
 *   down_s + seed box       Sec. 3.1 (pixel masks and boxes onto the grid)
 *
 * Readings where the paper is silent or ambiguous:
 *   - dilate_r is a Chebyshev (square) dilation by r cells;
 *   - the streak counter is updated from the mask the selection consumes, and
 *     the fallback radius uses the incremented value (first empty frame -> r_s+1);
 *   - energies are ranked in a canonical fp32 order (see or_energy_canonical);
 *     ties go to the lower grid index; the keep-set is emitted in ascending
 *     grid order; k = floor(rho * mn) (Table 4 lists 819/1228/2048/2867/4096);
 *   - the score scale is 1/sqrt(d) per head; an empty bank reads out zeros;
 *   - a decoder mask is logit > 0; the closure treats the object as a set of
 *     the unbounded plane with nothing set outside the image (so it neither
 *     grows an object out to the border nor erodes one that touches it); the
 *     palette gives each pixel to the object with the largest logit among
 *     those whose closed mask holds it, the lower object on equal logits;
 *   - down_s samples pixel (i*s, j*s) for grid cell (i, j); a pixel box maps
 *     onto the grid by dividing each corner by s, rounding down.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------- */
/* Geometry: bbox(M) (Sec. 3.1) and dilate_r (Eq. 1, Eq. 2, Eq. 4)            */
/* ------------------------------------------------------------------------- */

/* Tight bounding box of the set cells, inclusive (y0, x0, y1, x1).
 * Returns 1 when the mask has a set cell, 0 otherwise (box untouched). */
int or_bbox(const uint8_t *M, int m, int n, int32_t *box)
{
    int found = 0;
    int y0 = 0, x0 = 0, y1 = 0, x1 = 0;
    for (int y = 0; y < m; ++y)
        for (int x = 0; x < n; ++x)
            if (M[(long)y * n + x]) {
                if (!found) {
                    y0 = y1 = y;
                    x0 = x1 = x;
                    found = 1;
                } else {
                    if (y < y0) y0 = y;
                    if (y > y1) y1 = y;
                    if (x < x0) x0 = x;
                    if (x > x1) x1 = x;
                }
            }
    if (found) {
        box[0] = y0; box[1] = x0; box[2] = y1; box[3] = x1;
    }
    return found;
}

/* out(y,x) = 1 iff some set cell (y',x') of M has |y-y'| <= r and |x-x'| <= r.
 * Direct neighbourhood scan (square structuring element of side 2r+1). */
void or_dilate(const uint8_t *M, int m, int n, int r, uint8_t *out)
{
    for (int y = 0; y < m; ++y)
        for (int x = 0; x < n; ++x) {
            int hit = 0;
            for (int yy = y - r; yy <= y + r && !hit; ++yy) {
                if (yy < 0 || yy >= m) continue;
                for (int xx = x - r; xx <= x + r; ++xx) {
                    if (xx < 0 || xx >= n) continue;
                    if (M[(long)yy * n + xx]) { hit = 1; break; }
                }
            }
            out[(long)y * n + x] = (uint8_t)hit;
        }
}

/* Rasterise an inclusive box into a fresh mask. */
static void raster_box(const int32_t *box, int m, int n, uint8_t *out)
{
    memset(out, 0, (size_t)m * n);
    for (int y = box[0]; y <= box[2]; ++y)
        for (int x = box[1]; x <= box[3]; ++x)
            if (y >= 0 && y < m && x >= 0 && x < n) out[(long)y * n + x] = 1;
}

#define OR_STREAK_SAT 0x3fffffff

/* One object's prior for the current frame and its tracker update.
 *   track = {y0, x0, y1, x1, valid, streak}
 * M is the previous frame's mask of this object (grid resolution, so down_s
 * is the identity).  Non-empty M: P = dilate_{r_s}(M) (Eq. 2) -- or
 * dilate_{r_s}(bbox(M)) in bbox mode (Eq. 1) -- and the tracker caches
 * bbox(M) with streak 0.  Empty M: streak += 1, and if a box was ever cached,
 * P = dilate_{r_s + min(streak, c)}(box) (Eq. 4); otherwise P is empty. */
void or_prior_unit(const uint8_t *M, int m, int n, int32_t *track, int r_s, int c,
                   int bbox_mode, uint8_t *P)
{
    long mn = (long)m * n;
    int32_t box[4];
    uint8_t *tmp = (uint8_t *)malloc((size_t)mn);
    if (or_bbox(M, m, n, box)) {
        track[0] = box[0]; track[1] = box[1]; track[2] = box[2]; track[3] = box[3];
        track[4] = 1;
        track[5] = 0;
        if (bbox_mode) {
            raster_box(box, m, n, tmp);
            or_dilate(tmp, m, n, r_s, P);
        } else {
            or_dilate(M, m, n, r_s, P);
        }
    } else {
        if (track[5] < OR_STREAK_SAT) track[5] += 1;
        if (track[4]) {
            int grow = track[5] < c ? track[5] : c;
            raster_box(track, m, n, tmp);
            or_dilate(tmp, m, n, r_s + grow, P);
        } else {
            memset(P, 0, (size_t)mn);
        }
    }
    free(tmp);
}

/* ------------------------------------------------------------------------- */
/* Energy ||z_i||^2 (Sec. 3.1, Eq. 5)                                         */
/* ------------------------------------------------------------------------- */

/* Canonical fp32 energy of each row (the ranking key).  The C channels are cut
 * into 8-channel chunks; partial sum s[l] (l = 0..31) takes the chunks
 * l, l+32, l+64, ... in that order, channels ascending inside a chunk, each
 * step s[l] = fmaf(z, z, s[l]).  The 32 partials are then added pairwise:
 * s[l] += s[l+w] for w = 16, 8, 4, 2, 1; the energy is s[0].  Requires
 * C % 8 == 0. */
void or_energy_canonical(const float *z, long rows, int C, float *e)
{
    int nchunk = C / 8;
    for (long i = 0; i < rows; ++i) {
        const float *zi = z + i * (long)C;
        float s[32];
        for (int l = 0; l < 32; ++l) {
            float acc = 0.0f;
            for (int ch = l; ch < nchunk; ch += 32)
                for (int k = 0; k < 8; ++k) {
                    float v = zi[ch * 8 + k];
                    acc = fmaf(v, v, acc);
                }
            s[l] = acc;
        }
        for (int w = 16; w >= 1; w /= 2)
            for (int l = 0; l < w; ++l) s[l] = s[l] + s[l + w];
        e[i] = s[0];
    }
}

/* Energy in fp64 (for checking the canonical order against exact ranking). */
void or_energy_exact(const float *z, long rows, int C, double *e)
{
    for (long i = 0; i < rows; ++i) {
        double acc = 0.0;
        for (int k = 0; k < C; ++k) {
            double v = (double)z[i * (long)C + k];
            acc += v * v;
        }
        e[i] = acc;
    }
}

/* ------------------------------------------------------------------------- */
/* Top-k keep-set inside the prior (Eq. 5)                                    */
/* ------------------------------------------------------------------------- */

long or_kmax(double rho, long mn)
{
    return (long)floor(rho * (double)mn);
}

typedef struct { float e; int32_t i; } cell_t;

static int cmp_rank(const void *a, const void *b)
{
    const cell_t *x = (const cell_t *)a, *y = (const cell_t *)b;
    if (x->e > y->e) return -1;   /* larger energy first */
    if (x->e < y->e) return 1;
    return (x->i < y->i) ? -1 : (x->i > y->i);   /* then lower index */
}

static int cmp_i32(const void *a, const void *b)
{
    int32_t x = *(const int32_t *)a, y = *(const int32_t *)b;
    return (x < y) ? -1 : (x > y);
}

/* K_r = the min(k, |P|) best cells of P by (energy desc, index asc), written
 * in ascending grid order.  Returns |K_r|. */
long or_topk(const uint8_t *P, const float *e, long mn, long k, int32_t *idx)
{
    cell_t *c = (cell_t *)malloc(sizeof(cell_t) * (size_t)(mn > 0 ? mn : 1));
    long np = 0;
    for (long i = 0; i < mn; ++i)
        if (P[i]) { c[np].e = e[i]; c[np].i = (int32_t)i; ++np; }
    qsort(c, (size_t)np, sizeof(cell_t), cmp_rank);
    long keep = np < k ? np : k;
    if (keep < 0) keep = 0;
    for (long j = 0; j < keep; ++j) idx[j] = c[j].i;
    qsort(idx, (size_t)keep, sizeof(int32_t), cmp_i32);
    free(c);
    return keep;
}

/* Full read-side selection for one frame (Algorithm 1, per-frame loop up to
 * the arg-top): per-unit priors, union over each group's objects when
 * union_mode is set, energies of the group's grid, top-k.
 *   z      [G][mn][C] fp32 values (bf16 inputs widened exactly)
 *   masks  [U][mn] previous-frame masks;  unit_group [U] in [0, G)
 *   track  [U][6] in/out;  idx [U][kmax];  count [U]
 *   prior_out [U][mn] (nullable): the prior each unit selected from
 *   energy_out [G][mn] (nullable): canonical energies */
void or_select(const float *z, int G, int m, int n, int C, const uint8_t *masks,
               const int32_t *unit_group, int U, int32_t *track, double rho, int r_s,
               int c, int union_mode, int bbox_mode, int32_t *idx, int32_t *count,
               uint8_t *prior_out, float *energy_out)
{
    long mn = (long)m * n;
    long k = or_kmax(rho, mn);
    uint8_t *own = (uint8_t *)malloc((size_t)(U > 0 ? U : 1) * (size_t)mn);
    float *e = (float *)malloc(sizeof(float) * (size_t)(G > 0 ? G : 1) * (size_t)mn);
    uint8_t *P = (uint8_t *)malloc((size_t)mn);
    for (int u = 0; u < U; ++u)
        or_prior_unit(masks + (long)u * mn, m, n, track + 6L * u, r_s, c, bbox_mode,
                      own + (long)u * mn);
    for (int g = 0; g < G; ++g) or_energy_canonical(z + (long)g * mn * C, mn, C, e + (long)g * mn);
    for (int u = 0; u < U; ++u) {
        int g = unit_group[u];
        if (union_mode) {
            memset(P, 0, (size_t)mn);
            for (int v = 0; v < U; ++v)
                if (unit_group[v] == g)
                    for (long i = 0; i < mn; ++i) P[i] |= own[(long)v * mn + i];
        } else {
            memcpy(P, own + (long)u * mn, (size_t)mn);
        }
        if (prior_out) memcpy(prior_out + (long)u * mn, P, (size_t)mn);
        count[u] = (int32_t)or_topk(P, e + (long)g * mn, mn, k, idx + (long)u * k);
    }
    if (energy_out) memcpy(energy_out, e, sizeof(float) * (size_t)G * (size_t)mn);
    free(own);
    free(e);
    free(P);
}

/* ------------------------------------------------------------------------- */
/* Sparse memory attention readout (Eq. 6) with RoPE by index (Eq. 7)         */
/* ------------------------------------------------------------------------- */

typedef struct {
    const double *q; long mn; int H, d;
    const int32_t *idx; long cnt;
    const double *K, *V; long N;
    const float *rope; double scale;
    double *A;
    int tid, nth;
} readout_job;

static void *readout_worker(void *arg)
{
    readout_job *jb = (readout_job *)arg;
    int H = jb->H, d = jb->d;
    long D = (long)H * d;
    double *qv = (double *)malloc(sizeof(double) * (size_t)d);
    double *s = (double *)malloc(sizeof(double) * (size_t)(jb->N > 0 ? jb->N : 1));
    for (long j = jb->tid; j < jb->cnt; j += jb->nth) {
        long cell = jb->idx[j];
        for (int h = 0; h < H; ++h) {
            const double *qs = jb->q + cell * D + (long)h * d;
            /* Eq. 7: rotate pair (2p, 2p+1) by the table entry of this query's
             * own grid cell, f[cell, p] = cos + i sin. */
            for (int p = 0; p < d / 2; ++p) {
                double a = qs[2 * p], b = qs[2 * p + 1];
                if (jb->rope) {
                    double cs = jb->rope[(cell * (d / 2) + p) * 2 + 0];
                    double sn = jb->rope[(cell * (d / 2) + p) * 2 + 1];
                    qv[2 * p] = a * cs - b * sn;
                    qv[2 * p + 1] = a * sn + b * cs;
                } else {
                    qv[2 * p] = a;
                    qv[2 * p + 1] = b;
                }
            }
            double *out = jb->A + j * D + (long)h * d;
            for (int c = 0; c < d; ++c) out[c] = 0.0;
            if (jb->N == 0) continue;
            double mx = -INFINITY;
            for (long t = 0; t < jb->N; ++t) {
                const double *kt = jb->K + t * D + (long)h * d;
                double acc = 0.0;
                for (int c = 0; c < d; ++c) acc += qv[c] * kt[c];
                s[t] = acc * jb->scale;
                if (s[t] > mx) mx = s[t];
            }
            double l = 0.0;
            for (long t = 0; t < jb->N; ++t) {
                s[t] = exp(s[t] - mx);
                l += s[t];
            }
            for (long t = 0; t < jb->N; ++t) {
                const double *vt = jb->V + t * D + (long)h * d;
                double p = s[t] / l;
                for (int c = 0; c < d; ++c) out[c] += p * vt[c];
            }
        }
    }
    free(qv);
    free(s);
    return NULL;
}

/* A[j] = softmax(q~_j K^T * scale) V per head, q~_j = q[idx[j]] (rotated by
 * f[idx[j]] when a table is given).  q [mn][H*d]; K, V [N][H*d] in the unit's
 * logical bank order; rope [mn][d/2][2] (cos, sin) or NULL; A [cnt][H*d].
 * Rows are independent, so the thread count does not change the result. */
void or_readout(const double *q, long mn, int H, int d, const int32_t *idx, long cnt,
                const double *K, const double *V, long N, const float *rope,
                double scale, double *A, int threads)
{
    if (threads < 1) threads = 1;
    if (threads > 256) threads = 256;
    pthread_t th[256];
    readout_job jb[256];
    for (int t = 0; t < threads; ++t) {
        readout_job x = {q, mn, H, d, idx, cnt, K, V, N, rope, scale, A, t, threads};
        jb[t] = x;
    }
    if (threads == 1) {
        readout_worker(&jb[0]);
        return;
    }
    for (int t = 0; t < threads; ++t) pthread_create(&th[t], NULL, readout_worker, &jb[t]);
    for (int t = 0; t < threads; ++t) pthread_join(th[t], NULL);
}

/* fp64 -> bf16 bits, one rounding (nearest, ties to even), for finite values in
 * the normal bf16 range.  The low 45 mantissa bits of the double are cut off,
 * which gives the candidate toward zero; the candidate one bf16 step further
 * out is compared by distance. */
uint16_t or_round_bf16(double x)
{
    union { double d; uint64_t u; } v = {x};
    union { float f; uint32_t u; } w;
    if (x == 0.0) return (uint16_t)((v.u >> 63) << 15);
    uint64_t lo_bits = v.u & ~((1ULL << 45) - 1);
    union { double d; uint64_t u; } lo = {0};
    lo.u = lo_bits;
    union { double d; uint64_t u; } hi = {0};
    hi.u = lo_bits + (1ULL << 45);            /* next bf16 step away from zero */
    double dlo = fabs(x - lo.d), dhi = fabs(hi.d - x);
    double pick;
    if (dlo < dhi) pick = lo.d;
    else if (dhi < dlo) pick = hi.d;
    else pick = ((lo_bits >> 45) & 1ULL) ? hi.d : lo.d;   /* tie: even mantissa */
    w.f = (float)pick;                         /* exact: pick has <= 8 significant bits */
    return (uint16_t)(w.u >> 16);
}

void or_round_bf16_array(const double *x, long n, uint16_t *out)
{
    for (long i = 0; i < n; ++i) out[i] = or_round_bf16(x[i]);
}

/* ------------------------------------------------------------------------- */
/* Write side: keep-set (Eq. 8) and bank commit (Algorithm 1, sparse write)  */
/* ------------------------------------------------------------------------- */

/* K_w per unit.  S = the unit's seed mask, or in union mode the union of the
 * seeds of its group.  If fall_through is set and |S|/mn > hi or < lo, K_w is
 * the full grid (Sec. 3.2: such frames are written unpruned);
 * otherwise K_w = dilate_{D_w}(S) (the union of per-object dilations equals
 * the dilation of the union). */
void or_write_keepset(const uint8_t *seeds, const int32_t *unit_group, int U, int m, int n,
                      int D_w, double fall_lo, double fall_hi, int fall_through,
                      int union_mode, uint8_t *kw)
{
    long mn = (long)m * n;
    uint8_t *S = (uint8_t *)malloc((size_t)mn);
    for (int u = 0; u < U; ++u) {
        memset(S, 0, (size_t)mn);
        for (int v = 0; v < U; ++v) {
            int take = union_mode ? (unit_group[v] == unit_group[u]) : (v == u);
            if (take)
                for (long i = 0; i < mn; ++i) S[i] |= seeds[(long)v * mn + i];
        }
        long area = 0;
        for (long i = 0; i < mn; ++i) area += S[i] ? 1 : 0;
        double frac = (double)area / (double)mn;
        if (fall_through && (frac > fall_hi || frac < fall_lo))
            memset(kw + (long)u * mn, 1, (size_t)mn);
        else
            or_dilate(S, m, n, D_w, kw + (long)u * mn);
    }
    free(S);
}

/* Bank of one unit.  Storage rows: [0, pinned_cap) pinned conditioning frames
 * packed in commit order; [pinned_cap, pinned_cap + ring_cap) a ring holding
 * the recent frames at logical positions p -> pinned_cap + (p mod ring_cap);
 * then n_ptr pointer rows.  state = {head, tail, cond_len, n_frames, oldest,
 * n_cond_frames, ptr_len, cond_frames_cap}; foff/flen: frame ring of
 * max_frames entries (logical offset, length), oldest at index `oldest`.
 *
 * Commit appends the rows of knew/vnew whose mask is set, in ascending grid
 * order (mask NULL = every row).  A conditioning commit goes to the pinned
 * region; any other commit first evicts the oldest ring frame when `window`
 * frames are held (window > 0).  A commit that does not fit (pinned frames
 * exhausted, ring full, frame table full) changes nothing and returns 2. */
int or_commit_unit(uint8_t *kst, uint8_t *vst, long row_bytes, const uint8_t *knew,
                   const uint8_t *vnew, const uint8_t *mask, long mn, int is_cond,
                   int window, long pinned_cap, long ring_cap, int max_frames,
                   int64_t *state, int64_t *foff, int32_t *flen)
{
    long L = 0;
    for (long i = 0; i < mn; ++i) L += (mask == NULL || mask[i]) ? 1 : 0;
    if (is_cond) {
        if (state[5] >= state[7]) return 2;
        if (state[2] + L > pinned_cap) return 2;
        long dst = state[2];
        for (long i = 0; i < mn; ++i)
            if (mask == NULL || mask[i]) {
                memcpy(kst + dst * row_bytes, knew + i * row_bytes, (size_t)row_bytes);
                memcpy(vst + dst * row_bytes, vnew + i * row_bytes, (size_t)row_bytes);
                ++dst;
            }
        state[2] += L;
        state[5] += 1;
        return 0;
    }
    int64_t head = state[0], tail = state[1];
    int64_t n_frames = state[3], oldest = state[4];
    if (window > 0 && n_frames == window) {      /* evict the oldest frame */
        head += flen[oldest];
        oldest = (oldest + 1) % max_frames;
        n_frames -= 1;
    }
    if (n_frames >= max_frames) return 2;
    if ((tail - head) + L > ring_cap) return 2;
    long j = 0;
    for (long i = 0; i < mn; ++i)
        if (mask == NULL || mask[i]) {
            long phys = pinned_cap + (long)((tail + j) % ring_cap);
            memcpy(kst + phys * row_bytes, knew + i * row_bytes, (size_t)row_bytes);
            memcpy(vst + phys * row_bytes, vnew + i * row_bytes, (size_t)row_bytes);
            ++j;
        }
    int64_t slot = (oldest + n_frames) % max_frames;
    foff[slot] = tail;
    flen[slot] = (int32_t)L;
    state[0] = head;
    state[1] = tail + L;
    state[3] = n_frames + 1;
    state[4] = oldest;
    return 0;
}

/* ------------------------------------------------------------------------- */
/* Decoder side (Sec. 3.3): per-object closure, then the palette argmax      */
/* ------------------------------------------------------------------------- */

/* out(y,x) = 1 iff every pixel (y',x') of the array with |y-y'| <= r and
 * |x-x'| <= r is set (the window clipped to the array). */
void or_erode(const uint8_t *M, int h, int w, int r, uint8_t *out)
{
    for (int y = 0; y < h; ++y)
        for (int x = 0; x < w; ++x) {
            int all = 1;
            for (int yy = y - r; yy <= y + r && all; ++yy) {
                if (yy < 0 || yy >= h) continue;
                for (int xx = x - r; xx <= x + r; ++xx) {
                    if (xx < 0 || xx >= w) continue;
                    if (!M[(long)yy * w + xx]) { all = 0; break; }
                }
            }
            out[(long)y * w + x] = (uint8_t)all;
        }
}

/* Closure with the (2r+1) x (2r+1) square: dilation, then erosion (Sec. 3.3
 * uses r = 4, a 9 x 9 element).  The object is a set of pixels of the
 * unbounded plane with nothing set outside the image; both operations are
 * taken in the plane and the result is cut back to the image.  Written out:
 * the image is embedded in a zero frame 2r pixels wide, where no clipped
 * window of the two passes reaches the frame's edge for the pixels kept. */
void or_close(const uint8_t *M, int h, int w, int r, uint8_t *out)
{
    int H = h + 4 * r, W = w + 4 * r;
    uint8_t *pad = (uint8_t *)calloc((size_t)H * W, 1);
    uint8_t *dil = (uint8_t *)malloc((size_t)H * W);
    uint8_t *ero = (uint8_t *)malloc((size_t)H * W);
    for (int y = 0; y < h; ++y)
        for (int x = 0; x < w; ++x) pad[(long)(y + 2 * r) * W + (x + 2 * r)] = M[(long)y * w + x];
    or_dilate(pad, H, W, r, dil);
    or_erode(dil, H, W, r, ero);
    for (int y = 0; y < h; ++y)
        for (int x = 0; x < w; ++x) out[(long)y * w + x] = ero[(long)(y + 2 * r) * W + (x + 2 * r)];
    free(pad);
    free(dil);
    free(ero);
}

/* One group of nobj objects at the decoder's resolution h x w.
 *   logits  [nobj][h][w] fp32 decoder mask logits; object o's binary mask is
 *           logit > 0
 *   closed  [nobj][h][w] out: close_r of each object's mask
 *   palette [h][w] out: 0 where no closed mask holds the pixel, otherwise
 *           1 + o for the object o with the largest logit among the objects
 *           whose closed mask holds it (the lower o on equal logits).
 * The closure comes first and the argmax second, the order of Sec. 3.3. */
void or_close_argmax(const float *logits, int nobj, int h, int w, int r, uint8_t *closed,
                     uint8_t *palette)
{
    long hw = (long)h * w;
    uint8_t *bin = (uint8_t *)malloc((size_t)hw);
    for (int o = 0; o < nobj; ++o) {
        for (long i = 0; i < hw; ++i) bin[i] = logits[(long)o * hw + i] > 0.0f;
        or_close(bin, h, w, r, closed + (long)o * hw);
    }
    for (long i = 0; i < hw; ++i) {
        int best = -1;
        for (int o = 0; o < nobj; ++o) {
            if (!closed[(long)o * hw + i]) continue;
            if (best < 0 || logits[(long)o * hw + i] > logits[(long)best * hw + i]) best = o;
        }
        palette[i] = (uint8_t)(best + 1);
    }
    free(bin);
}

/* ------------------------------------------------------------------------- */
/* Pixel space to token grid (Sec. 3.1: down_s and the seed box of Eq. 1)    */
/* ------------------------------------------------------------------------- */

/* Nearest-neighbour down_s: grid cell (i, j) of the (h/s) x (w/s) grid takes
 * pixel (i*s, j*s). */
void or_downsample(const uint8_t *M, int h, int w, int s, uint8_t *out)
{
    int m = h / s, n = w / s;
    for (int i = 0; i < m; ++i)
        for (int j = 0; j < n; ++j) out[(long)i * n + j] = M[(long)i * s * w + (long)j * s] != 0;
}

/* Seed of one object: the tight pixel box of M (inclusive), each corner
 * coordinate divided by s with the quotient rounded down.  track = {y0, x0,
 * y1, x1, valid, streak}: valid 1 and streak 0 when M has a set pixel; an
 * empty M gives {0, 0, 0, 0, 0, 0}.  Returns valid. */
int or_seed_track(const uint8_t *M, int h, int w, int s, int32_t *track)
{
    int32_t box[4];
    for (int k = 0; k < 6; ++k) track[k] = 0;
    if (!or_bbox(M, h, w, box)) return 0;
    for (int k = 0; k < 4; ++k) track[k] = box[k] / s;
    track[4] = 1;
    return 1;
}
