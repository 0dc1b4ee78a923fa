// rs3_bank.cu -- ragged per-unit memory bank and the write-pruned commit
// (Sec. 3.2, Eq. 8; Algorithm 1's sparse write).
//
// A commit is one launch (k_commit): a CTA per (128-cell chunk, unit) ranks
// its kept cells with ballot/popc and copies their K and V rows with 128-bit
// accesses, the first rows' loads in flight while the unit's counts and the
// capacity decision are made; the last CTA of each unit publishes the new
// counters.
#include "rs3_internal.cuh"

#include <cstdlib>
#include <cstring>

namespace {

struct BankDev {
    int64_t *meta;
    int64_t stride_words;
    int32_t max_frames, window, n_cond, n_ptr;
    int64_t pinned_cap, ring_cap, rows_per_unit;
};

BankDev bank_dev(const rs3_bank *b)
{
    BankDev v;
    v.meta = static_cast<int64_t *>(b->meta);
    v.stride_words = b->meta_stride / 8;
    v.max_frames = b->max_frames;
    v.window = b->window;
    v.n_cond = b->n_cond;
    v.n_ptr = b->n_ptr;
    v.pinned_cap = b->pinned_cap;
    v.ring_cap = b->ring_cap;
    v.rows_per_unit = b->rows_per_unit;
    return v;
}

// Copies `nvec` 16-byte words of one row (one warp).
__device__ __forceinline__ void copy_row(uint4 *__restrict__ dk, uint4 *__restrict__ dv,
                                         const uint4 *__restrict__ sk, const uint4 *__restrict__ sv,
                                         int nvec, int lane)
{
    for (int v = lane; v < nvec; v += 32) {
        const uint4 a = __ldcs(sk + v);
        const uint4 b = __ldcs(sv + v);
        dk[v] = a;
        dv[v] = b;
    }
}

// Eq. 7 on the key side: one 16-byte piece of a key row (bf16: four pairs,
// fp32: two pairs; element 2i and 2i + 1 of a head form pair i) rotated by
// the (cos, sin) of those pairs at the row's own cell, in fp32, then rounded
// once to the stored type.  f points at the first pair's (cos, sin).
__device__ __forceinline__ uint4 rotate_piece(uint4 v, const float *__restrict__ f, int esz)
{
    if (esz == 2) {
        const float4 a = __ldg(reinterpret_cast<const float4 *>(f));
        const float4 b = __ldg(reinterpret_cast<const float4 *>(f) + 1);
        const float cs[4] = {a.x, a.z, b.x, b.z}, sn[4] = {a.y, a.w, b.y, b.w};
        uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float x0 = __uint_as_float(w[i] << 16), x1 = __uint_as_float(w[i] & 0xffff0000u);
            const float y0 = x0 * cs[i] - x1 * sn[i], y1 = x0 * sn[i] + x1 * cs[i];
            uint32_t r;
            asm("cvt.rn.bf16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(y1), "f"(y0));
            w[i] = r;
        }
        return make_uint4(w[0], w[1], w[2], w[3]);
    }
    const float4 a = __ldg(reinterpret_cast<const float4 *>(f));
    const float x0 = __uint_as_float(v.x), x1 = __uint_as_float(v.y);
    const float x2 = __uint_as_float(v.z), x3 = __uint_as_float(v.w);
    return make_uint4(__float_as_uint(x0 * a.x - x1 * a.y), __float_as_uint(x0 * a.y + x1 * a.x),
                      __float_as_uint(x2 * a.z - x3 * a.w), __float_as_uint(x2 * a.w + x3 * a.z));
}

// Number of nonzero bytes in a 16-byte word.
__device__ __forceinline__ int nonzero_bytes(uint4 w)
{
    return (__popc(__vcmpne4(w.x, 0u)) + __popc(__vcmpne4(w.y, 0u)) + __popc(__vcmpne4(w.z, 0u)) +
            __popc(__vcmpne4(w.w, 0u))) >> 3;
}

// The commit of one frame, in one launch: CTA (c, u) owns cells
// [c * CHUNK, (c+1) * CHUNK) of unit u, one cell per thread (CHUNK = 128, or
// 64 where 128-cell chunks would give fewer than two CTAs per SM).
// Its latency chain is two memory round trips: (1) the chunk's own mask bytes
// and the unit's whole mask row (the kept rows before the chunk and in the
// unit) are loaded together; (2) as soon as the chunk's kept cells are ranked
// (ballot / popc) their first K and V pieces are loaded into registers, and
// the unit's counts and the eviction / capacity decision (thread 0, from the
// old counters) are made while those loads are in flight; then the pieces
// are stored at their ring rows.  Every CTA arrives on the unit's counter
// once thread 0 has read the old counters, and the last to arrive publishes
// the new ones after its own stores, so no CTA can read counters of the frame
// it copies (the readers of the bank are later launches).
constexpr int COMMIT_PF = 8;        // kept rows per warp and batch (one piece per lane and row)

// Loads piece v of rows j0, j0 + NW, ... of the chunk's kept list (NW warps).
template <int NW>
__device__ __forceinline__ void commit_load(uint4 (&kk)[COMMIT_PF], uint4 (&vv)[COMMIT_PF],
                                            const int32_t *s_list, int nk, int j0, int v, int nvec,
                                            const uint8_t *ksrc, const uint8_t *vsrc, int64_t row_bytes)
{
#pragma unroll
    for (int r = 0; r < COMMIT_PF; ++r) {
        const int j = j0 + NW * r;
        if (j < nk && v < nvec) {
            const int64_t so = (int64_t)s_list[j] * row_bytes + 16 * v;
            kk[r] = __ldcs(reinterpret_cast<const uint4 *>(ksrc + so));
            vv[r] = __ldcs(reinterpret_cast<const uint4 *>(vsrc + so));
        }
    }
}

// Stores those pieces at bank row row0 + j (a ring position, wrapped once,
// past the pinned region; or a pinned row for a conditioning frame).
template <int NW, bool ROPE>
__device__ __forceinline__ void commit_store(const uint4 (&kk)[COMMIT_PF], const uint4 (&vv)[COMMIT_PF],
                                             const int32_t *s_list, int nk, int j0, int v, int nvec,
                                             int64_t row0, int is_cond, const BankDev &bk,
                                             uint8_t *kdst, uint8_t *vdst, int64_t row_bytes,
                                             const float *rope, int d, int esz)
{
#pragma unroll
    for (int r = 0; r < COMMIT_PF; ++r) {
        const int j = j0 + NW * r;
        if (j < nk && v < nvec) {
            int64_t row = row0 + j;
            if (!is_cond) row = bk.pinned_cap + (row >= bk.ring_cap ? row - bk.ring_cap : row);
            const int64_t dst = row * row_bytes + 16 * v;
            uint4 k = kk[r];
            if (ROPE) {                                    // keys stored rotated by their own cell
                const int e = (16 * v) / esz;              // first element of the piece
                k = rotate_piece(k, rope + ((int64_t)s_list[j] * (d / 2) + (e % d) / 2) * 2, esz);
            }
            *reinterpret_cast<uint4 *>(kdst + dst) = k;
            *reinterpret_cast<uint4 *>(vdst + dst) = vv[r];
        }
    }
}

template <int CHUNK, bool ROPE>
__global__ void __launch_bounds__(CHUNK)
k_commit(const uint8_t *__restrict__ k_new, const uint8_t *__restrict__ v_new,
         const uint8_t *__restrict__ mask, int mn, int is_cond, int64_t row_bytes, BankDev bk,
         uint8_t *__restrict__ k_store, uint8_t *__restrict__ v_store, int32_t *status,
         const float *__restrict__ rope, int d, int esz)
{
    constexpr int NW = CHUNK / 32;
    pdl_wait();
    __shared__ int32_t s_list[CHUNK];
    __shared__ int32_t s_wc[NW];
    __shared__ int32_t s_red[2][NW];
    __shared__ int64_t s_row0;
    __shared__ int s_ok;
    const int u = blockIdx.y, ch = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int c0 = ch * CHUNK;
    int64_t *mu = bk.meta + (int64_t)u * bk.stride_words;
    const uint8_t *Mu = mask ? mask + (size_t)u * mn : nullptr;

    // the unit's old counters (thread 0 decides for the CTA)
    int64_t head0 = 0, tail0 = 0, nf0 = 0, oldest0 = 0, cond_len0 = 0, ncond0 = 0;
    if (threadIdx.x == 0) {
        head0 = mu[BM_HEAD]; tail0 = mu[BM_TAIL];
        nf0 = mu[BM_NFRAMES]; oldest0 = mu[BM_OLDEST];
        cond_len0 = mu[BM_COND_LEN]; ncond0 = mu[BM_NCOND];
    }

    // round trip 1: this thread's cell, and the kept rows of the unit and of
    // the chunks before this one (16-byte loads when the unit's mask row is
    // aligned, bytes for the rest)
    const int cell = c0 + threadIdx.x;
    const bool keep = cell < mn && (Mu ? Mu[cell] != 0 : true);
    int total = 0, before = 0;
    if (Mu) {
        const int nvec16 = (reinterpret_cast<uintptr_t>(Mu) & 15u) == 0 ? (mn >> 4) : 0;
#pragma unroll 4
        for (int i = threadIdx.x; i < nvec16; i += CHUNK) {
            const int c = nonzero_bytes(__ldg(reinterpret_cast<const uint4 *>(Mu) + i));
            total += c;
            before += i * 16 < c0 ? c : 0;
        }
        for (int i = nvec16 * 16 + threadIdx.x; i < mn; i += CHUNK) {
            const int c = Mu[i] != 0;
            total += c;
            before += i < c0 ? c : 0;
        }
    }

    // ranks of the chunk's kept cells, in cell order
    const uint32_t bal = __ballot_sync(0xffffffffu, keep);
    if (lane == 0) s_wc[warp] = __popc(bal);
    __syncthreads();
    int off = 0, nk = 0;
#pragma unroll
    for (int w = 0; w < NW; ++w) {
        off += w < warp ? s_wc[w] : 0;
        nk += s_wc[w];
    }
    if (keep) {
        uint32_t lm;
        asm("mov.u32 %0, %%lanemask_lt;" : "=r"(lm));
        s_list[off + __popc(bal & lm)] = cell;
    }
    __syncthreads();

    // round trip 2: the first batch of the chunk's rows in flight ...
    const int nvec = (int)(row_bytes / 16);
    const uint8_t *ksrc = k_new + (size_t)u * mn * row_bytes;
    const uint8_t *vsrc = v_new + (size_t)u * mn * row_bytes;
    uint4 kk[COMMIT_PF], vv[COMMIT_PF];
    commit_load<NW>(kk, vv, s_list, nk, warp, lane, nvec, ksrc, vsrc, row_bytes);

    // ... while the unit's counts are summed and thread 0 decides
    if (Mu) {
        total = warp_sum(total);
        before = warp_sum(before);
        if (lane == 0) { s_red[0][warp] = total; s_red[1][warp] = before; }
    }
    __syncthreads();
    bool ok = false;
    int64_t L = 0, head = head0, oldest = oldest0, nf = nf0;
    if (threadIdx.x == 0) {
        int64_t pre = 0;
        if (Mu) {
#pragma unroll
            for (int w = 0; w < NW; ++w) { L += s_red[0][w]; pre += s_red[1][w]; }
        } else {
            L = mn;
            pre = c0;
        }
        int64_t row0 = 0;
        if (is_cond) {
            ok = ncond0 < bk.n_cond && cond_len0 + L <= bk.pinned_cap;
            row0 = cond_len0 + pre;
        } else {
            const bool sane = head0 >= 0 && tail0 >= head0 && nf0 >= 0 && nf0 <= bk.max_frames &&
                              oldest0 >= 0 && oldest0 < bk.max_frames;
            if (!sane) {
                if (ch == 0) latch_status(status, RS3_EINTERNAL);
            } else {
                if (bk.window > 0 && nf == bk.window) {      // evict the oldest ring frame
                    head += mu[BM_HEADER_WORDS + bk.max_frames + oldest];
                    oldest = oldest + 1 == bk.max_frames ? 0 : oldest + 1;
                    nf -= 1;
                }
                ok = nf < bk.max_frames && (tail0 - head) + L <= bk.ring_cap;
                if (ok && L > 0) row0 = (tail0 + pre) % bk.ring_cap;   // it fits: rows wrap at most once
            }
        }
        s_ok = ok;
        s_row0 = row0;
    }
    __syncthreads();

    // every read of the old counters by this CTA is done: arrive
    unsigned long long arrived = 0;
    if (threadIdx.x == 0) {
        __threadfence();
        arrived = atomicAdd(reinterpret_cast<unsigned long long *>(mu + BM_ARRIVE), 1ull);
    }

    if (s_ok) {
        const int64_t row0 = s_row0;
        uint8_t *kdst = k_store + (size_t)u * bk.rows_per_unit * row_bytes;
        uint8_t *vdst = v_store + (size_t)u * bk.rows_per_unit * row_bytes;
        commit_store<NW, ROPE>(kk, vv, s_list, nk, warp, lane, nvec, row0, is_cond, bk, kdst, vdst,
                               row_bytes, rope, d, esz);
        // the rest of the chunk (rows past the first batch, pieces past 32 per row)
        for (int vb = 0; vb < nvec; vb += 32) {
            for (int jb = vb == 0 ? NW * COMMIT_PF : 0; jb < nk; jb += NW * COMMIT_PF) {
                commit_load<NW>(kk, vv, s_list, nk, jb + warp, vb + lane, nvec, ksrc, vsrc, row_bytes);
                commit_store<NW, ROPE>(kk, vv, s_list, nk, jb + warp, vb + lane, nvec, row0, is_cond, bk, kdst,
                                       vdst, row_bytes, rope, d, esz);
            }
        }
    }

    // the last CTA of the unit to arrive publishes the new counters
    if (threadIdx.x != 0 || arrived != (unsigned long long)(gridDim.x - 1)) return;
    __threadfence();
    mu[BM_ARRIVE] = 0;
    if (!ok) {
        if (is_cond || (head0 >= 0 && tail0 >= head0)) latch_status(status, RS3_ECAPACITY);
        return;
    }
    if (is_cond) {
        mu[BM_COND_LEN] = cond_len0 + L;
        mu[BM_NCOND] = ncond0 + 1;
    } else {
        int64_t *fo = mu + BM_HEADER_WORDS;
        int64_t *fl = fo + bk.max_frames;
        const int64_t slot = (oldest + nf) % bk.max_frames;
        fo[slot] = tail0;
        fl[slot] = L;
        mu[BM_HEAD] = head;
        mu[BM_TAIL] = tail0 + L;
        mu[BM_NFRAMES] = nf + 1;
        mu[BM_OLDEST] = oldest;
    }
}

__global__ void k_set_pointers(const uint8_t *__restrict__ kp, const uint8_t *__restrict__ vp,
                               int64_t row_bytes, BankDev bk, uint8_t *__restrict__ k_store,
                               uint8_t *__restrict__ v_store)
{
    pdl_wait();
    const int u = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    const int nvec = (int)(row_bytes / 16);
    const int64_t row0 = bk.pinned_cap + bk.ring_cap;
    for (int j = warp; j < bk.n_ptr; j += nw) {
        const size_t src = ((size_t)u * bk.n_ptr + j) * row_bytes;
        const size_t dst = ((size_t)u * bk.rows_per_unit + row0 + j) * row_bytes;
        copy_row(reinterpret_cast<uint4 *>(k_store + dst), reinterpret_cast<uint4 *>(v_store + dst),
                 reinterpret_cast<const uint4 *>(kp + src), reinterpret_cast<const uint4 *>(vp + src),
                 nvec, lane);
    }
    __syncthreads();
    if (threadIdx.x == 0) bk.meta[(int64_t)u * bk.stride_words + BM_PTRLEN] = bk.n_ptr;
}

__global__ void k_bank_reset(BankDev bk, int unit, int U)
{
    pdl_wait();
    const int u0 = unit < 0 ? 0 : unit, u1 = unit < 0 ? U : unit + 1;
    for (int u = u0 + blockIdx.x; u < u1; u += gridDim.x) {
        int64_t *mu = bk.meta + (int64_t)u * bk.stride_words;
        for (int w = threadIdx.x; w < BM_HEADER_WORDS; w += blockDim.x) mu[w] = 0;
    }
}

bool bank_ok(const rs3_bank *b)
{
    return b && b->magic == RS3_BANK_MAGIC && b->meta && b->k_store && b->v_store && b->U >= 1;
}

size_t elem_bytes(int dtype) { return dtype == RS3_BF16 ? 2 : 4; }

}  // namespace

extern "C" rs3_status rs3_bank_layout(int U, int H, int d, rs3_dtype dtype, int mn, int n_cond,
                                      int window, int64_t ring_cap_rows, int max_frames, int n_ptr,
                                      int64_t *rows_per_unit, size_t *meta_bytes)
{
    if (U < 1 || H < 1 || d < 1 || mn < 1 || n_cond < 0 || n_ptr < 0 || ring_cap_rows < 0)
        return RS3_EINVAL;
    if (dtype != RS3_F32 && dtype != RS3_BF16) return RS3_EINVAL;
    if (mn > RS3_MAX_MN) return RS3_EUNSUPPORTED;
    if (U > 65535) return RS3_EUNSUPPORTED;          // a commit's grid holds a row of CTAs per unit
    if (((int64_t)H * d * (int64_t)elem_bytes(dtype)) % 16 != 0) return RS3_EINVAL;
    if (window == 0 || window < -1) return RS3_EINVAL;
    if (window > 0) {
        if (max_frames != window) return RS3_EINVAL;
        if (ring_cap_rows < (int64_t)window * mn) return RS3_EINVAL;
    } else if (max_frames < 1) {
        return RS3_EINVAL;
    }
    const int64_t rows = (int64_t)n_cond * mn + ring_cap_rows + n_ptr;
    if (rows_per_unit) *rows_per_unit = rows;
    if (meta_bytes) *meta_bytes = (size_t)U * (size_t)bank_meta_words(max_frames) * 8;
    return RS3_OK;
}

extern "C" rs3_status rs3_bank_init(rs3_bank *bank, int U, int H, int d, rs3_dtype dtype, int mn,
                                    int n_cond, int window, int64_t ring_cap_rows, int max_frames,
                                    int n_ptr, void *k_store, void *v_store, void *meta,
                                    rs3_stream_t stream)
{
    if (!bank || !k_store || !v_store || !meta) return RS3_EINVAL;
    int64_t rows;
    size_t mb;
    const rs3_status s = rs3_bank_layout(U, H, d, dtype, mn, n_cond, window, ring_cap_rows,
                                         max_frames, n_ptr, &rows, &mb);
    if (s != RS3_OK) return s;
    if (!rs3_aligned16(k_store) || !rs3_aligned16(v_store) || !rs3_aligned16(meta)) return RS3_EINVAL;
    std::memset(bank, 0, sizeof(*bank));
    bank->U = U; bank->H = H; bank->d = d; bank->D = H * d;
    bank->dtype = dtype; bank->mn = mn; bank->n_cond = n_cond; bank->window = window;
    bank->max_frames = max_frames; bank->n_ptr = n_ptr;
    bank->pinned_cap = (int64_t)n_cond * mn;
    bank->ring_cap = ring_cap_rows;
    bank->rows_per_unit = rows;
    bank->meta_stride = bank_meta_words(max_frames) * 8;
    bank->k_store = k_store; bank->v_store = v_store; bank->meta = meta;
    bank->magic = RS3_BANK_MAGIC;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const size_t store_bytes = (size_t)U * (size_t)rows * (size_t)H * d * elem_bytes(dtype);
    if (cudaMemsetAsync(meta, 0, mb, st) != cudaSuccess ||
        cudaMemsetAsync(k_store, 0, store_bytes, st) != cudaSuccess ||
        cudaMemsetAsync(v_store, 0, store_bytes, st) != cudaSuccess)
        return RS3_ECUDA;
    return RS3_OK;
}

namespace {

rs3_status commit_launch(const rs3_bank *bank, const void *k_new, const void *v_new, const uint8_t *keep_mask,
                         int is_cond, const float *rope, int32_t *status, rs3_stream_t stream)
{
    if (!bank_ok(bank) || !k_new || !v_new || !status) return RS3_EINVAL;
    if (is_cond != 0 && is_cond != 1) return RS3_EINVAL;
    if (is_cond && bank->n_cond == 0) return RS3_EINVAL;
    if (!rs3_aligned16(k_new) || !rs3_aligned16(v_new)) return RS3_EINVAL;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    const BankDev bk = bank_dev(bank);
    const int mn = bank->mn;
    const int64_t row_bytes = (int64_t)bank->D * (int64_t)elem_bytes(bank->dtype);
    // 128-cell chunks, or 64-cell ones where those would give under two CTAs per SM
    const bool small = (int64_t)((mn + 127) / 128) * bank->U < 2ll * rs3_sm_count();
    const int chunk = small ? 64 : 128;
    const dim3 grid((unsigned)((mn + chunk - 1) / chunk), (unsigned)bank->U);
    void (*kern)(const uint8_t *, const uint8_t *, const uint8_t *, int, int, int64_t, BankDev, uint8_t *,
                 uint8_t *, int32_t *, const float *, int, int) =
        small ? (rope ? k_commit<64, true> : k_commit<64, false>)
              : (rope ? k_commit<128, true> : k_commit<128, false>);
    launch_pdl(kern, grid, dim3(chunk), 0, st,
        static_cast<const uint8_t *>(k_new), static_cast<const uint8_t *>(v_new), keep_mask, mn, is_cond,
        row_bytes, bk, static_cast<uint8_t *>(bank->k_store), static_cast<uint8_t *>(bank->v_store), status,
        rope, bank->d, elem_bytes(bank->dtype));
    if (cudaGetLastError() != cudaSuccess) return RS3_ECUDA;
    return RS3_OK;
}

}  // namespace

extern "C" rs3_status rs3_bank_commit(const rs3_bank *bank, const void *k_new, const void *v_new,
                                      const uint8_t *keep_mask, int is_cond, int32_t *status,
                                      rs3_stream_t stream)
{
    return commit_launch(bank, k_new, v_new, keep_mask, is_cond, nullptr, status, stream);
}

extern "C" rs3_status rs3_bank_commit_rope(const rs3_bank *bank, const void *k_new, const void *v_new,
                                           const uint8_t *keep_mask, int is_cond, const float *rope_cos_sin,
                                           int32_t *status, rs3_stream_t stream)
{
    if (!rope_cos_sin || !rs3_aligned16(rope_cos_sin)) return RS3_EINVAL;
    if (bank_ok(bank) && bank->d % 8 != 0) return RS3_EUNSUPPORTED;   // whole pairs in every 16-byte piece
    return commit_launch(bank, k_new, v_new, keep_mask, is_cond, rope_cos_sin, status, stream);
}

extern "C" rs3_status rs3_bank_set_pointers(const rs3_bank *bank, const void *k_ptr,
                                            const void *v_ptr, int32_t *status, rs3_stream_t stream)
{
    if (!bank_ok(bank) || !k_ptr || !v_ptr || !status) return RS3_EINVAL;
    if (bank->n_ptr == 0) return RS3_EINVAL;
    if (!rs3_aligned16(k_ptr) || !rs3_aligned16(v_ptr)) return RS3_EINVAL;
    const int64_t row_bytes = (int64_t)bank->D * (int64_t)elem_bytes(bank->dtype);
    launch_pdl(k_set_pointers, dim3(bank->U), dim3(256), 0, reinterpret_cast<cudaStream_t>(stream),
        static_cast<const uint8_t *>(k_ptr), static_cast<const uint8_t *>(v_ptr), row_bytes,
        bank_dev(bank), static_cast<uint8_t *>(bank->k_store), static_cast<uint8_t *>(bank->v_store));
    if (cudaGetLastError() != cudaSuccess) return RS3_ECUDA;
    return RS3_OK;
}

extern "C" rs3_status rs3_bank_reset(const rs3_bank *bank, int unit, rs3_stream_t stream)
{
    if (!bank_ok(bank)) return RS3_EINVAL;
    if (unit < -1 || unit >= bank->U) return RS3_EINVAL;
    const int blocks = unit < 0 ? (bank->U < 1024 ? bank->U : 1024) : 1;
    launch_pdl(k_bank_reset, dim3(blocks), dim3(32), 0, reinterpret_cast<cudaStream_t>(stream), bank_dev(bank), unit,
                                                                            bank->U);
    if (cudaGetLastError() != cudaSuccess) return RS3_ECUDA;
    return RS3_OK;
}

extern "C" rs3_status rs3_bank_read_meta(const rs3_bank *bank, int64_t *host_out,
                                         int64_t *frames_out, rs3_stream_t stream)
{
    if (!bank_ok(bank) || !host_out) return RS3_EINVAL;
    const size_t words = (size_t)bank->U * (size_t)(bank->meta_stride / 8);
    int64_t *tmp = static_cast<int64_t *>(std::malloc(words * 8));
    if (!tmp) return RS3_ECAPACITY;
    cudaStream_t st = reinterpret_cast<cudaStream_t>(stream);
    if (cudaMemcpyAsync(tmp, bank->meta, words * 8, cudaMemcpyDeviceToHost, st) != cudaSuccess ||
        cudaStreamSynchronize(st) != cudaSuccess) {
        std::free(tmp);
        return RS3_ECUDA;
    }
    const int64_t sw = bank->meta_stride / 8;
    for (int u = 0; u < bank->U; ++u) {
        const int64_t *mu = tmp + u * sw;
        int64_t *o = host_out + 8 * (int64_t)u;
        for (int w = 0; w < 7; ++w) o[w] = mu[w];
        o[7] = mu[BM_COND_LEN] + (mu[BM_TAIL] - mu[BM_HEAD]) + mu[BM_PTRLEN];
        if (frames_out) {
            const int64_t *foff = mu + BM_HEADER_WORDS;
            const int64_t *flen = foff + bank->max_frames;
            int64_t *fo = frames_out + (int64_t)u * bank->max_frames * 2;
            for (int i = 0; i < bank->max_frames; ++i) {
                if (i < mu[BM_NFRAMES]) {
                    const int64_t s = (mu[BM_OLDEST] + i) % bank->max_frames;
                    fo[2 * i] = foff[s];
                    fo[2 * i + 1] = flen[s];
                } else {
                    fo[2 * i] = -1;
                    fo[2 * i + 1] = -1;
                }
            }
        }
    }
    std::free(tmp);
    return RS3_OK;
}
