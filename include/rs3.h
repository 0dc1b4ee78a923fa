/*
 * rs3.h -- C ABI of librs3, the GB300 (sm_103a) hot path of RS3-Prune
 * ("Read-Sparse, Store-Sparse Token Pruning for Video Object Segmentation").
 *
 * The library implements the two hooks of the paper's Sec. 3 on a memory-bank
 * VOS network, per frame:
 *   read side  (Sec. 3.1)  rs3_select_queries  -- prior (Eq. 1, 2, 4), energy
 *                                                top-k keep-set K_r (Eq. 5)
 *                          rs3_memory_readout  -- gather (+ RoPE by index,
 *                                                Eq. 7), cross-attention over
 *                                                the unit's bank and scatter
 *                                                back to the grid (Eq. 6)
 *   write side (Sec. 3.2)  rs3_write_keepset   -- K_w (Eq. 8, fall-through)
 *                          rs3_bank_commit     -- append the kept tokens to a
 *                                                ragged per-unit bank
 *                                                (Algorithm 1, sparse write)
 *   decoder side (Sec. 3.3) rs3_close_argmax   -- per-object 9 x 9 closure,
 *                                                palette argmax, down_s of the
 *                                                closed masks onto the grid
 *   front end (Sec. 3.1)   rs3_seed_from_masks -- seed box of Eq. 1 from
 *                                                pixel masks, down_s
 *
 * Vocabulary.  A *unit* is one (stream, object) pair: it owns one keep-set,
 * one memory bank and one output grid.  A *group* is the set of units that
 * share a query grid Z (the objects of one stream).  The token grid has
 * m x n cells (mn = m*n), row-major, cell i = y*n + x.  D = H*d is the width
 * of a query / key / value row (H heads of dimension d; head h owns columns
 * [h*d, (h+1)*d)).  Masks are given at grid resolution (the down_s of
 * Eq. 1/2/8 already applied), except where rs3_close_argmax and
 * rs3_seed_from_masks take pixel-resolution input and apply it.
 *
 * Conventions for every call.
 *   - Device pointers are owned by the caller; the library never allocates,
 *     frees or retains memory.  Host pointers are read before the call returns.
 *   - Calls are asynchronous on `stream` and never synchronise it, except
 *     rs3_bank_read_meta (documented there).
 *   - Argument errors are returned synchronously (RS3_EINVAL, RS3_EUNSUPPORTED)
 *     and nothing is launched.  A failed launch returns RS3_ECUDA.
 *   - Conditions found on the device (a count above k_max, a bank without
 *     room for a commit, a group id out of range) are latched into the
 *     caller's device word `*status` (first error wins: it is set only while
 *     it holds 0); the affected unit's work is skipped, others proceed.  No
 *     kernel traps and no kernel waits without bound.
 *   - Element rows (z, q, residual, out, K/V) must start on 16-byte
 *     boundaries: every base pointer 16-byte aligned and D * sizeof(elem) a
 *     multiple of 16.  Inputs must be finite.
 *   - bf16 values are stored as IEEE bfloat16 bit patterns (uint16).
 */
#ifndef RS3_H
#define RS3_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Same object as cudaStream_t; NULL is the legacy default stream. */
typedef struct CUstream_st *rs3_stream_t;

typedef enum {
    RS3_OK = 0,
    RS3_EINVAL = 1,        /* bad argument (host) or bad device value (status word) */
    RS3_ECAPACITY = 2,     /* bank or workspace too small */
    RS3_EUNSUPPORTED = 3,  /* valid but not implemented (dtype / head dim / grid size) */
    RS3_ECUDA = 4,         /* a CUDA launch or query failed */
    RS3_EINTERNAL = 5,     /* inconsistent bank metadata */
    RS3_ETIMEOUT = 6       /* a device-side wait gave up (status word only) */
} rs3_status;

typedef enum { RS3_F32 = 0, RS3_BF16 = 1 } rs3_dtype;

/* Hyper-parameters (Algorithm 1: rho = 0.3, r_s = 4, c = 14; D_w = 24 is the
 * SAM2 default of Sec. 5.3; the 5% / 95% fall-through of Sec. 3.2). */
typedef struct {
    double rho;            /* read keep ratio: k_max = floor(rho * mn) (Table 4) */
    int32_t r_s;           /* prior dilation radius, Chebyshev, grid cells (Eq. 1, 2) */
    int32_t c;             /* fallback growth cap (Eq. 4): radius r_s + min(streak, c) */
    int32_t D_w;           /* write keep-set dilation radius (Eq. 8) */
    int32_t union_mode;    /* 1: one prior per group, the union over its units
                              (Eq. 2, P = U_o P_o); 0: each unit selects from
                              its own P_o (per-object banks) */
    double fall_lo;        /* write fall-through when seed coverage < fall_lo ... */
    double fall_hi;        /* ... or > fall_hi (fractions of mn, strict) */
    int32_t fall_through;  /* 1: apply the fall-through in rs3_write_keepset */
    int32_t bbox_mode;     /* 1: dilate the tight box of a non-empty mask
                              (Eq. 1's seed prior); 0: dilate the mask (Eq. 2) */
} rs3_params;

/* Per-unit tracker state of Eq. 4 (device memory, updated by
 * rs3_select_queries): the last non-empty box (inclusive), whether one was
 * ever seen, and the count of consecutive empty masks. */
typedef struct {
    int32_t y0, x0, y1, x1;
    int32_t valid;
    int32_t streak;
} rs3_track;

/* Fills the paper's defaults: rho 0.3, r_s 4, c 14, D_w 24, union_mode 1,
 * fall 0.05 / 0.95 with fall_through 1, bbox_mode 0. */
void rs3_default_params(rs3_params *p);

/* k_max = floor(rho * mn), evaluated in double (Table 4: 1228 at rho 0.3 and
 * mn 4096).  Returns -1 for rho outside [0, 1] or mn < 0. */
int64_t rs3_kmax(double rho, int64_t mn);

const char *rs3_status_string(int code);
int rs3_version(void);

/* ------------------------------------------------------------------------ */
/* Read side: keep-set selection (Sec. 3.1; Eq. 1, 2, 4, 5)                 */
/* ------------------------------------------------------------------------ */

/* Bytes of device workspace rs3_select_queries needs (a group "needed-cell"
 * bitmap, per-unit priors and group energies). */
size_t rs3_select_workspace_bytes(int G, int U, int m, int n);

/*
 * Per unit u (group g = unit_group[u]): builds the prior P_u from the previous
 * frame's mask prev_masks[u] and the tracker track[u] --
 *   mask non-empty: P_u = dilate_{r_s}(mask)   (Eq. 2; bbox_mode: its box, Eq. 1)
 *                   and track <- {bbox(mask), valid 1, streak 0};
 *   mask empty:     streak += 1; if valid, P_u = dilate_{r_s + min(streak, c)}(box)
 *                   (Eq. 4), else P_u is empty --
 * takes P = union of P_v over the units v of group g (union_mode) or P = P_u,
 * ranks the cells of P by the energy e_i = ||z_{g,i}||^2 (Eq. 5) and keeps the
 * k = min(k_max, |P|) best by (energy desc, index asc).
 *
 *   z          device [G][mn][C], dtype; C % 8 == 0, 8 <= C <= 4096
 *   prev_masks device uint8 [U][mn] (nonzero = set)
 *   unit_group device int32 [U], values in [0, G)
 *   track      device rs3_track [U], read and updated
 *   p          host; rho, r_s, c, union_mode, bbox_mode are used
 *   idx        device int32 [U][k_max], k_max = rs3_kmax(p->rho, mn):
 *              row u holds the keep-set in ascending cell order; entries past
 *              count[u] are left unspecified
 *   count      device int32 [U]
 *   workspace  device, >= rs3_select_workspace_bytes(G, U, m, n) bytes,
 *              16-byte aligned; contents are scratch
 *   status     device int32 word (see conventions)
 * The energy is the canonical fp32 sum: 32 partials, partial l takes the
 * 8-channel chunks l, l+32, ... with channels ascending, each step
 * s = fmaf(z, z, s); then s[l] += s[l+w] for w = 16, 8, 4, 2, 1.  Ties go to
 * the lower cell index, so the keep-set is a function of the bits of z.
 * Limits: 1 <= m, n and mn <= 16384; r_s, c >= 0.
 */
rs3_status rs3_select_queries(const void *z, rs3_dtype dtype, int G, int m, int n, int C,
                              const uint8_t *prev_masks, const int32_t *unit_group, int U,
                              rs3_track *track, const rs3_params *p, int32_t *idx,
                              int32_t *count, void *workspace, size_t workspace_bytes,
                              int32_t *status, rs3_stream_t stream);

/*
 * rs3_select_queries for callers that cannot allocate device memory.  The
 * paper has no counterpart: this is a deployment convenience of the library.
 * Some callers have no allocator to ask for the workspace (code running while
 * a stream is captured in the global capture mode, serving loops that must not
 * allocate after start-up, hosts that pass only input and output buffers
 * through a plugin interface); this call instead uses scratch memory compiled
 * into the library: an 8 MiB device array that every GPU loading the library
 * holds until the process exits.  Arguments and results are those of
 * rs3_select_queries without the workspace pair.
 *   - Sizes whose workspace (rs3_select_workspace_bytes(G, U, m, n)) exceeds
 *     8 MiB are rejected with RS3_ECAPACITY; nothing is launched.
 *   - The call allocates nothing (no cudaMalloc / cudaFree, no allocating
 *     library routine).
 *   - The first call on a device looks up the array's device address with
 *     that device current and caches it; make that first call before any
 *     stream capture.  The cache remembers the context the address belongs
 *     to: after a device reset the next call looks the address up again, so
 *     make that call before any capture too.
 *   - All calls on a device share the one array, and it keeps the previous
 *     call's contents (the call clears what must start at zero itself), so
 *     calls whose executions overlap on the GPU (different streams without
 *     ordering between them) race and must not be issued.
 */
rs3_status rs3_select_queries_noalloc(const void *z, rs3_dtype dtype, int G, int m, int n, int C,
                                      const uint8_t *prev_masks, const int32_t *unit_group, int U,
                                      rs3_track *track, const rs3_params *p, int32_t *idx,
                                      int32_t *count, int32_t *status, rs3_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Memory bank (Sec. 3.2; Algorithm 1's sparse write)                        */
/* ------------------------------------------------------------------------ */

/*
 * Host descriptor of a set of U per-unit banks.  Storage per unit is
 * rows_per_unit rows of D elements in k_store and in v_store
 * ([U][rows_per_unit][D]):
 *   rows [0, pinned_cap)                 pinned conditioning frames, packed
 *                                        in commit order (pinned_cap = n_cond*mn)
 *   rows [pinned_cap, +ring_cap)         ring of recent frames: logical ring
 *                                        position p lives at row
 *                                        pinned_cap + (p mod ring_cap)
 *   rows [pinned_cap+ring_cap, +n_ptr)   pointer rows (rs3_bank_set_pointers)
 * A unit's bank, in logical order, is: its pinned rows, its ring frames
 * oldest first, its pointer rows.  `meta` is device memory of meta_bytes
 * (rs3_bank_layout) holding the per-unit counters and frame table.
 */
typedef struct {
    int32_t U, H, d, D;
    int32_t dtype;          /* rs3_dtype */
    int32_t mn;             /* grid cells: the longest frame a commit can add */
    int32_t n_cond;         /* pinned conditioning frames per unit */
    int32_t window;         /* ring frames kept (oldest evicted first); -1 = unbounded */
    int32_t max_frames;     /* frame-table entries per unit (== window when windowed) */
    int32_t n_ptr;          /* pointer rows per unit */
    int64_t pinned_cap, ring_cap, rows_per_unit;
    int64_t meta_stride;    /* bytes of meta per unit */
    void *k_store;
    void *v_store;
    void *meta;
    uint32_t magic;         /* set by rs3_bank_init */
    uint32_t reserved;
} rs3_bank;

/* Sizes for a bank: rows per unit of each store and bytes of meta.
 * window > 0 requires ring_cap_rows >= window * mn (the ring then always holds
 * the window); window == -1 (unbounded) needs ring_cap_rows >= 0 and
 * max_frames >= 1.  Returns RS3_EINVAL on an inconsistent layout and
 * RS3_EUNSUPPORTED for mn > 16384 or U > 65535. */
rs3_status rs3_bank_layout(int U, int H, int d, rs3_dtype dtype, int mn, int n_cond, int window,
                           int64_t ring_cap_rows, int max_frames, int n_ptr,
                           int64_t *rows_per_unit, size_t *meta_bytes);

/* Fills *bank and clears `meta`, `k_store` and `v_store` on `stream` (the
 * banks start empty; storage rows never written read as zeros).
 * k_store / v_store: device [U][rows_per_unit][H*d]; meta: device, meta_bytes. */
rs3_status rs3_bank_init(rs3_bank *bank, int U, int H, int d, rs3_dtype dtype, int mn, int n_cond,
                         int window, int64_t ring_cap_rows, int max_frames, int n_ptr,
                         void *k_store, void *v_store, void *meta, rs3_stream_t stream);

/*
 * Write-pruned commit (Sec. 3.2 and Algorithm 1's sparse write): for every
 * unit u, the rows k_new[u][i], v_new[u][i] with keep_mask[u][i] != 0 are
 * appended, in ascending i, as one new frame of the unit's bank.
 *   k_new, v_new  device [U][mn][D] in the bank's dtype (bank->mn cells)
 *   keep_mask     device uint8 [U][mn], or NULL to keep every row
 *   is_cond       1: the frame is a pinned conditioning frame; 0: a ring frame.
 * A ring commit first evicts the oldest ring frame when `window` frames are
 * held.  A commit that does not fit (all pinned slots used, ring full of an
 * unbounded bank, frame table full) is dropped whole for that unit and latches
 * RS3_ECAPACITY into *status; other units proceed.
 */
rs3_status rs3_bank_commit(const rs3_bank *bank, const void *k_new, const void *v_new,
                           const uint8_t *keep_mask, int is_cond, int32_t *status,
                           rs3_stream_t stream);

/* rs3_bank_commit with RoPE on the key side (Sec. 3.1, Eq. 7: keys are
 * rotated by their own grid position, as the queries are by theirs).  Every
 * kept key row k_new[u][i] is stored rotated by the (cos, sin) of its own
 * cell i: in each head, elements (2p, 2p+1) become
 *   (k0 cos - k1 sin, k0 sin + k1 cos),  (cos, sin) = rope_cos_sin[i][p]
 * computed in fp32 and rounded once to the bank dtype (nearest-even for
 * bf16).  Values are stored as given.  A rotation is linear in the key and
 * depends only on the key's own cell, so storing rotated keys and rotating
 * them at every read give the same attention; the commit does it once per
 * key.  Pointer rows (rs3_bank_set_pointers) are stored unrotated: object
 * pointers carry no grid position.
 * rope_cos_sin: device fp32 [mn][d/2][2], the same table rs3_memory_readout
 * takes for the queries, 16-byte aligned.  Errors as rs3_bank_commit, plus
 * RS3_EINVAL for a NULL or misaligned table and RS3_EUNSUPPORTED when d is
 * not a multiple of 8. */
rs3_status rs3_bank_commit_rope(const rs3_bank *bank, const void *k_new, const void *v_new,
                                const uint8_t *keep_mask, int is_cond, const float *rope_cos_sin,
                                int32_t *status, rs3_stream_t stream);

/* Replaces every unit's pointer rows with k_ptr[u], v_ptr[u] (device
 * [U][n_ptr][D]).  RS3_EINVAL when the bank has n_ptr == 0. */
rs3_status rs3_bank_set_pointers(const rs3_bank *bank, const void *k_ptr, const void *v_ptr,
                                 int32_t *status, rs3_stream_t stream);

/* Empties unit `unit` (all units when unit == -1): counters only, no data
 * movement. */
rs3_status rs3_bank_reset(const rs3_bank *bank, int unit, rs3_stream_t stream);

/* Copies the per-unit counters to host memory and SYNCHRONISES `stream`
 * (tests and tools only).  host_out: int64 [U][8] =
 * {head, tail, cond_len, n_frames, oldest, n_cond_frames, ptr_len, length}
 * where length = cond_len + (tail - head) + ptr_len rows.  When frames_out is
 * not NULL it receives int64 [U][max_frames][2] (logical offset, length) of
 * the ring frames, oldest first; unused entries are -1. */
rs3_status rs3_bank_read_meta(const rs3_bank *bank, int64_t *host_out, int64_t *frames_out,
                              rs3_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Read side: pruned memory readout (Sec. 3.1; Eq. 6, Eq. 7)                 */
/* ------------------------------------------------------------------------ */

/* Bytes of device workspace rs3_memory_readout needs for these sizes (the
 * work list, and the split-KV partial results of long banks). */
size_t rs3_readout_workspace_bytes(int U, int H, int d, int k_max, rs3_dtype dtype);

/*
 * For every unit u (group g = unit_group[u]) and kept query j < count[u] at
 * cell i = idx[u][j], for every head h:
 *   q~    = q[g][i][h*d : (h+1)*d], rotated pairwise (2p, 2p+1) by
 *           (cos, sin) = rope[i][p] when rope != NULL        (Eq. 7)
 *   A     = softmax(q~ K_h^T * scale) V_h over the unit's whole bank
 *           (pinned frames, ring frames, pointer rows)      (Eq. 6)
 *   out[u][i][h*d : (h+1)*d] = residual[u][i][...] + A, rounded once to dtype
 * and every other cell i of out[u] equals residual[u][i] bit for bit (zeros
 * when residual is NULL, which is Eq. 6's literal scatter S_K).  An empty bank
 * reads A = 0.
 *   q         device [G][mn][H*d], dtype == bank dtype (q = the grid's query
 *             projection; the benchmark uses q = Z)
 *   unit_group, idx, count  as produced for rs3_select_queries
 *   k_max     row stride of idx; count[u] > k_max latches RS3_EINVAL
 *   rope      device fp32 [mn][d/2][2] or NULL
 *   residual  device [U][mn][H*d], NULL, or == out (in place: only the kept
 *             rows are written)
 *   out       device [U][mn][H*d]
 *   scale     softmax scale; 0 selects 1/sqrt(d) (Eq. 6's 1/sqrt(C_k) per head)
 *   workspace device, >= rs3_readout_workspace_bytes(...), 16-byte aligned
 * bf16: tensor-core path for d in {64, 128, 256}, fp32 accumulation.  fp32:
 * CUDA-core FFMA path for d % 16 == 0, d <= 256.
 * Limits: U <= 4096, mn <= 16384; the work list holds fewer than 2^21
 * entries (U * H * ceil(k_max / BM) plus one per SM, BM = 128 on the bf16
 * path and 32 on the fp32 path), else RS3_EUNSUPPORTED.
 */
rs3_status rs3_memory_readout(const void *q, rs3_dtype dtype, int G, int mn, int H, int d,
                              const int32_t *unit_group, const int32_t *idx,
                              const int32_t *count, int k_max, const rs3_bank *bank,
                              const float *rope, const void *residual, void *out, float scale,
                              void *workspace, size_t workspace_bytes, int32_t *status,
                              rs3_stream_t stream);

/*
 * Time limit of every wait inside the readout kernels launched after this
 * call, in nanoseconds of the GPU's global timer (default 1000000000, one
 * second; 0 gives up at the first wait whose condition does not already
 * hold).  A kernel whose wait runs out stops issuing work, lets its copies
 * and matrix operations in flight complete, frees its tensor memory, latches
 * RS3_ETIMEOUT into the call's status word and returns; the rows it did not
 * finish hold unspecified values.  The setting is process-wide; it exists so
 * that the timeout path can be exercised on purpose.  No paper counterpart.
 */
void rs3_set_wait_limit_ns(uint64_t ns);
uint64_t rs3_get_wait_limit_ns(void);

/*
 * The same readout in two phases, with the arguments of rs3_memory_readout
 * (the same values must be passed to both calls of one readout):
 *   rs3_memory_readout_attend   the attention over the bank: writes the rows
 *                               of unsplit work directly and leaves split-KV
 *                               partial results in `workspace`;
 *   rs3_memory_readout_merge    merges those partials and writes their rows.
 * attend then merge on one stream is exactly rs3_memory_readout (same kernels,
 * same results bit for bit).  The merge reads only the workspace, idx, count,
 * unit_group, residual and out, never the bank, so once attend has completed
 * a commit to the bank (Eq. 8, the write side of the same frame) may run on
 * another stream concurrently with the merge.  Ordering is the caller's:
 * merge after attend (e.g. through an event), the next attend or any other
 * use of the same workspace after merge, and readers of `out` after merge.
 */
rs3_status rs3_memory_readout_attend(const void *q, rs3_dtype dtype, int G, int mn, int H, int d,
                                     const int32_t *unit_group, const int32_t *idx,
                                     const int32_t *count, int k_max, const rs3_bank *bank,
                                     const float *rope, const void *residual, void *out, float scale,
                                     void *workspace, size_t workspace_bytes, int32_t *status,
                                     rs3_stream_t stream);
rs3_status rs3_memory_readout_merge(const void *q, rs3_dtype dtype, int G, int mn, int H, int d,
                                    const int32_t *unit_group, const int32_t *idx,
                                    const int32_t *count, int k_max, const rs3_bank *bank,
                                    const float *rope, const void *residual, void *out, float scale,
                                    void *workspace, size_t workspace_bytes, int32_t *status,
                                    rs3_stream_t stream);

/*
 * rs3_memory_readout_attend split in its two launches, with the same
 * arguments (Sec. 3.1, Eq. 6):
 *   rs3_memory_readout_plan  the pass-through of unselected cells (out of
 *                            place only) and the work list in `workspace`:
 *                            the bank's row ranges from its counters and the
 *                            split of the work over the SMs;
 *   rs3_memory_readout_run   the attention kernel over that work list.
 * plan then run on one stream is exactly rs3_memory_readout_attend.  run
 * reads the bank's rows but not its counters, so the work list describes the
 * bank as it was when plan ran; ordering is the caller's (run after plan, and
 * no commit to the bank between them).  Separate calls let a caller time or
 * schedule the attention kernel on its own.
 */
rs3_status rs3_memory_readout_plan(const void *q, rs3_dtype dtype, int G, int mn, int H, int d,
                                   const int32_t *unit_group, const int32_t *idx,
                                   const int32_t *count, int k_max, const rs3_bank *bank,
                                   const float *rope, const void *residual, void *out, float scale,
                                   void *workspace, size_t workspace_bytes, int32_t *status,
                                   rs3_stream_t stream);
rs3_status rs3_memory_readout_run(const void *q, rs3_dtype dtype, int G, int mn, int H, int d,
                                  const int32_t *unit_group, const int32_t *idx,
                                  const int32_t *count, int k_max, const rs3_bank *bank,
                                  const float *rope, const void *residual, void *out, float scale,
                                  void *workspace, size_t workspace_bytes, int32_t *status,
                                  rs3_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Write side: keep-set (Sec. 3.2; Eq. 8)                                    */
/* ------------------------------------------------------------------------ */

/*
 * K_w for every unit: S = seed_masks[u] (or, in union_mode, the union of the
 * seeds of u's group); if p->fall_through and |S|/mn > fall_hi or < fall_lo,
 * K_w is the whole grid, else K_w = dilate_{D_w}(S) (Chebyshev radius D_w).
 * The caller evaluates it at each object's first-appearance frame and keeps
 * the result fixed, which gives the bank a constant per-frame stride.
 *   seed_masks device uint8 [U][mn]; unit_group device int32 [U];
 *   kw_out     device uint8 [U][mn] (0 / 1).  mn <= 16384.
 */
rs3_status rs3_write_keepset(const uint8_t *seed_masks, const int32_t *unit_group, int U, int m,
                             int n, const rs3_params *p, uint8_t *kw_out, int32_t *status,
                             rs3_stream_t stream);

/* ------------------------------------------------------------------------ */
/* Decoder side (Sec. 3.3) and the pixel-space front end (Sec. 3.1)          */
/* ------------------------------------------------------------------------ */

/*
 * Per-frame post-processing of the mask decoder's output (Sec. 3.3,
 * Algorithm 1 after the decoder): each object's binary mask (logit > 0) is
 * closed with the (2*radius+1)^2 square -- a dilation, then an erosion; the
 * paper uses radius 4, the 9 x 9 element -- and then every pixel goes to the
 * object with the largest logit among the objects of its stream whose closed
 * mask holds it (the palette mask; 0 = background; equal logits go to the
 * object listed first).  The closure treats an object as a set of the
 * unbounded plane with nothing set outside the image, so it is extensive and
 * idempotent, fills holes and bridges gaps of at most 2*radius pixels, and
 * neither grows an object out to the image border nor erodes one touching it.
 *   logits      device fp32 [U][h][w], decoder mask logits at the decoder's
 *               resolution (finite values)
 *   group_start device int32 [G+1]: the objects of stream g are the units
 *               [group_start[g], group_start[g+1]), at most 255 of them; a
 *               stream whose range is not inside [0, U] or holds more than 255
 *               objects latches RS3_EINVAL into *status and is skipped
 *   palette     device uint8 [G][h][w] or NULL: 0, or 1 + the object's index
 *               within its stream
 *   closed      device uint8 [U][h][w] or NULL: each object's closed mask (0/1),
 *               the per-object masks M_t|o that Algorithm 1's tracker reads
 *   grid_masks  device uint8 [U][h/s][w/s] or NULL: down_s of each closed mask
 *               (cell (i, j) takes pixel (i*s, j*s), Sec. 3.1), the previous-
 *               frame masks that rs3_select_queries consumes next frame
 *   status      device int32 word (see conventions)
 * Limits: w a multiple of 32, 0 <= radius <= 8, G <= 65535; h and w multiples
 * of s when grid_masks is given.
 */
rs3_status rs3_close_argmax(const float *logits, const int32_t *group_start, int G, int U, int h,
                            int w, int radius, int s, uint8_t *palette, uint8_t *closed,
                            uint8_t *grid_masks, int32_t *status, rs3_stream_t stream);

/*
 * Seed of every object from its pixel-resolution mask (Sec. 3.1, Eq. 1): the
 * tight pixel box of the set pixels, each corner divided by the encoder
 * stride s and rounded down, becomes the unit's tracker state ({y0, x0, y1,
 * x1} on the grid, valid 1, streak 0; an empty mask gives all zeros), so the
 * first rs3_select_queries call dilates down_s of the seed box: by r_s when
 * box_masks is passed as the previous mask (Eq. 1), or by r_s + 1 when the
 * previous mask is empty (Eq. 4's fallback, whose streak counter is already 1
 * on that first empty frame).
 *   masks      device uint8 [U][h][w] (nonzero = set), 16-byte aligned
 *   track      device rs3_track [U], written
 *   grid_masks device uint8 [U][h/s][w/s] or NULL: down_s of the mask (cell
 *              (i, j) takes pixel (i*s, j*s))
 *   box_masks  device uint8 [U][h/s][w/s] or NULL: the projected box, filled
 * Limits: w a multiple of 16; h and w multiples of s; U <= 65535.
 */
rs3_status rs3_seed_from_masks(const uint8_t *masks, int U, int h, int w, int s, rs3_track *track,
                               uint8_t *grid_masks, uint8_t *box_masks, rs3_stream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* RS3_H */
