// rs3_readout_tc.cu -- tensor-core readout for bf16 (Sec. 3.1, Eq. 6 and
// Eq. 7) on sm_103a: tcgen05.mma with fp32 accumulators in TMEM, K/V tiles
// staged by TMA (cp.async.bulk.tensor, 128-byte swizzle), online softmax in
// the log2 domain.
//
// One persistent CTA per SM runs its slice of the stream-K plan: work items
// (unit, head, 128-query tile, range of BN-key tiles).  Warps:
//   warp 0      K producer: TMA of the key tile (d/64 boxes of BN rows x 64)
//   warp 2      V producer: TMA of the value tile
//   warp 1      TMEM allocation; lane 0 issues S_j = Q K_j^T (M 128, N BN,
//               K d; A = Q in TMEM, B = K tile, K-major) into one of two TMEM
//               buffers as soon as the softmax has read the one before
//   warp 3      lane 0 issues O += P_j V_j (M 128, N d, K BN; A = P_j in
//               shared memory, B = V tile, MN-major) once P_j is written.  The
//               two issuers share no operand, so each one's waits overlap the
//               other's MMAs.
//   warp 3      lanes 1..31: L2 prefetch of the query rows of later items
//   warps 4..   2 x 4 softmax warps; warps w and w + 4 own the same TMEM lane
//               quarter (rows 32 (w % 4) + lane) and split the columns.  Per
//               item each thread loads its slice of the kept query row,
//               rotates it by the RoPE table of its own cell (Eq. 7) and
//               writes it to TMEM as bf16 pairs; per tile it reads its slice
//               of S_j, takes the exps against a running reference that moves
//               only when the row max grows by more than 2^8 (O is then
//               rescaled in TMEM), and writes P_j to shared memory (three
//               buffers).  The slices of a row exchange their maxima through
//               shared memory at a named barrier that also ANDs their wait
//               results.  Epilogue: O / l + residual, or split-KV partials.
// TMEM (512 columns): O in [0, d), S_0 / S_1 from S_COL, Q at Q_COL.
// Shapes: d = 256 and d = 128 use 64-key tiles, d = 64 128-key tiles; K and V
// rings fill what shared memory leaves after the three P buffers.
// Every mbarrier wait is bounded (a launch parameter, 1 s of %globaltimer by
// default): on expiry the CTA
// raises an abort flag, drains its copies and MMAs, frees TMEM and the launch
// latches RS3_ETIMEOUT.
#include "rs3_readout_common.cuh"
#include "rs3_tc_ptx.cuh"

#include <cudaTypedefs.h>

namespace tc {

constexpr int BM = 128;
constexpr uint32_t TMEM_COLS = 512;

template <int DH>
struct Cfg {
    static constexpr int BN = DH == 64 ? 128 : 64;           // keys per tile
    static constexpr int KVBYTES = BN * DH * 2;              // one K (or V) stage
    static constexpr int PBYTES = BM * BN * 2;               // one P buffer
    static constexpr int NPB = 3;                            // P buffers (and PV barriers)
    static constexpr int NSPLIT = 2;                         // softmax warps per TMEM lane quarter
    // K stages, V stages: what the 227 KB of shared memory leave after the P
    // buffers, the row exchange, the barriers and the alignment slack
    static constexpr int NKV = (232448 - 1024 - 16 - 64 * 8 - 3 * NSPLIT * BM * 4 - NPB * PBYTES) / KVBYTES;
    static constexpr int KSTK = (NKV + 1) / 2, KSTV = NKV / 2;
    static constexpr int NTHREADS = 128 + 128 * NSPLIT;
    static constexpr int SCOLS = BN / NSPLIT;                // S columns of one softmax warp
    static constexpr int PCOLS = SCOLS / 2;                  // its P pairs
    static constexpr int OCOLS = DH / NSPLIT;                // its O columns
    static constexpr int QCOLS = DH / 2 / NSPLIT;            // its Q columns (bf16 pairs)
    static constexpr uint32_t S_COL = 256;                   // S_0 at S_COL, S_1 at S_COL + BN
    static constexpr uint32_t Q_COL = DH == 256 ? 384 : DH;  // d/2 columns of bf16 pairs
    static constexpr int OFF_K = 0;
    static constexpr int OFF_V = OFF_K + KSTK * KVBYTES;
    static constexpr int OFF_P = OFF_V + KSTV * KVBYTES;
    static constexpr int OFF_RED = OFF_P + NPB * PBYTES;     // float [3][NSPLIT][BM]
    static constexpr int OFF_BAR = OFF_RED + 3 * NSPLIT * BM * 4;
    static constexpr int NBAR = 2 * KSTK + 2 * KSTV + 6 + 2 * NPB;
    static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
    static constexpr int SMEM = OFF_MISC + 16 + 1024;        // + alignment slack
    // barrier indices
    static constexpr int B_KFULL = 0, B_KEMPTY = KSTK, B_VFULL = 2 * KSTK, B_VEMPTY = 2 * KSTK + KSTV;
    // SFULL / SFREE per S buffer; PFULL / PVDONE per P buffer: the softmax
    // writes P_{t+3} only after PV_t, so no barrier runs two phases ahead of
    // its waiter
    static constexpr int B_SFULL = 2 * KSTK + 2 * KSTV, B_SFREE = B_SFULL + 2, B_QFULL = B_SFULL + 4;
    static constexpr int B_DRAIN = B_SFULL + 5, B_PFULL = B_SFULL + 6, B_PVDONE = B_PFULL + NPB;
    static_assert(S_COL + 2 * BN <= TMEM_COLS && Q_COL + DH / 2 <= TMEM_COLS, "TMEM budget");
    static_assert(Q_COL >= (uint32_t)DH && (Q_COL + DH / 2 <= S_COL || Q_COL >= S_COL + 2 * BN), "TMEM overlap");
    static_assert(SCOLS % 8 == 0 && PCOLS % 8 == 0 && QCOLS % 8 == 0 && OCOLS % 16 == 0, "warp slices");
    static_assert(KSTK >= 2 && KSTV >= 2 && NBAR <= 64, "K/V stages");
    static_assert(4 * NSPLIT * 32 * 36 * 4 <= NPB * PBYTES, "epilogue staging fits in the P ring");
    static_assert(OCOLS % 32 == 0, "epilogue stages 32 columns at a time");
};
static_assert(Cfg<256>::SMEM <= 232448 && Cfg<128>::SMEM <= 232448 && Cfg<64>::SMEM <= 232448,
              "shared memory budget");

// Softmax pieces of one row's S tile (raw scores as fp32 bits).
template <int N>
__device__ __forceinline__ float row_max(const uint32_t (&sr)[N], int nv, bool full)
{
    float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
    for (int c = 0; c < N; c += 2) {
        m0 = fmaxf(m0, (full || c < nv) ? __uint_as_float(sr[c]) : -INFINITY);
        m1 = fmaxf(m1, (full || c + 1 < nv) ? __uint_as_float(sr[c + 1]) : -INFINITY);
    }
    return fmaxf(m0, m1);
}

// p = 2^(s * sc - ref) of one slice's scores (raw fp32 bits), as bf16 pairs;
// returns the sum of the p.  The scale-and-shift and the sums run on packed
// fp32 pairs (f32x2), the exps on the SFU; four partial sums keep the adds
// independent.  Columns at or past nv (invalid keys) give p = 0.
template <int N>
__device__ __forceinline__ float row_exp(const uint32_t (&sr)[N], uint32_t (&pk)[N / 2], float sc, float ref,
                                         int nv, bool full)
{
    const uint64_t sc2 = f2pack(sc, sc), nref2 = f2pack(-ref, -ref);
    uint64_t acc[4] = {0ull, 0ull, 0ull, 0ull};
#pragma unroll
    for (int c = 0; c < N / 2; ++c) {
        float x0, x1;
        f2unpack(fma2(f2pack(__uint_as_float(sr[2 * c]), __uint_as_float(sr[2 * c + 1])), sc2, nref2), x0, x1);
        float p0 = ex2_approx(x0), p1 = ex2_approx(x1);
        if (!full) {
            p0 = 2 * c < nv ? p0 : 0.f;
            p1 = 2 * c + 1 < nv ? p1 : 0.f;
        }
        acc[c & 3] = add2(acc[c & 3], f2pack(p0, p1));
        pk[c] = pack_bf16x2(p0, p1);
    }
    float a0, a1, a2, a3, a4, a5, a6, a7;
    f2unpack(acc[0], a0, a1);
    f2unpack(acc[1], a2, a3);
    f2unpack(acc[2], a4, a5);
    f2unpack(acc[3], a6, a7);
    return ((a0 + a1) + (a2 + a3)) + ((a4 + a5) + (a6 + a7));
}

// NW consecutive bf16 pairs of one thread's kept query row -> its TMEM lane,
// columns [tq, tq + NW) (element 2i in the low half).  With a RoPE table,
// pair i is rotated by the (cos, sin) at rope[2i], rope[2i + 1] of the row's
// own cell (Eq. 7).  qrow == nullptr writes zeros (rows past the kept count).
template <int NW>
__device__ __forceinline__ void q_pairs_to_tmem(const uint16_t *qrow, const float *rope, uint32_t tq)
{
    uint32_t w[NW];
    if (qrow) {
#pragma unroll
        for (int i = 0; i < NW / 4; ++i) {
            const uint4 v = __ldg(reinterpret_cast<const uint4 *>(qrow) + i);
            w[4 * i] = v.x; w[4 * i + 1] = v.y; w[4 * i + 2] = v.z; w[4 * i + 3] = v.w;
        }
        if (rope) {
#pragma unroll
            for (int p = 0; p < NW; p += 2) {
                const float4 f = __ldg(reinterpret_cast<const float4 *>(rope) + p / 2);
                const float x0 = __uint_as_float(w[p] << 16), x1 = __uint_as_float(w[p] & 0xffff0000u);
                const float y0 = __uint_as_float(w[p + 1] << 16), y1 = __uint_as_float(w[p + 1] & 0xffff0000u);
                w[p] = pack_bf16x2(x0 * f.x - x1 * f.y, x0 * f.y + x1 * f.x);
                w[p + 1] = pack_bf16x2(y0 * f.z - y1 * f.w, y0 * f.w + y1 * f.z);
            }
        }
    } else {
#pragma unroll
        for (int i = 0; i < NW; ++i) w[i] = 0u;
    }
    tmem_st_cols<NW>(tq, w);
}

template <int DH>
__global__ void __launch_bounds__(Cfg<DH>::NTHREADS, 1)
k_readout_tc(const ReadoutArgs a, const __grid_constant__ CUtensorMap tmk,
             const __grid_constant__ CUtensorMap tmv)
{
    using C = Cfg<DH>;
    constexpr int KSTK = C::KSTK, KSTV = C::KSTV, BN = C::BN;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *gbase = smem_raw + (base - raw);
    const uint32_t sK = base + C::OFF_K, sV = base + C::OFF_V, sP = base + C::OFF_P;
    const uint32_t bars = base + C::OFF_BAR;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(gbase + C::OFF_MISC);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(gbase + C::OFF_MISC + 8);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#define BAR(i) (bars + 8u * (uint32_t)(i))

    if (threadIdx.x == 0) {
        for (int s = 0; s < KSTK; ++s) {
            mbar_init(BAR(C::B_KFULL + s), 1);
            mbar_init(BAR(C::B_KEMPTY + s), 1);
        }
        for (int s = 0; s < KSTV; ++s) {
            mbar_init(BAR(C::B_VFULL + s), 1);
            mbar_init(BAR(C::B_VEMPTY + s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(BAR(C::B_SFULL + b), 1);
            mbar_init(BAR(C::B_SFREE + b), 4 * C::NSPLIT); // one arrival per softmax warp
        }
        for (int b = 0; b < C::NPB; ++b) {
            mbar_init(BAR(C::B_PFULL + b), 4 * C::NSPLIT);
            mbar_init(BAR(C::B_PVDONE + b), 1);
        }
        mbar_init(BAR(C::B_QFULL), 4 * C::NSPLIT);
        mbar_init(BAR(C::B_DRAIN), 2);                    // both MMA issuers
        *abort_flag = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        fence_proxy_async();
    }
    if (warp == 1) {
        asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;"
                     ::"r"(smem_u32(tmem_slot)), "r"(TMEM_COLS) : "memory");
        asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    }
    if (threadIdx.x == 64) {
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmk)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmv)) : "memory");
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = *tmem_slot;
    const uint64_t wait_ns = a.wait_ns;
    // the set-up above touches no global memory; the plan is read after the
    // previous kernel of the stream has completed
    pdl_wait();
    // this CTA's slice of the stream-K plan
    const int it_begin = a.cta_items[2 * blockIdx.x], it_end = a.cta_items[2 * blockIdx.x + 1];

    if ((warp == 0 || warp == 2) && lane == 0) {
        // ------------------------------------------------------------------
        // TMA producers (warp 0: keys, warp 2: values)
        // ------------------------------------------------------------------
        const bool is_k = warp == 0;
        const CUtensorMap *map = is_k ? &tmk : &tmv;
        const uint32_t dst0 = is_k ? sK : sV;
        const int b_full = is_k ? C::B_KFULL : C::B_VFULL;
        const int b_empty = is_k ? C::B_KEMPTY : C::B_VEMPTY;
        const uint32_t nst = is_k ? (uint32_t)KSTK : (uint32_t)KSTV;
        uint32_t cnt = 0;
        for (int it = it_begin; it < it_end && !*abort_flag; ++it) {
            const WorkItem w = a.items[it];
            const RangeSet *rs = a.ranges + w.u;
            for (int t = w.tile_begin; t < w.tile_end; ++t, ++cnt) {
                const uint32_t st = cnt % nst, ph = (cnt / nst) & 1u;
                if (!mbar_wait(BAR(b_empty + st), ph ^ 1u, abort_flag, wait_ns)) goto producer_done;
                int64_t row0;
                int nvalid;
                tile_rows(rs, t, BN, row0, nvalid);
                const int y = (int)((int64_t)w.u * a.rows_per_unit + row0);
                mbar_expect_tx(BAR(b_full + st), (uint32_t)C::KVBYTES);
#pragma unroll
                for (int c = 0; c < DH / 64; ++c)
                    tma_load_2d(dst0 + st * C::KVBYTES + c * (BN * 128), map, BAR(b_full + st),
                                w.h * DH + c * 64, y);
            }
        }
    producer_done:
        // let every copy this thread issued land before the CTA can exit
        for (uint32_t k = (cnt > nst ? cnt - nst : 0); k < cnt; ++k)
            mbar_drain(BAR(b_full + k % nst), (k / nst) & 1u);
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------------------------
        // S issuer: S_t = Q K_t^T into TMEM buffer t & 1, once the softmax
        // has read S_{t-2}; runs up to two tiles ahead of the softmax
        // ------------------------------------------------------------------
        constexpr uint32_t ID_S = idesc_bf16(BM, BN, false);
        // descriptors built once; a k-step only adds its byte offset / 16 to the
        // start-address field (every address stays below 256 KB, so the 14-bit
        // field cannot carry)
        const uint64_t dk0 = desc_sw128(sK, 16, 1024);
        constexpr uint32_t STAGE16 = C::KVBYTES >> 4;
        uint32_t tcnt = 0, icnt = 0;
        bool ok = true;
        for (int it = it_begin; it < it_end && ok; ++it) {
            const WorkItem w = a.items[it];
            const int n = w.tile_end - w.tile_begin;
            if (n <= 0) continue;
            if (!mbar_wait(BAR(C::B_QFULL), icnt & 1u, abort_flag, wait_ns)) { ok = false; break; }
            ++icnt;
            for (int j = 0; j < n; ++j) {
                const uint32_t t = tcnt + (uint32_t)j, st = t % KSTK, b = t & 1u;
                if (!mbar_wait(BAR(C::B_SFREE + b), ((t >> 1) & 1u) ^ 1u, abort_flag, wait_ns)) { ok = false; break; }
                if (!mbar_wait(BAR(C::B_KFULL + st), (t / KSTK) & 1u, abort_flag, wait_ns)) { ok = false; break; }
                tc_fence_after();
                const uint64_t dks = dk0 + st * STAGE16;
                const uint32_t dst = tmem + C::S_COL + (uint32_t)BN * b;
#pragma unroll
                for (int kk = 0; kk < DH / 16; ++kk) {
                    const uint32_t offk = (uint32_t)((kk >> 2) * (BN * 128) + (kk & 3) * 32);
                    tc_mma_ts(dst, tmem + C::Q_COL + 8u * kk, dks + (offk >> 4), ID_S, kk > 0 ? 1u : 0u);
                }
                tc_commit(BAR(C::B_SFULL + b));
                tc_commit(BAR(C::B_KEMPTY + st));
            }
            tcnt += (uint32_t)n;
        }
        // every MMA issued by this thread completes before TMEM is released
        tc_commit(BAR(C::B_DRAIN));
        mbar_drain(BAR(C::B_DRAIN), 0);
    } else if (warp == 3 && lane == 0) {
        // ------------------------------------------------------------------
        // PV issuer: O += P_t V_t once the softmax has written P_t; its own
        // thread, so its waits overlap the S issue and the other way round
        // ------------------------------------------------------------------
        constexpr uint32_t ID_PV = idesc_bf16(BM, DH, true);
        const uint64_t dv0 = desc_sw128(sV, BN * 128, 1024), dp0 = desc_sw128(sP, 16, 1024);
        constexpr uint32_t STAGE16 = C::KVBYTES >> 4, PBUF16 = C::PBYTES >> 4;
        uint32_t tcnt = 0;
        bool ok = true;
        for (int it = it_begin; it < it_end && ok; ++it) {
            const WorkItem w = a.items[it];
            const int n = w.tile_end - w.tile_begin;
            if (n <= 0) continue;
            for (int j = 0; j < n; ++j) {
                const uint32_t tj = tcnt + (uint32_t)j, pb = tj % C::NPB, st = tj % KSTV;
                if (!mbar_wait(BAR(C::B_PFULL + pb), (tj / C::NPB) & 1u, abort_flag, wait_ns)) { ok = false; break; }
                if (!mbar_wait(BAR(C::B_VFULL + st), (tj / KSTV) & 1u, abort_flag, wait_ns)) { ok = false; break; }
                tc_fence_after();
                const uint64_t dvs = dv0 + st * STAGE16, dps = dp0 + pb * PBUF16;
#pragma unroll
                for (int kk = 0; kk < BN / 16; ++kk) {
                    const uint32_t offp = (uint32_t)((kk >> 2) * (BM * 128) + (kk & 3) * 32);
                    tc_mma(tmem, dps + (offp >> 4), dvs + (uint32_t)((kk * 2048) >> 4), ID_PV,
                           (j > 0 || kk > 0) ? 1u : 0u);
                }
                tc_commit(BAR(C::B_PVDONE + pb));
                tc_commit(BAR(C::B_VEMPTY + st));
            }
            tcnt += (uint32_t)n;
        }
        tc_commit(BAR(C::B_DRAIN));
        mbar_drain(BAR(C::B_DRAIN), 0);
    } else if (warp == 3) {
        // ------------------------------------------------------------------
        // lanes 1..31: L2 prefetch of the kept query rows (and their RoPE
        // rows) of this CTA's later items, so their loads do not wait on DRAM
        // ------------------------------------------------------------------
        for (int it = it_begin + 1; it < it_end && !*abort_flag; ++it) {
            const WorkItem w = a.items[it];
            if (w.tile_end <= w.tile_begin) continue;
            const int cnt = __ldg(&a.ranges[w.u].cnt);
            const int gq = a.unit_group[w.u];
            for (int rr = lane - 1; rr < BM && w.qt * BM + rr < cnt; rr += 31) {
                int cell = a.idx[(int64_t)w.u * a.k_max + w.qt * BM + rr];
                cell = (cell < 0 || cell >= a.mn) ? 0 : cell;
                const char *qr = reinterpret_cast<const char *>(static_cast<const uint16_t *>(a.q) +
                                                                ((int64_t)gq * a.mn + cell) * a.D + w.h * DH);
#pragma unroll
                for (int l = 0; l < 2 * DH; l += 128) prefetch_l2(qr + l);
                if (a.rope) {
                    const char *fr = reinterpret_cast<const char *>(a.rope + (int64_t)cell * DH);
#pragma unroll
                    for (int l = 0; l < 4 * DH; l += 128) prefetch_l2(fr + l);
                }
            }
        }
    } else if (warp >= 4) {
        // ------------------------------------------------------------------
        // query rows, softmax / correction, epilogue.  NSPLIT warps share a
        // TMEM lane quarter (the same 32 rows, thread = row r); warp slice h
        // owns columns [h SCOLS, (h+1) SCOLS) of S, the matching P pairs,
        // O columns [h OCOLS, (h+1) OCOLS) and Q pairs [h QCOLS, (h+1) QCOLS).
        // The slices of a row agree on the softmax reference through a named
        // barrier per tile that also ANDs their wait results, so a timeout
        // makes all of them leave together.
        // ------------------------------------------------------------------
        constexpr int NSPLIT = C::NSPLIT, SCOLS = C::SCOLS, PCOLS = C::PCOLS, OCOLS = C::OCOLS,
                      QCOLS = C::QCOLS;
        const int q4 = warp & 3, h = (warp - 4) >> 2;
        const int r = 32 * q4 + lane;                 // query row of the tile
        const uint32_t tl = tmem + ((uint32_t)(32 * q4) << 16);
        const uint32_t bar_id = 1u + (uint32_t)q4, bar_n = 32u * NSPLIT;
        float *red = reinterpret_cast<float *>(gbase + C::OFF_RED);   // [3][NSPLIT][BM]
        uint32_t tcnt = 0;
        bool ok = true;
        for (int it = it_begin; it < it_end && ok; ++it) {
            const WorkItem w = a.items[it];
            const RangeSet *rs = a.ranges + w.u;
            const int n = w.tile_end - w.tile_begin;
            const int jrow = w.qt * BM + r;
            const bool valid = jrow < __ldg(&rs->cnt);
            int cell = valid ? a.idx[(int64_t)w.u * a.k_max + jrow] : 0;
            cell = (cell < 0 || cell >= a.mn) ? 0 : cell;
            if (n > 0) {
                // Q of the previous item is no longer read: its last PV, which
                // completes after every earlier MMA, was waited for
                const int gq = a.unit_group[w.u];
                const uint16_t *qrow = valid ? static_cast<const uint16_t *>(a.q) +
                                                   ((int64_t)gq * a.mn + cell) * a.D + w.h * DH + 2 * h * QCOLS
                                             : nullptr;
                const float *rope = a.rope ? a.rope + (int64_t)cell * DH + 2 * h * QCOLS : nullptr;
                q_pairs_to_tmem<QCOLS>(qrow, rope, tl + C::Q_COL + (uint32_t)(h * QCOLS));
                tmem_wait_st();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(BAR(C::B_QFULL));
            }
            // the unit's ranges in registers: tile t's valid rows without
            // global loads in the tile loop
            int rtiles[4], rlen[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                rtiles[q] = __ldg(&rs->tiles[q]);
                rlen[q] = __ldg(&rs->len[q]);
            }
            float m_run = -INFINITY, l_part = 0.f;
            for (int j = 0; j < n; ++j) {
                const uint32_t tj = tcnt + (uint32_t)j, b = tj & 1u;
                const bool okw = __all_sync(0xffffffffu, mbar_wait(BAR(C::B_SFULL + b), (tj >> 1) & 1u, abort_flag, wait_ns));
                int nvt = 0;
                {
                    int t = w.tile_begin + j;
#pragma unroll
                    for (int q = 0; q < 4; ++q) {
                        if (t >= 0 && t < rtiles[q]) nvt = min(BN, rlen[q] - t * BN);
                        t -= rtiles[q];
                    }
                }
                const int nv = nvt - h * SCOLS;       // valid columns of this slice (may be <= 0)
                const bool full = nv >= SCOLS;
                const uint32_t scol = tl + C::S_COL + (uint32_t)BN * b;
                const float sc = a.scale_log2;
                uint32_t sr[SCOLS], pk[PCOLS];
                float rowsum = 0.f;
                if (okw) {
                    tc_fence_after();
                    tmem_ld_cols<SCOLS>(scol + (uint32_t)(h * SCOLS), sr);
                    tmem_wait_ld();
                    // S_j is in registers: its TMEM buffer may take S_{j+2}
                    tc_fence_before();
                    __syncwarp();
                    if (lane == 0) mbar_arrive(BAR(C::B_SFREE + b));
                }
                float *redt = red + (b * NSPLIT) * BM;
                float m_new = m_run;
                if (j == 0) {
                    // the first tile of an item sets the reference: the row max
                    // over the slices (the scale is positive, so it is applied
                    // to the max of the raw scores)
                    redt[h * BM + r] = okw ? row_max<SCOLS>(sr, nv, full) : -INFINITY;
                    if (!bar_and(bar_id, bar_n, okw)) { ok = false; break; }
                    float mrow = redt[r];
#pragma unroll
                    for (int q = 1; q < NSPLIT; ++q) mrow = fmaxf(mrow, redt[q * BM + r]);
                    m_new = mrow * sc;
                    rowsum = row_exp<SCOLS>(sr, pk, sc, m_new, nv, full);
                } else {
                    // Later tiles take their exps against the running reference.
                    // It moves only if the row max grows past it by more than
                    // 2^8, i.e. if some p > 2^8; a row whose sum stays <= 2^8 has
                    // none, so only rows above that (or a timeout) take the slow
                    // path, together with their quarter: exact maxima exchanged,
                    // exps redone against a moved reference, O rescaled.
                    if (okw) rowsum = row_exp<SCOLS>(sr, pk, sc, m_run, nv, full);
                    const bool slow = !(rowsum <= 256.0f);
                    if (bar_or(bar_id, bar_n, slow || !okw)) {
                        redt[h * BM + r] = okw ? row_max<SCOLS>(sr, nv, full) : -INFINITY;
                        if (!bar_and(bar_id, bar_n, okw)) { ok = false; break; }
                        float mrow = redt[r];
#pragma unroll
                        for (int q = 1; q < NSPLIT; ++q) mrow = fmaxf(mrow, redt[q * BM + r]);
                        if (mrow * sc > m_run + 8.0f) {
                            m_new = mrow * sc;
                            rowsum = row_exp<SCOLS>(sr, pk, sc, m_new, nv, full);
                        }
                        const bool grow = m_new != m_run;
                        const float alpha = grow ? ex2_approx(m_run - m_new) : 1.0f;
                        if (__any_sync(0xffffffffu, grow)) {
                            // O must hold tile j-1 before its rows are rescaled; on
                            // a timeout the rescale is skipped and the next tile's
                            // barrier takes every slice out
                            const uint32_t tp = tj - 1u;
                            if (__all_sync(0xffffffffu, mbar_wait(BAR(C::B_PVDONE + tp % C::NPB),
                                                                  (tp / C::NPB) & 1u, abort_flag, wait_ns))) {
                                tc_fence_after();
#pragma unroll 1
                                for (int c16 = 0; c16 < OCOLS / 16; ++c16) {
                                    uint32_t o[16];
                                    const uint32_t ta = tl + (uint32_t)(h * OCOLS) + 16u * c16;
                                    tmem_ld16(ta, o);
                                    tmem_wait_ld();
#pragma unroll
                                    for (int e = 0; e < 16; ++e)
                                        o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                                    tmem_st16(ta, o);
                                }
                            }
                        }
                        l_part *= alpha;
                    }
                }
                l_part += rowsum;
                m_run = m_new;
                // P_j (bf16) into shared buffer j % 3, K-major and 128-byte
                // swizzled as the A operand of PV_j; the buffer was last read by
                // PV_{j-3}.  On a timeout the store is skipped and the next
                // barrier takes every slice out.
                if (__all_sync(0xffffffffu, mbar_wait(BAR(C::B_PVDONE + tj % C::NPB),
                                                      ((tj / C::NPB) & 1u) ^ 1u, abort_flag, wait_ns))) {
                    const uint32_t pbase = sP + (tj % C::NPB) * C::PBYTES;
#pragma unroll
                    for (int cc = 0; cc < PCOLS / 4; ++cc) {
                        const uint32_t off = sw128_offset(BM, r, h * (SCOLS / 8) + cc);
                        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(pbase + off), "r"(pk[4 * cc]),
                                     "r"(pk[4 * cc + 1]), "r"(pk[4 * cc + 2]), "r"(pk[4 * cc + 3]) : "memory");
                    }
                    fence_proxy_async();
                }
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(BAR(C::B_PFULL + tj % C::NPB));
            }
            if (!ok) break;
            float l_run = 0.f;
            if (n > 0) {
                const uint32_t tlast = tcnt + (uint32_t)n - 1u;
                const bool okw = __all_sync(0xffffffffu, mbar_wait(BAR(C::B_PVDONE + tlast % C::NPB),
                                                                   (tlast / C::NPB) & 1u, abort_flag, wait_ns));
                float *redl = red + (2 * NSPLIT) * BM;
                redl[h * BM + r] = l_part;
                if (!bar_and(bar_id, bar_n, okw)) { ok = false; break; }
                tc_fence_after();
#pragma unroll
                for (int q = 0; q < NSPLIT; ++q) l_run += redl[q * BM + r];
            }
            tcnt += (uint32_t)n;
            const float inv = l_run > 0.f ? 1.0f / l_run : 0.f;
            if (w.slot >= 0) {
                // split-KV partial (fp32, unnormalised): 32 columns at a time are
                // staged through shared memory so that each store instruction
                // writes four whole rows of 128 bytes.  The staging area is this
                // warp's part of the P ring, idle from the item's last PV (waited
                // for above) until the next item's first P, which no warp writes
                // before every warp has passed this epilogue (QFULL).
                float *stg = reinterpret_cast<float *>(gbase + C::OFF_P) + (warp - 4) * (32 * 36);
                float *pdst = a.part_o + ((int64_t)w.slot * BM + 32 * q4) * DH + h * OCOLS;
#pragma unroll 1
                for (int c0 = 0; c0 < OCOLS; c0 += 32) {
                    uint32_t o[32];
                    if (n > 0) {
                        tmem_ld32(tl + (uint32_t)(h * OCOLS + c0), o);
                        tmem_wait_ld();
                    } else {
#pragma unroll
                        for (int e = 0; e < 32; ++e) o[e] = 0u;
                    }
                    __syncwarp();
#pragma unroll
                    for (int k = 0; k < 8; ++k)
                        *reinterpret_cast<uint4 *>(stg + lane * 36 + 4 * k) =
                            make_uint4(o[4 * k], o[4 * k + 1], o[4 * k + 2], o[4 * k + 3]);
                    __syncwarp();
#pragma unroll
                    for (int q = 0; q < 8; ++q) {
                        const int row = 4 * q + (lane >> 3), c4 = 4 * (lane & 7);
                        __stcg(reinterpret_cast<float4 *>(pdst + (int64_t)row * DH + c0 + c4),
                               *reinterpret_cast<const float4 *>(stg + row * 36 + c4));
                    }
                }
            } else {
                // out = residual + O / l at the kept cell, rounded once to bf16;
                // EG chunks of 16 columns at a time with their residual loads
                // issued together
                constexpr int EG = OCOLS >= 32 ? 2 : 1;
#pragma unroll 1
                for (int c0 = 0; c0 < OCOLS; c0 += 16 * EG) {
                    const int col0 = h * OCOLS + c0;
                    const int64_t off = ((int64_t)w.u * a.mn + cell) * a.D + w.h * DH + col0;
                    uint4 res[2 * EG];
                    if (valid) {
#pragma unroll
                        for (int q = 0; q < 2 * EG; ++q)
                            res[q] = a.residual ? __ldg(reinterpret_cast<const uint4 *>(
                                                      static_cast<const uint16_t *>(a.residual) + off) + q)
                                                : make_uint4(0u, 0u, 0u, 0u);
                    }
                    uint32_t o[16 * EG];
                    if (n > 0) {
#pragma unroll
                        for (int e = 0; e < EG; ++e) tmem_ld16(tl + (uint32_t)(col0 + 16 * e), o + 16 * e);
                        tmem_wait_ld();
                    } else {
#pragma unroll
                        for (int e = 0; e < 16 * EG; ++e) o[e] = 0u;
                    }
                    if (!valid) continue;
                    uint4 *dp = reinterpret_cast<uint4 *>(static_cast<uint16_t *>(a.out) + off);
#pragma unroll
                    for (int q = 0; q < 2 * EG; ++q) {
                        const uint32_t xw[4] = {res[q].x, res[q].y, res[q].z, res[q].w};
                        uint32_t pw[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int k0 = 8 * q + 2 * e;
                            pw[e] = pack_bf16x2(__uint_as_float(xw[e] << 16) + __uint_as_float(o[k0]) * inv,
                                                __uint_as_float(xw[e] & 0xffff0000u) + __uint_as_float(o[k0 + 1]) * inv);
                        }
                        dp[q] = make_uint4(pw[0], pw[1], pw[2], pw[3]);
                    }
                }
            }
            if (valid && w.slot >= 0 && h == 0)
                reinterpret_cast<float2 *>(a.part_ml)[(int64_t)w.slot * BM + r] = make_float2(m_run, l_run);
            tc_fence_before();
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(TMEM_COLS) : "memory");
    }
    if (threadIdx.x == 0 && *abort_flag) latch_status(a.status, RS3_ETIMEOUT);
#undef BAR
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------
PFN_cuTensorMapEncodeTiled_v12000 encode_fn()
{
    static PFN_cuTensorMapEncodeTiled_v12000 fn = nullptr;
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(p);
    }
    return fn;
}

bool make_kv_map(CUtensorMap *m, const void *store, int64_t D, int64_t rows, int box_rows)
{
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)box_rows};
    const cuuint32_t es[2] = {1, 1};
    return enc(m, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(store), dims, strides, box, es,
               CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
               CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

template <int DH>
rs3_status launch(const ReadoutArgs &a, cudaStream_t st)
{
    if (rs3_kernel_smem((const void *)k_readout_tc<DH>, Cfg<DH>::SMEM) != RS3_OK) return RS3_ECUDA;
    const int64_t rows = (int64_t)a.U * a.rows_per_unit;
    if (rows >= (int64_t)1 << 31) return RS3_EUNSUPPORTED;
    CUtensorMap mk, mv;
    if (!make_kv_map(&mk, a.k_store, a.D, rows, Cfg<DH>::BN) ||
        !make_kv_map(&mv, a.v_store, a.D, rows, Cfg<DH>::BN))
        return RS3_ECUDA;
    const int64_t grid = a.grid_ctas;               // the plan's slices; unused ones exit at once
    launch_pdl(k_readout_tc<DH>, dim3((unsigned)grid), dim3(Cfg<DH>::NTHREADS), Cfg<DH>::SMEM, st, a, mk, mv);
    return cudaGetLastError() == cudaSuccess ? RS3_OK : RS3_ECUDA;
}

}  // namespace tc

bool rs3_tc_supported(int d) { return d == 64 || d == 128 || d == 256; }

int rs3_tc_block_n(int d)
{
    switch (d) {
    case 64: return tc::Cfg<64>::BN;
    case 128: return tc::Cfg<128>::BN;
    default: return tc::Cfg<256>::BN;
    }
}

rs3_status rs3_launch_tc_readout(const ReadoutArgs &a, cudaStream_t st)
{
    switch (a.d) {
    case 64: return tc::launch<64>(a, st);
    case 128: return tc::launch<128>(a, st);
    case 256: return tc::launch<256>(a, st);
    default: return RS3_EUNSUPPORTED;
    }
}
