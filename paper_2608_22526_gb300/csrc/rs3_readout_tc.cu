// rs3_readout_tc.cu -- tensor-core readout for bf16 (Sec. 3.1, Eq. 6 and
// Eq. 7) on sm_103a: tcgen05.mma with fp32 accumulators in TMEM, K/V tiles
// staged by TMA (cp.async.bulk.tensor, 128-byte swizzle), online softmax in
// the log2 domain.
//
// One persistent CTA per SM runs its slice of the stream-K plan: work items
// (unit, head, 128-query tile, range of BN-key tiles).  Warps:
//   warp 0      K producer: TMA of the key tile (d/64 boxes of BN rows x 64)
//   warp 2      V producer: TMA of the value tile
//   warp 1      TMEM allocation; one lane issues every MMA:
//               S_j = Q K_j^T   (M 128, N BN, K d; A = Q, B = K, both K-major)
//               O  += P_j V_j   (M 128, N d, K BN; A = P K-major, B = V MN-major)
//               S and P are double-buffered, so S_{j+1} runs while the softmax
//               of S_j is computed and P_{j+1} is written while PV_j runs.
//   warps 4..   NSM softmax warpgroups.  Warp w reads TMEM lanes 32 (w % 4)..,
//               i.e. query row r = 32 (w % 4) + lane; its group g = (w - 4) / 4
//               owns columns [g CPT, (g+1) CPT) of S (CPT = 32 or 64) and
//               columns [g d / NSM, (g+1) d / NSM) of O.  The groups gather
//               the kept query rows with cp.async into the swizzled Q tile
//               (rotated by RoPE of their own cell, Eq. 7, when a table is
//               given), exchange row maxima through shared memory, write P_j
//               as bf16, rescale O in TMEM only when the running max grows by
//               more than 2^8, and run the epilogue (O / l + residual, or
//               split-KV partials).
// Shapes: d = 256 uses 64-key tiles with 2 K/V stages and 2 softmax groups,
// d = 128 128-key tiles, 2 stages, 2 groups, d = 64 128-key tiles, 3 stages,
// 4 groups.  TMEM: O in columns [0, d), S buffers from column 256 (512 columns).
// Every mbarrier wait is bounded (1 s of %globaltimer): on expiry the CTA
// raises an abort flag, drains its copies and MMAs, frees TMEM and the launch
// latches RS3_ETIMEOUT.
#include "rs3_readout_common.cuh"
#include "rs3_tc_ptx.cuh"

#include <cudaTypedefs.h>

namespace tc {

constexpr int BM = 128;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t S_COL0 = 256;

template <int DH>
struct Cfg {
    static constexpr int BN = DH == 256 ? 64 : 128;          // keys per tile
    static constexpr int KST = DH == 64 ? 3 : 2;             // K / V stages
    static constexpr int NSM = 1;                            // softmax warpgroups
    static constexpr int CPT = BN / NSM;                     // S columns per softmax thread
    static constexpr int OCT = DH / NSM;                     // O columns per softmax thread
    static constexpr int NTHREADS = 128 + 128 * NSM;
    static constexpr int SMT = 128 * NSM;                    // softmax threads
    static constexpr int QBYTES = BM * DH * 2;
    static constexpr int KVBYTES = BN * DH * 2;              // one stage
    static constexpr int PBYTES = BM * BN * 2;               // one P buffer
    static constexpr int OFF_Q = 0;
    static constexpr int OFF_K = OFF_Q + QBYTES;
    static constexpr int OFF_V = OFF_K + KST * KVBYTES;
    static constexpr int OFF_P = OFF_V + KST * KVBYTES;
    static constexpr int OFF_RED = OFF_P + 2 * PBYTES;       // [NSM][128] floats
    static constexpr int OFF_BAR = OFF_RED + NSM * BM * 4;
    static constexpr int NBAR = 4 * KST + 11;
    static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
    static constexpr int SMEM = OFF_MISC + 16 + 1024;                  // + alignment slack
    // barrier indices
    static constexpr int B_KFULL = 0, B_KEMPTY = KST, B_VFULL = 2 * KST, B_VEMPTY = 3 * KST;
    static constexpr int B_SFULL = 4 * KST, B_SFREE = 4 * KST + 2, B_PFULL = 4 * KST + 4;
    static constexpr int B_PVDONE = 4 * KST + 6, B_QFULL = 4 * KST + 8, B_DRAIN = 4 * KST + 9;
    static constexpr int B_GRP = 4 * KST + 10;               // softmax groups' exchange barrier
    static_assert(CPT % 32 == 0 && OCT % 16 == 0, "softmax slice shapes");
};
static_assert(Cfg<256>::SMEM <= 232448 && Cfg<128>::SMEM <= 232448 && Cfg<64>::SMEM <= 232448,
              "shared memory budget");

// Softmax pieces of one thread's S slice (raw scores as fp32 bits).
template <int N>
__device__ __forceinline__ float slice_max(const uint32_t (&sr)[N])
{
    float m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
    for (int c = 0; c < N; c += 2) {
        m0 = fmaxf(m0, __uint_as_float(sr[c]));
        m1 = fmaxf(m1, __uint_as_float(sr[c + 1]));
    }
    return fmaxf(m0, m1);
}

template <int N>
__device__ __forceinline__ float slice_max_masked(const uint32_t (&sr)[N], int nv)
{
    float m = -INFINITY;
#pragma unroll
    for (int c = 0; c < N; ++c) m = fmaxf(m, c < nv ? __uint_as_float(sr[c]) : -INFINITY);
    return m;
}

// p = 2^(s * sc - ref) packed as bf16 pairs; returns the sum of the p.
template <int N>
__device__ __forceinline__ float slice_exp(const uint32_t (&sr)[N], uint32_t (&pk)[N / 2], float sc, float ref,
                                           int nv, bool full)
{
    const float nref = -ref;
    float r0 = 0.f, r1 = 0.f;
#pragma unroll
    for (int c = 0; c < N / 2; ++c) {
        float p0 = ex2_approx(fmaf(__uint_as_float(sr[2 * c]), sc, nref));
        float p1 = ex2_approx(fmaf(__uint_as_float(sr[2 * c + 1]), sc, nref));
        if (!full) {
            p0 = 2 * c < nv ? p0 : 0.f;
            p1 = 2 * c + 1 < nv ? p1 : 0.f;
        }
        r0 += p0;
        r1 += p1;
        pk[c] = pack_bf16x2(p0, p1);
    }
    return r0 + r1;
}

// slice_exp against `ref`, and the max of the valid raw scores in the same pass.
template <int N>
__device__ __forceinline__ float slice_exp_max(const uint32_t (&sr)[N], uint32_t (&pk)[N / 2], float sc,
                                               float ref, int nv, bool full, float &mx)
{
    const float nref = -ref;
    float r0 = 0.f, r1 = 0.f, m0 = -INFINITY, m1 = -INFINITY;
#pragma unroll
    for (int c = 0; c < N / 2; ++c) {
        const float s0 = __uint_as_float(sr[2 * c]), s1 = __uint_as_float(sr[2 * c + 1]);
        float p0 = ex2_approx(fmaf(s0, sc, nref));
        float p1 = ex2_approx(fmaf(s1, sc, nref));
        if (full) {
            m0 = fmaxf(m0, s0);
            m1 = fmaxf(m1, s1);
        } else {
            p0 = 2 * c < nv ? p0 : 0.f;
            p1 = 2 * c + 1 < nv ? p1 : 0.f;
            m0 = fmaxf(m0, 2 * c < nv ? s0 : -INFINITY);
            m1 = fmaxf(m1, 2 * c + 1 < nv ? s1 : -INFINITY);
        }
        r0 += p0;
        r1 += p1;
        pk[c] = pack_bf16x2(p0, p1);
    }
    mx = fmaxf(m0, m1);
    return r0 + r1;
}

template <int DH>
__global__ void __launch_bounds__(Cfg<DH>::NTHREADS, 1)
k_readout_tc(const ReadoutArgs a, const __grid_constant__ CUtensorMap tmk,
             const __grid_constant__ CUtensorMap tmv)
{
    using C = Cfg<DH>;
    constexpr int KST = C::KST, BN = C::BN, NSM = C::NSM, CPT = C::CPT, OCT = C::OCT;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *gbase = smem_raw + (base - raw);
    const uint32_t sQ = base + C::OFF_Q, sK = base + C::OFF_K, sV = base + C::OFF_V, sP = base + C::OFF_P;
    float *red = reinterpret_cast<float *>(gbase + C::OFF_RED);
    const uint32_t bars = base + C::OFF_BAR;
    volatile int *abort_flag = reinterpret_cast<volatile int *>(gbase + C::OFF_MISC);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(gbase + C::OFF_MISC + 8);
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
#define BAR(i) (bars + 8u * (uint32_t)(i))

    if (threadIdx.x == 0) {
        for (int s = 0; s < KST; ++s) {
            mbar_init(BAR(C::B_KFULL + s), 1);
            mbar_init(BAR(C::B_KEMPTY + s), 1);
            mbar_init(BAR(C::B_VFULL + s), 1);
            mbar_init(BAR(C::B_VEMPTY + s), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(BAR(C::B_SFULL + b), 1);
            mbar_init(BAR(C::B_SFREE + b), 4 * NSM);      // one arrival per softmax warp
            mbar_init(BAR(C::B_PFULL + b), 4 * NSM);
            mbar_init(BAR(C::B_PVDONE + b), 1);
        }
        mbar_init(BAR(C::B_QFULL), 4 * NSM);
        mbar_init(BAR(C::B_DRAIN), 1);
        mbar_init(BAR(C::B_GRP), 4 * NSM);
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
    // this CTA's slice of the stream-K plan
    const int it_begin = a.cta_items[blockIdx.x], it_end = a.cta_items[blockIdx.x + 1];

    if ((warp == 0 || warp == 2) && lane == 0) {
        // ------------------------------------------------------------------
        // TMA producers (warp 0: keys, warp 2: values)
        // ------------------------------------------------------------------
        const bool is_k = warp == 0;
        const CUtensorMap *map = is_k ? &tmk : &tmv;
        const uint32_t dst0 = is_k ? sK : sV;
        const int b_full = is_k ? C::B_KFULL : C::B_VFULL;
        const int b_empty = is_k ? C::B_KEMPTY : C::B_VEMPTY;
        uint32_t cnt = 0;
        for (int it = it_begin; it < it_end && !*abort_flag; ++it) {
            const WorkItem w = a.items[it];
            const RangeSet rs = a.ranges[w.u];
            for (int t = w.tile_begin; t < w.tile_end; ++t, ++cnt) {
                const uint32_t st = cnt % KST, ph = (cnt / KST) & 1u;
                if (!mbar_wait(BAR(b_empty + st), ph ^ 1u, abort_flag)) goto producer_done;
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
        for (uint32_t k = (cnt > (uint32_t)KST ? cnt - KST : 0); k < cnt; ++k)
            mbar_drain(BAR(b_full + k % KST), (k / KST) & 1u);
    } else if (warp == 1 && lane == 0) {
        // ------------------------------------------------------------------
        // MMA issuer
        // ------------------------------------------------------------------
        constexpr uint32_t ID_S = idesc_bf16(BM, BN, false);
        constexpr uint32_t ID_PV = idesc_bf16(BM, DH, true);
        // descriptors built once; a k-step only adds its byte offset / 16 to the
        // start-address field (every address stays below 256 KB, so the 14-bit
        // field cannot carry)
        const uint64_t dq = desc_sw128(sQ, 16, 1024);
        uint64_t dk[KST], dv[KST], dp[2];
#pragma unroll
        for (int s = 0; s < KST; ++s) {
            dk[s] = desc_sw128(sK + s * C::KVBYTES, 16, 1024);
            dv[s] = desc_sw128(sV + s * C::KVBYTES, BN * 128, 1024);
        }
        dp[0] = desc_sw128(sP, 16, 1024);
        dp[1] = desc_sw128(sP + C::PBYTES, 16, 1024);
        uint32_t tcnt = 0, icnt = 0;
        auto issue_s = [&](uint32_t tj) -> bool {
            const uint32_t st = tj % KST, b = tj & 1u;
            if (!mbar_wait(BAR(C::B_KFULL + st), (tj / KST) & 1u, abort_flag)) return false;
            if (!mbar_wait(BAR(C::B_SFREE + b), ((tj >> 1) & 1u) ^ 1u, abort_flag)) return false;
            tc_fence_after();
            const uint64_t dks = dk[st];
            const uint32_t dst = tmem + S_COL0 + (uint32_t)BN * b;
#pragma unroll
            for (int kk = 0; kk < DH / 16; ++kk) {
                const uint32_t offq = (uint32_t)((kk >> 2) * (BM * 128) + (kk & 3) * 32);
                const uint32_t offk = (uint32_t)((kk >> 2) * (BN * 128) + (kk & 3) * 32);
                tc_mma(dst, dq + (offq >> 4), dks + (offk >> 4), ID_S, kk > 0 ? 1u : 0u);
            }
            tc_commit(BAR(C::B_SFULL + b));
            tc_commit(BAR(C::B_KEMPTY + st));
            return true;
        };
        bool ok = true;
        for (int it = it_begin; it < it_end && ok; ++it) {
            const WorkItem w = a.items[it];
            const int n = w.tile_end - w.tile_begin;
            if (n <= 0) continue;
            if (!mbar_wait(BAR(C::B_QFULL), icnt & 1u, abort_flag)) { ok = false; break; }
            ++icnt;
            tc_fence_after();
            if (!issue_s(tcnt)) { ok = false; break; }
            for (int j = 0; j < n; ++j) {
                const uint32_t tj = tcnt + (uint32_t)j, pb = tj & 1u;
                if (j + 1 < n && !issue_s(tj + 1)) { ok = false; break; }
                const uint32_t st = tj % KST;
                if (!mbar_wait(BAR(C::B_PFULL + pb), (tj >> 1) & 1u, abort_flag)) { ok = false; break; }
                if (!mbar_wait(BAR(C::B_VFULL + st), (tj / KST) & 1u, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint64_t dvs = dv[st], dps = dp[pb];
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
        // every MMA issued by this thread completes before TMEM is released
        tc_commit(BAR(C::B_DRAIN));
        mbar_drain(BAR(C::B_DRAIN), 0);
    } else if (warp >= 4) {
        // ------------------------------------------------------------------
        // gather, softmax / correction, epilogue
        // ------------------------------------------------------------------
        const int ts = threadIdx.x - 128;             // 0 .. SMT-1
        const int g = ts >> 7;                        // softmax group: column slice
        const int wq = warp & 3;                      // TMEM lane quarter
        const int r = 32 * wq + lane;                 // query row of the tile
        const uint32_t tl = tmem + ((uint32_t)(32 * wq) << 16);
        constexpr int CPR = DH / 8;                   // 16-byte chunks per query row
        constexpr int NCH = BM * CPR / C::SMT;        // chunks gathered per thread
        uint32_t tcnt = 0;
        bool ok = true;
        float *red_r = red + r;                       // red[g * 128 + r]
        // barrier of all softmax warps (one arrival per warp), bounded like
        // every other wait so that an abort cannot strand a group
        uint32_t grp_phase = 0;
        auto grp_sync = [&]() -> bool {
            __syncwarp();
            if (lane == 0) mbar_arrive(BAR(C::B_GRP));
            const bool okw = __all_sync(0xffffffffu, mbar_wait(BAR(C::B_GRP), grp_phase & 1u, abort_flag));
            ++grp_phase;
            return okw;
        };
        for (int it = it_begin; it < it_end && ok; ++it) {
            const WorkItem w = a.items[it];
            const RangeSet rs = a.ranges[w.u];
            const int n = w.tile_end - w.tile_begin;
            if (n > 0) {
                // gather the kept query rows of this tile: chunk e = ts + SMT k
                // is 16 bytes of row e / CPR; rows past count are zero-filled
                const int gq = a.unit_group[w.u];
                const uint16_t *qg = static_cast<const uint16_t *>(a.q) + (int64_t)gq * a.mn * a.D + w.h * DH;
                int cellk[NCH];
#pragma unroll
                for (int k = 0; k < NCH; ++k) {
                    const int row = (ts + C::SMT * k) / CPR;
                    const int jrow = w.qt * BM + row;
                    int cell = -1;
                    if (jrow < rs.cnt) {
                        cell = a.idx[(int64_t)w.u * a.k_max + jrow];
                        cell = (cell < 0 || cell >= a.mn) ? 0 : cell;
                    }
                    cellk[k] = cell;
                }
#pragma unroll
                for (int k = 0; k < NCH; ++k) {
                    const int e = ts + C::SMT * k, row = e / CPR, ch = e % CPR;
                    const int cell = cellk[k];
                    const uint16_t *src = qg + (int64_t)(cell < 0 ? 0 : cell) * a.D + ch * 8;
                    cp_async16(sQ + sw128_offset(BM, row, ch), src, cell < 0 ? 0u : 16u);
                }
                cp_async_wait_all();
                if (a.rope) {
                    // Eq. 7: rotate each pair by f[cell] of the query's own cell
#pragma unroll
                    for (int k = 0; k < NCH; ++k) {
                        const int cell = cellk[k];
                        if (cell < 0) continue;
                        const int e = ts + C::SMT * k, row = e / CPR, ch = e % CPR;
                        const uint32_t sa = sQ + sw128_offset(BM, row, ch);
                        uint32_t wv[4];
                        asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                                     : "=r"(wv[0]), "=r"(wv[1]), "=r"(wv[2]), "=r"(wv[3]) : "r"(sa));
                        const float4 *f = reinterpret_cast<const float4 *>(
                            a.rope + ((int64_t)cell * (DH / 2) + ch * 4) * 2);
                        const float4 f0 = __ldg(f), f1 = __ldg(f + 1);
                        const float cs[4] = {f0.x, f0.z, f1.x, f1.z};
                        const float sn[4] = {f0.y, f0.w, f1.y, f1.w};
#pragma unroll
                        for (int p = 0; p < 4; ++p) {
                            const float x0 = __uint_as_float(wv[p] << 16);
                            const float x1 = __uint_as_float(wv[p] & 0xffff0000u);
                            wv[p] = pack_bf16x2(x0 * cs[p] - x1 * sn[p], x0 * sn[p] + x1 * cs[p]);
                        }
                        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(sa), "r"(wv[0]),
                                     "r"(wv[1]), "r"(wv[2]), "r"(wv[3]) : "memory");
                    }
                }
                fence_proxy_async();
                __syncwarp();
                if (lane == 0) mbar_arrive(BAR(C::B_QFULL));
            }
            const int jrow = w.qt * BM + r;
            const bool valid = jrow < rs.cnt;
            int cell = valid ? a.idx[(int64_t)w.u * a.k_max + jrow] : 0;
            cell = (cell < 0 || cell >= a.mn) ? 0 : cell;
            float m_run = -INFINITY, l_part = 0.f;
            for (int j = 0; j < n; ++j) {
                const uint32_t tj = tcnt + (uint32_t)j, b = tj & 1u;
                if (!__all_sync(0xffffffffu, mbar_wait(BAR(C::B_SFULL + b), (tj >> 1) & 1u, abort_flag))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                int64_t row0;
                int nvalid;
                tile_rows(rs, w.tile_begin + j, BN, row0, nvalid);
                uint32_t sr[CPT];
#pragma unroll
                for (int c4 = 0; c4 < CPT / 32; ++c4)
                    tmem_ld32(tl + S_COL0 + (uint32_t)BN * b + (uint32_t)(g * CPT) + 32u * c4, sr + 32 * c4);
                tmem_wait_ld();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(BAR(C::B_SFREE + b));
                // Valid columns of this slice.  After the first tile of an item
                // the exps are taken against the running reference m_run with
                // the tile max gathered in the same pass; only if the max grows
                // past m_run + 8 (a factor 2^8) are they redone against the new
                // max (and O rescaled below).  The first tile takes its max
                // first.  The scale is positive, so it is applied to the max of
                // the raw scores.
                const int nv = nvalid - g * CPT;      // may be <= 0 for a late slice
                const bool full = nv >= CPT;
                const float sc = a.scale_log2;
                uint32_t pk[CPT / 2];
                float rowsum, m_new;
                if (j == 0 || NSM > 1) {
                    float mt = full ? slice_max<CPT>(sr) : slice_max_masked<CPT>(sr, nv);
                    if (NSM > 1) {
                        red_r[g * BM] = mt;
                        if (!grp_sync()) { ok = false; break; }
#pragma unroll
                        for (int q = 0; q < NSM; ++q) mt = fmaxf(mt, red_r[q * BM]);
                        if (!grp_sync()) { ok = false; break; }
                    }
                    mt *= sc;
                    m_new = (j == 0) ? mt : (mt > m_run + 8.0f ? mt : m_run);
                    rowsum = slice_exp<CPT>(sr, pk, sc, m_new, nv, full);
                } else {
                    float mt;
                    rowsum = slice_exp_max<CPT>(sr, pk, sc, m_run, nv, full, mt);
                    m_new = m_run;
                    if (mt * sc > m_run + 8.0f) {
                        m_new = mt * sc;
                        rowsum = slice_exp<CPT>(sr, pk, sc, m_new, nv, full);
                    }
                }
                // P buffer b was last read by PV of tile tj - 2
                if (!__all_sync(0xffffffffu, mbar_wait(BAR(C::B_PVDONE + b), ((tj >> 1) & 1u) ^ 1u, abort_flag))) {
                    ok = false;
                    break;
                }
                if (j > 0) {
                    const bool grow = m_new != m_run;
                    const float alpha = grow ? ex2_approx(m_run - m_new) : 1.0f;
                    if (__any_sync(0xffffffffu, grow)) {
                        // O must hold tile j-1 before its slice is rescaled
                        const uint32_t tp = tj - 1u;
                        if (!__all_sync(0xffffffffu,
                                        mbar_wait(BAR(C::B_PVDONE + (tp & 1u)), (tp >> 1) & 1u, abort_flag))) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
#pragma unroll 1
                        for (int c16 = 0; c16 < OCT / 16; ++c16) {
                            uint32_t o[16];
                            const uint32_t ta = tl + (uint32_t)(g * OCT) + 16u * c16;
                            tmem_ld16(ta, o);
                            tmem_wait_ld();
#pragma unroll
                            for (int e = 0; e < 16; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                            tmem_st16(ta, o);
                        }
                        tmem_wait_st();
                    }
                    l_part *= alpha;
                }
                l_part += rowsum;
                m_run = m_new;
                const uint32_t pbase = sP + b * C::PBYTES;
#pragma unroll
                for (int cc = 0; cc < CPT / 8; ++cc) {
                    const uint32_t off = sw128_offset(BM, r, g * (CPT / 8) + cc);
                    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(pbase + off), "r"(pk[4 * cc]),
                                 "r"(pk[4 * cc + 1]), "r"(pk[4 * cc + 2]), "r"(pk[4 * cc + 3]) : "memory");
                }
                fence_proxy_async();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(BAR(C::B_PFULL + b));
            }
            if (!ok) break;
            if (n > 0) {
                const uint32_t tlast = tcnt + (uint32_t)n - 1u;
                if (!__all_sync(0xffffffffu,
                                mbar_wait(BAR(C::B_PVDONE + (tlast & 1u)), (tlast >> 1) & 1u, abort_flag))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
            }
            tcnt += (uint32_t)n;
            // row sum over the groups' slices
            float l_run = l_part;
            if (NSM > 1) {
                red_r[g * BM] = l_part;
                if (!grp_sync()) { ok = false; break; }
                l_run = 0.f;
#pragma unroll
                for (int q = 0; q < NSM; ++q) l_run += red_r[q * BM];
                if (!grp_sync()) { ok = false; break; }
            }
            // epilogue: this group's O columns [g OCT, (g+1) OCT)
            const float inv = l_run > 0.f ? 1.0f / l_run : 0.f;
#pragma unroll 1
            for (int c16 = 0; c16 < OCT / 16; ++c16) {
                uint32_t o[16];
                const int col = g * OCT + 16 * c16;
                if (n > 0) {
                    tmem_ld16(tl + (uint32_t)col, o);
                    tmem_wait_ld();
                } else {
#pragma unroll
                    for (int e = 0; e < 16; ++e) o[e] = 0u;
                }
                if (!valid) continue;
                if (w.slot < 0) {
                    const int64_t off = ((int64_t)w.u * a.mn + cell) * a.D + w.h * DH + col;
                    float res[16];
                    if (a.residual) {
                        const uint4 *rp = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(a.residual) + off);
#pragma unroll
                        for (int q4 = 0; q4 < 2; ++q4) {
                            const uint4 x = rp[q4];
                            const uint32_t xw[4] = {x.x, x.y, x.z, x.w};
#pragma unroll
                            for (int e = 0; e < 4; ++e) {
                                res[8 * q4 + 2 * e] = __uint_as_float(xw[e] << 16);
                                res[8 * q4 + 2 * e + 1] = __uint_as_float(xw[e] & 0xffff0000u);
                            }
                        }
                    } else {
#pragma unroll
                        for (int e = 0; e < 16; ++e) res[e] = 0.f;
                    }
                    uint4 *dp = reinterpret_cast<uint4 *>(static_cast<uint16_t *>(a.out) + off);
#pragma unroll
                    for (int q4 = 0; q4 < 2; ++q4) {
                        uint32_t pw[4];
#pragma unroll
                        for (int e = 0; e < 4; ++e) {
                            const int k0 = 8 * q4 + 2 * e;
                            pw[e] = pack_bf16x2(res[k0] + __uint_as_float(o[k0]) * inv,
                                                res[k0 + 1] + __uint_as_float(o[k0 + 1]) * inv);
                        }
                        dp[q4] = make_uint4(pw[0], pw[1], pw[2], pw[3]);
                    }
                } else {
                    float4 *po = reinterpret_cast<float4 *>(a.part_o + ((int64_t)w.slot * BM + r) * DH + col);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4)
                        po[q4] = make_float4(__uint_as_float(o[4 * q4]), __uint_as_float(o[4 * q4 + 1]),
                                             __uint_as_float(o[4 * q4 + 2]), __uint_as_float(o[4 * q4 + 3]));
                }
            }
            if (valid && w.slot >= 0 && g == 0)
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
    static bool attr = false;
    if (!attr) {
        if (cudaFuncSetAttribute(k_readout_tc<DH>, cudaFuncAttributeMaxDynamicSharedMemorySize, Cfg<DH>::SMEM) !=
            cudaSuccess)
            return RS3_ECUDA;
        attr = true;
    }
    const int64_t rows = (int64_t)a.U * a.rows_per_unit;
    if (rows >= (int64_t)1 << 31) return RS3_EUNSUPPORTED;
    CUtensorMap mk, mv;
    if (!make_kv_map(&mk, a.k_store, a.D, rows, Cfg<DH>::BN) ||
        !make_kv_map(&mv, a.v_store, a.D, rows, Cfg<DH>::BN))
        return RS3_ECUDA;
    const int64_t grid = a.grid_ctas;               // the plan's slices; unused ones exit at once
    k_readout_tc<DH><<<(unsigned)grid, Cfg<DH>::NTHREADS, Cfg<DH>::SMEM, st>>>(a, mk, mv);
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
