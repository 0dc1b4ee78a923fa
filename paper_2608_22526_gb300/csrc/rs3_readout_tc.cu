// rs3_readout_tc.cu -- tensor-core readout for bf16 (Sec. 3.1, Eq. 6 and
// Eq. 7) on sm_103a: tcgen05.mma with fp32 accumulators in TMEM, K/V tiles
// staged by TMA (cp.async.bulk.tensor, 128-byte swizzle), online softmax in
// the log2 domain.
//
// One persistent CTA per SM walks the planner's work items (unit, head,
// 128-query tile, range of 128-key tiles).  Per CTA, 8 warps:
//   warp 0      K producer: TMA of the key tile (d/64 boxes of 128 rows x 64)
//   warp 2      V producer: TMA of the value tile
//   warp 1      TMEM allocation; one lane issues every MMA:
//               S_j = Q K_j^T   (M 128, N 128, K d; A = Q, B = K, both K-major)
//               O  += P_j V_j   (M 128, N d, K 128; A = P K-major, B = V MN-major)
//               S is double-buffered in TMEM so S_{j+1} runs while the
//               softmax of S_j is computed.
//   warps 4-7   one thread per query row: gather the kept query rows (and
//               rotate them by RoPE of their own cell, Eq. 7) into shared
//               memory, softmax of S_j from TMEM, P_j to shared memory as bf16,
//               O rescaled in TMEM only when the running max grows by more
//               than 2^8, and the epilogue (O / l + residual, or split-KV
//               partials).
// TMEM: O in columns [0, d), S buffers at 256 and 384 (512 columns).
// Every mbarrier wait is bounded (1 s of %globaltimer): on expiry the CTA
// raises an abort flag, drains its copies and MMAs, frees TMEM and the launch
// latches RS3_ETIMEOUT.
#include "rs3_readout_common.cuh"

#include <cuda.h>
#include <cudaTypedefs.h>

namespace tc {

constexpr int BM = 128;
constexpr int BN = 128;
constexpr int NTHREADS = 256;
constexpr uint64_t WAIT_LIMIT_NS = 1000000000ull;
constexpr uint32_t TMEM_COLS = 512;
constexpr uint32_t S_COL0 = 256;

template <int DH>
struct Cfg {
    static constexpr int KST = DH == 256 ? 1 : (DH == 128 ? 2 : 3);   // K / V stages
    static constexpr int QBYTES = BM * DH * 2;
    static constexpr int KVBYTES = BN * DH * 2;                          // one stage
    static constexpr int PBYTES = BM * BN * 2;
    static constexpr int OFF_Q = 0;
    static constexpr int OFF_K = OFF_Q + QBYTES;
    static constexpr int OFF_V = OFF_K + KST * KVBYTES;
    static constexpr int OFF_P = OFF_V + KST * KVBYTES;
    static constexpr int OFF_BAR = OFF_P + PBYTES;
    static constexpr int NBAR = 4 * KST + 8;
    static constexpr int OFF_MISC = OFF_BAR + NBAR * 8;
    static constexpr int SMEM = OFF_MISC + 16 + 1024;                  // + alignment slack
    // barrier indices
    static constexpr int B_KFULL = 0, B_KEMPTY = KST, B_VFULL = 2 * KST, B_VEMPTY = 3 * KST;
    static constexpr int B_SFULL = 4 * KST, B_SFREE = 4 * KST + 2, B_PFULL = 4 * KST + 4;
    static constexpr int B_PVDONE = 4 * KST + 5, B_QFULL = 4 * KST + 6, B_DRAIN = 4 * KST + 7;
};
static_assert(Cfg<256>::SMEM <= 232448, "shared memory budget");

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------
__device__ __forceinline__ uint32_t smem_u32(const void *p)
{
    return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count)
{
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar)
{
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(uint32_t bar, uint32_t bytes)
{
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

__device__ __forceinline__ bool mbar_try(uint32_t bar, uint32_t parity)
{
    uint32_t ok;
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
        "selp.u32 %0, 1, 0, p;\n\t}"
        : "=r"(ok)
        : "r"(bar), "r"(parity)
        : "memory");
    return ok != 0;
}

__device__ __forceinline__ uint64_t gtimer()
{
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

// Waits for the phase with parity `parity` to complete; gives up (and raises
// the CTA's abort flag) after WAIT_LIMIT_NS, or at once if the flag is up.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, volatile int *abort_flag)
{
    if (mbar_try(bar, parity)) return true;
    const uint64_t t0 = gtimer();
    while (true) {
        if (mbar_try(bar, parity)) return true;
        if (*abort_flag) return false;
        if (gtimer() - t0 > WAIT_LIMIT_NS) {
            *abort_flag = 1;
            return false;
        }
    }
}

// Bounded wait that ignores the abort flag (used to drain work in flight).
__device__ __forceinline__ void mbar_drain(uint32_t bar, uint32_t parity)
{
    const uint64_t t0 = gtimer();
    while (!mbar_try(bar, parity))
        if (gtimer() - t0 > WAIT_LIMIT_NS) return;
}

__device__ __forceinline__ void fence_proxy_async()
{
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

__device__ __forceinline__ void tma_load_2d(uint32_t dst, const CUtensorMap *map, uint32_t bar, int x, int y)
{
    asm volatile(
        "cp.async.bulk.tensor.2d.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1, {%2, %3}], [%4];"
        ::"r"(dst), "l"(reinterpret_cast<uint64_t>(map)), "r"(x), "r"(y), "r"(bar)
        : "memory");
}

__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }

__device__ __forceinline__ void tc_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}

__device__ __forceinline__ void tc_mma(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate)
{
    asm volatile(
        "{\n\t.reg .pred p;\n\t"
        "setp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}"
        ::"r"(d_tmem), "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}

__device__ __forceinline__ void tmem_ld32(uint32_t taddr, uint32_t *r)
{
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
        "{%0, %1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, "
        "%16, %17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]),
          "=r"(r[15]), "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]),
          "=r"(r[22]), "=r"(r[23]), "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]),
          "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
}

__device__ __forceinline__ void tmem_st32(uint32_t taddr, const uint32_t *r)
{
    asm volatile(
        "tcgen05.st.sync.aligned.32x32b.x32.b32 [%0], "
        "{%1, %2, %3, %4, %5, %6, %7, %8, %9, %10, %11, %12, %13, %14, %15, %16, "
        "%17, %18, %19, %20, %21, %22, %23, %24, %25, %26, %27, %28, %29, %30, %31, %32};"
        ::"r"(taddr), "r"(r[0]), "r"(r[1]), "r"(r[2]), "r"(r[3]), "r"(r[4]), "r"(r[5]), "r"(r[6]),
          "r"(r[7]), "r"(r[8]), "r"(r[9]), "r"(r[10]), "r"(r[11]), "r"(r[12]), "r"(r[13]), "r"(r[14]),
          "r"(r[15]), "r"(r[16]), "r"(r[17]), "r"(r[18]), "r"(r[19]), "r"(r[20]), "r"(r[21]),
          "r"(r[22]), "r"(r[23]), "r"(r[24]), "r"(r[25]), "r"(r[26]), "r"(r[27]), "r"(r[28]),
          "r"(r[29]), "r"(r[30]), "r"(r[31])
        : "memory");
}

__device__ __forceinline__ void tmem_wait_ld() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }
__device__ __forceinline__ void tmem_wait_st() { asm volatile("tcgen05.wait::st.sync.aligned;" ::: "memory"); }

// Shared-memory matrix descriptor, 128-byte swizzle (tcgen05 format: start
// address, leading / stride byte offsets in 16-byte units, version 1 at bit 46,
// swizzle mode 2 at bits 61-63).  K-major tiles: SBO = 1024 (8 rows of 128 B),
// LBO unused.  MN-major tiles: LBO = distance between 64-element column
// blocks, SBO = 1024 (8 rows).
__device__ __forceinline__ uint64_t desc_sw128(uint32_t saddr, uint32_t lbo, uint32_t sbo)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)((lbo >> 4) & 0x3FFFu) << 16;
    d |= (uint64_t)((sbo >> 4) & 0x3FFFu) << 32;
    d |= (uint64_t)1 << 46;
    d |= (uint64_t)2 << 61;
    return d;
}

// Instruction descriptor of kind::f16: bf16 A and B, fp32 D, A K-major,
// B K-major or MN-major, N >> 3 at bit 17, M >> 4 at bit 24.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N, bool b_mn_major)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | ((b_mn_major ? 1u : 0u) << 16) |
           ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// Byte offset of 16-byte chunk `ch` (of 8 bf16) in row `r` of a K-major tile
// with `rows` rows stored as 128-byte-swizzled 64-column blocks.
__device__ __forceinline__ uint32_t sw128_offset(int rows, int r, int ch)
{
    return (uint32_t)((ch >> 3) * rows * 128 + r * 128 + (((ch & 7) ^ (r & 7)) << 4));
}

// ---------------------------------------------------------------------------
// the kernel
// ---------------------------------------------------------------------------
template <int DH>
__global__ void __launch_bounds__(NTHREADS, 1)
k_readout_tc(const ReadoutArgs a, const __grid_constant__ CUtensorMap tmk,
             const __grid_constant__ CUtensorMap tmv)
{
    using C = Cfg<DH>;
    constexpr int KST = C::KST;
    extern __shared__ uint8_t smem_raw[];
    const uint32_t raw = smem_u32(smem_raw);
    const uint32_t base = (raw + 1023u) & ~1023u;
    uint8_t *gbase = smem_raw + (base - raw);
    const uint32_t sQ = base + C::OFF_Q, sK = base + C::OFF_K, sV = base + C::OFF_V, sP = base + C::OFF_P;
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
        mbar_init(BAR(C::B_SFULL + 0), 1);
        mbar_init(BAR(C::B_SFULL + 1), 1);
        mbar_init(BAR(C::B_SFREE + 0), 128);
        mbar_init(BAR(C::B_SFREE + 1), 128);
        mbar_init(BAR(C::B_PFULL), 128);
        mbar_init(BAR(C::B_PVDONE), 1);
        mbar_init(BAR(C::B_QFULL), 128);
        mbar_init(BAR(C::B_DRAIN), 1);
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
    const int n_items = a.header->n_items;

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
        for (int it = blockIdx.x; it < n_items && !*abort_flag; it += gridDim.x) {
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
        uint32_t tcnt = 0, icnt = 0;
        auto issue_s = [&](uint32_t tj) -> bool {
            const uint32_t st = tj % KST, b = tj & 1u;
            if (!mbar_wait(BAR(C::B_KFULL + st), (tj / KST) & 1u, abort_flag)) return false;
            if (!mbar_wait(BAR(C::B_SFREE + b), ((tj >> 1) & 1u) ^ 1u, abort_flag)) return false;
            tc_fence_after();
            const uint32_t kb = sK + st * C::KVBYTES;
#pragma unroll
            for (int kk = 0; kk < DH / 16; ++kk) {
                const uint32_t off = (uint32_t)((kk >> 2) * (BM * 128) + (kk & 3) * 32);
                const uint32_t offk = (uint32_t)((kk >> 2) * (BN * 128) + (kk & 3) * 32);
                tc_mma(tmem + S_COL0 + 128u * b, desc_sw128(sQ + off, 16, 1024),
                       desc_sw128(kb + offk, 16, 1024), ID_S, kk > 0 ? 1u : 0u);
            }
            tc_commit(BAR(C::B_SFULL + b));
            tc_commit(BAR(C::B_KEMPTY + st));
            return true;
        };
        bool ok = true;
        for (int it = blockIdx.x; it < n_items && ok; it += gridDim.x) {
            const WorkItem w = a.items[it];
            const int n = w.tile_end - w.tile_begin;
            if (n <= 0) continue;
            if (!mbar_wait(BAR(C::B_QFULL), icnt & 1u, abort_flag)) { ok = false; break; }
            ++icnt;
            tc_fence_after();
            if (!issue_s(tcnt)) { ok = false; break; }
            for (int j = 0; j < n; ++j) {
                const uint32_t tj = tcnt + (uint32_t)j;
                if (j + 1 < n && !issue_s(tj + 1)) { ok = false; break; }
                const uint32_t st = tj % KST;
                if (!mbar_wait(BAR(C::B_PFULL), tj & 1u, abort_flag)) { ok = false; break; }
                if (!mbar_wait(BAR(C::B_VFULL + st), (tj / KST) & 1u, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t vb = sV + st * C::KVBYTES;
#pragma unroll
                for (int kk = 0; kk < BN / 16; ++kk) {
                    const uint32_t offp = (uint32_t)((kk >> 2) * (BM * 128) + (kk & 3) * 32);
                    tc_mma(tmem, desc_sw128(sP + offp, 16, 1024),
                           desc_sw128(vb + (uint32_t)kk * 2048u, BN * 128, 1024), ID_PV,
                           (j > 0 || kk > 0) ? 1u : 0u);
                }
                tc_commit(BAR(C::B_PVDONE));
                tc_commit(BAR(C::B_VEMPTY + st));
            }
            tcnt += (uint32_t)n;
        }
        // every MMA issued by this thread completes before TMEM is released
        tc_commit(BAR(C::B_DRAIN));
        mbar_drain(BAR(C::B_DRAIN), 0);
    } else if (warp >= 4) {
        // ------------------------------------------------------------------
        // softmax / correction / epilogue: thread = query row
        // ------------------------------------------------------------------
        const int r = threadIdx.x - 128;              // 0..127 = TMEM lane
        const int wq = warp - 4;                      // TMEM lane quarter
        const uint32_t tl = tmem + ((uint32_t)(32 * wq) << 16);
        constexpr int CPR = DH / 8;                   // 16-byte chunks per query row
        constexpr int RPI = 32 / CPR;                 // rows per warp per step
        constexpr int QIT = BM / (4 * RPI);           // steps per warp
        uint32_t tcnt = 0;
        bool ok = true;
        for (int it = blockIdx.x; it < n_items && ok; it += gridDim.x) {
            const WorkItem w = a.items[it];
            const RangeSet rs = a.ranges[w.u];
            const int n = w.tile_end - w.tile_begin;
            const int g = a.unit_group[w.u];
            if (n > 0) {
                // gather q~ rows of this query tile into the swizzled Q tile
                const uint16_t *qg = static_cast<const uint16_t *>(a.q) + (int64_t)g * a.mn * a.D + w.h * DH;
#pragma unroll 1
                for (int i0 = 0; i0 < QIT; i0 += 8) {
                    uint4 v[8];
                    int rr[8];
#pragma unroll
                    for (int u8 = 0; u8 < 8; ++u8) {
                        const int i = i0 + u8;
                        v[u8] = make_uint4(0, 0, 0, 0);
                        rr[u8] = -1;
                        if (i < QIT) {
                            const int row = (i * 4 + wq) * RPI + lane / CPR;
                            const int ch = lane % CPR;
                            rr[u8] = row;
                            const int jrow = w.qt * BM + row;
                            if (jrow < rs.cnt) {
                                int cell = a.idx[(int64_t)w.u * a.k_max + jrow];
                                cell = (cell < 0 || cell >= a.mn) ? 0 : cell;
                                v[u8] = __ldg(reinterpret_cast<const uint4 *>(qg + (int64_t)cell * a.D + ch * 8));
                                if (a.rope) {
                                    const float4 *f = reinterpret_cast<const float4 *>(
                                        a.rope + ((int64_t)cell * (DH / 2) + ch * 4) * 2);
                                    const float4 f0 = __ldg(f), f1 = __ldg(f + 1);
                                    const float cs[4] = {f0.x, f0.z, f1.x, f1.z};
                                    const float sn[4] = {f0.y, f0.w, f1.y, f1.w};
                                    uint32_t wv[4] = {v[u8].x, v[u8].y, v[u8].z, v[u8].w};
#pragma unroll
                                    for (int p = 0; p < 4; ++p) {
                                        const float x0 = __uint_as_float(wv[p] << 16);
                                        const float x1 = __uint_as_float(wv[p] & 0xffff0000u);
                                        wv[p] = pack_bf16x2(x0 * cs[p] - x1 * sn[p], x0 * sn[p] + x1 * cs[p]);
                                    }
                                    v[u8] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
                                }
                            }
                        }
                    }
#pragma unroll
                    for (int u8 = 0; u8 < 8; ++u8) {
                        if (rr[u8] < 0) continue;
                        const uint32_t off = sw128_offset(BM, rr[u8], lane % CPR);
                        asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(sQ + off), "r"(v[u8].x),
                                     "r"(v[u8].y), "r"(v[u8].z), "r"(v[u8].w) : "memory");
                    }
                }
                fence_proxy_async();
                mbar_arrive(BAR(C::B_QFULL));
            }
            const int jrow = w.qt * BM + r;
            const bool valid = jrow < rs.cnt;
            int cell = valid ? a.idx[(int64_t)w.u * a.k_max + jrow] : 0;
            cell = (cell < 0 || cell >= a.mn) ? 0 : cell;
            float m_run = -INFINITY, l_run = 0.f;
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
                uint32_t sr[BN];
#pragma unroll
                for (int c4 = 0; c4 < BN / 32; ++c4) tmem_ld32(tl + S_COL0 + 128u * b + 32u * c4, sr + 32 * c4);
                tmem_wait_ld();
                tc_fence_before();
                mbar_arrive(BAR(C::B_SFREE + b));
                float s[BN];
                float mt = -INFINITY;
#pragma unroll
                for (int c = 0; c < BN; ++c) {
                    s[c] = c < nvalid ? __uint_as_float(sr[c]) * a.scale_log2 : -INFINITY;
                    mt = fmaxf(mt, s[c]);
                }
                const float m_new = (j == 0) ? mt : (mt > m_run + 8.0f ? mt : m_run);
                float rowsum = 0.f;
                uint32_t pk[BN / 2];
#pragma unroll
                for (int c = 0; c < BN / 2; ++c) {
                    const float p0 = exp2f(s[2 * c] - m_new);
                    const float p1 = exp2f(s[2 * c + 1] - m_new);
                    rowsum += p0 + p1;
                    pk[c] = pack_bf16x2(p0, p1);
                }
                if (j > 0) {
                    // P_{j-1} consumed and O final for tile j-1
                    if (!__all_sync(0xffffffffu, mbar_wait(BAR(C::B_PVDONE), (tj - 1u) & 1u, abort_flag))) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const bool grow = m_new != m_run;
                    const float alpha = grow ? exp2f(m_run - m_new) : 1.0f;
                    if (__any_sync(0xffffffffu, grow)) {
#pragma unroll 1
                        for (int c4 = 0; c4 < DH / 32; ++c4) {
                            uint32_t o[32];
                            tmem_ld32(tl + 32u * c4, o);
                            tmem_wait_ld();
#pragma unroll
                            for (int e = 0; e < 32; ++e) o[e] = __float_as_uint(__uint_as_float(o[e]) * alpha);
                            tmem_st32(tl + 32u * c4, o);
                        }
                        tmem_wait_st();
                    }
                    l_run *= alpha;
                }
                l_run += rowsum;
                m_run = m_new;
#pragma unroll
                for (int cc = 0; cc < BN / 8; ++cc) {
                    const uint32_t off = sw128_offset(BM, r, cc);
                    asm volatile("st.shared.v4.b32 [%0], {%1, %2, %3, %4};" ::"r"(sP + off), "r"(pk[4 * cc]),
                                 "r"(pk[4 * cc + 1]), "r"(pk[4 * cc + 2]), "r"(pk[4 * cc + 3]) : "memory");
                }
                fence_proxy_async();
                tc_fence_before();
                mbar_arrive(BAR(C::B_PFULL));
            }
            if (!ok) break;
            if (n > 0) {
                if (!__all_sync(0xffffffffu,
                                mbar_wait(BAR(C::B_PVDONE), (tcnt + (uint32_t)n - 1u) & 1u, abort_flag))) {
                    ok = false;
                    break;
                }
                tc_fence_after();
            }
            tcnt += (uint32_t)n;
            // epilogue
            const float inv = l_run > 0.f ? 1.0f / l_run : 0.f;
#pragma unroll 1
            for (int c4 = 0; c4 < DH / 32; ++c4) {
                uint32_t o[32];
                if (n > 0) {
                    tmem_ld32(tl + 32u * c4, o);
                    tmem_wait_ld();
                } else {
#pragma unroll
                    for (int e = 0; e < 32; ++e) o[e] = 0u;
                }
                if (!valid) continue;
                if (w.slot < 0) {
                    const int64_t off = ((int64_t)w.u * a.mn + cell) * a.D + w.h * DH + 32 * c4;
                    float res[32];
                    if (a.residual) {
                        const uint4 *rp = reinterpret_cast<const uint4 *>(static_cast<const uint16_t *>(a.residual) + off);
#pragma unroll
                        for (int q4 = 0; q4 < 4; ++q4) {
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
                        for (int e = 0; e < 32; ++e) res[e] = 0.f;
                    }
                    uint4 *dp = reinterpret_cast<uint4 *>(static_cast<uint16_t *>(a.out) + off);
#pragma unroll
                    for (int q4 = 0; q4 < 4; ++q4) {
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
                    float4 *po = reinterpret_cast<float4 *>(a.part_o + ((int64_t)w.slot * BM + r) * DH + 32 * c4);
#pragma unroll
                    for (int q4 = 0; q4 < 8; ++q4)
                        po[q4] = make_float4(__uint_as_float(o[4 * q4]), __uint_as_float(o[4 * q4 + 1]),
                                             __uint_as_float(o[4 * q4 + 2]), __uint_as_float(o[4 * q4 + 3]));
                }
            }
            if (valid && w.slot >= 0)
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

bool make_kv_map(CUtensorMap *m, const void *store, int64_t D, int64_t rows)
{
    PFN_cuTensorMapEncodeTiled_v12000 enc = encode_fn();
    if (!enc) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)D, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)D * 2};
    const cuuint32_t box[2] = {64, (cuuint32_t)BN};
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
    if (!make_kv_map(&mk, a.k_store, a.D, rows) || !make_kv_map(&mv, a.v_store, a.D, rows)) return RS3_ECUDA;
    int64_t grid = a.max_items;
    if (grid > a.n_sm) grid = a.n_sm;
    if (grid < 1) grid = 1;
    k_readout_tc<DH><<<(unsigned)grid, NTHREADS, Cfg<DH>::SMEM, st>>>(a, mk, mv);
    return cudaGetLastError() == cudaSuccess ? RS3_OK : RS3_ECUDA;
}

}  // namespace tc

bool rs3_tc_supported(int d) { return d == 64 || d == 128 || d == 256; }
int rs3_tc_block_n(int d) { (void)d; return tc::BN; }

rs3_status rs3_launch_tc_readout(const ReadoutArgs &a, cudaStream_t st)
{
    switch (a.d) {
    case 64: return tc::launch<64>(a, st);
    case 128: return tc::launch<128>(a, st);
    case 256: return tc::launch<256>(a, st);
    default: return RS3_EUNSUPPORTED;
    }
}
