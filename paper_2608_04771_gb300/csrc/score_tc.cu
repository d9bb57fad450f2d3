// score_tc.cu -- tensor-core (tcgen05) passes of the Eq. 2 cache scores for bf16 caches.
//
// Both passes are persistent (one CTA per SM walking a contiguous range of (unit,
// 2048-key chunk) items, barrier phases running on across items) with these roles:
//   warp 0  lane 0 : TMA producer (window queries once per unit, then a ring of K tiles)
//   warp 1         : allocates 512 TMEM columns; lane 0 issues tcgen05.mma (bf16 in,
//                    fp32 accumulate in TMEM) and commits to mbarriers
//   warps 2-3      : pass 2 only: add the epilogue groups' partial column sums of a tile
//                    in a fixed order and store them
//   warps 4..      : epilogue warp groups, reading accumulators with tcgen05.ld (one TMEM
//                    lane per thread) into the softmax arithmetic
// Operands sit in shared memory in the 128-byte-swizzled K-major layout the TMA writes
// (rows of 64 bf16, 8-row atoms of 1024 bytes); each MMA takes a K=16 slice.  The
// accumulators rotate through a ring of TMEM buffers, so the MMAs of the next tiles run
// while the epilogue groups work on earlier ones.
//
// Pass 1 (row statistics): queries on M (128-row tiles), keys on N, so each thread owns
//   one window row and keeps a running (reference, sum) over the chunk's keys.  The
//   epilogue groups split each tile's key columns and leave one partial each.  A full tile
//   is exponentiated against the row's current reference without a max pass; only a
//   row's first tile, a masked tile, or a tile whose sum could overflow takes its max.
// Pass 2 (column sums): keys on M (128 per tile), queries on N, split into up to four
//   column blocks, one per epilogue group, so each thread sums 2^(c*l - b_r) over its
//   block's window rows for one key; warps 2-3 add the groups' partials.
// Every mbarrier wait is bounded; a wait that runs out sets the device error word and
// the CTA stops issuing work, waits (bounded) for nothing further and frees its TMEM.
#include <cuda.h>

#include "common.cuh"
#include "internal.h"
#include "tma.cuh"

namespace reco {

// ---------------------------------------------------------------- tcgen05 wrappers
__device__ __forceinline__ void tmem_alloc(uint32_t dst_smem, uint32_t ncols)
{
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(dst_smem), "r"(ncols)
                 : "memory");
}
__device__ __forceinline__ void tmem_relinquish()
{
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols)
{
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols) : "memory");
}
__device__ __forceinline__ void tc_fence_before() { asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_fence_after() { asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory"); }
__device__ __forceinline__ void tc_commit(uint32_t bar)
{
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
                 : "memory");
}
// D[tmem] (+)= A[smem desc] * B[smem desc]^T, kind::f16 (both operands bf16 here).
__device__ __forceinline__ void tc_mma(uint32_t dtmem, uint64_t adesc, uint64_t bdesc, uint32_t idesc,
                                       uint32_t accumulate)
{
    asm volatile(
        "{\n .reg .pred p;\n setp.ne.b32 p, %4, 0;\n"
        " tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n}" ::"r"(dtmem),
        "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
        : "memory");
}
// 32 consecutive fp32 columns of the calling thread's TMEM lane (no wait: call
// tmem_ld_wait() before using the values).
__device__ __forceinline__ void tmem_ld32_nowait(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}
__device__ __forceinline__ void tmem_ld_wait() { asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory"); }

// 16 consecutive fp32 columns of the calling thread's TMEM lane (no wait).
__device__ __forceinline__ void tmem_ld16_nowait(uint32_t taddr, float (&v)[16])
{
    uint32_t r[16];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x16.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15}, [%16];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15])
        : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 16; ++i) v[i] = __uint_as_float(r[i]);
}

// Wait for this thread's TMEM loads, then pass the NV loaded registers through an empty
// asm so that no use of them can be scheduled before the wait.
template <int NV>
__device__ __forceinline__ void tmem_ld_wait_regs(float *v)
{
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < NV; i += 8)
        asm volatile(""
                     : "+f"(v[i]), "+f"(v[i + 1]), "+f"(v[i + 2]), "+f"(v[i + 3]), "+f"(v[i + 4]), "+f"(v[i + 5]),
                       "+f"(v[i + 6]), "+f"(v[i + 7]));
}

// 32 consecutive fp32 columns of the calling thread's TMEM lane.
__device__ __forceinline__ void tmem_ld32(uint32_t taddr, float (&v)[32])
{
    uint32_t r[32];
    asm volatile(
        "tcgen05.ld.sync.aligned.32x32b.x32.b32 {%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
        "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
        : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7]),
          "=r"(r[8]), "=r"(r[9]), "=r"(r[10]), "=r"(r[11]), "=r"(r[12]), "=r"(r[13]), "=r"(r[14]), "=r"(r[15]),
          "=r"(r[16]), "=r"(r[17]), "=r"(r[18]), "=r"(r[19]), "=r"(r[20]), "=r"(r[21]), "=r"(r[22]), "=r"(r[23]),
          "=r"(r[24]), "=r"(r[25]), "=r"(r[26]), "=r"(r[27]), "=r"(r[28]), "=r"(r[29]), "=r"(r[30]), "=r"(r[31])
        : "r"(taddr));
    asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
    for (int i = 0; i < 32; ++i) v[i] = __uint_as_float(r[i]);
}

// Shared-memory matrix descriptor: K-major operand, 128-byte swizzle, 8-row atoms of
// 1024 bytes (stride byte offset 1024), descriptor version 1.  The start address sits in
// the low 14 bits as address / 16; a shared-memory address stays below 2^18 bytes, so
// the descriptor of (address + offset) is this one plus offset / 16 (no carry out).
__device__ __forceinline__ uint64_t sw128_desc(uint32_t saddr)
{
    uint64_t d = 0;
    d |= (uint64_t)((saddr >> 4) & 0x3FFFu);
    d |= (uint64_t)1u << 16;            // leading byte offset (unused for swizzled K-major)
    d |= (uint64_t)(1024u >> 4) << 32;  // stride byte offset
    d |= (uint64_t)1u << 46;            // version
    d |= (uint64_t)2u << 61;            // SWIZZLE_128B
    return d;
}

// Instruction descriptor, kind::f16: bf16 A and B (K-major), fp32 D, shape M x N.
__host__ __device__ constexpr uint32_t idesc_bf16(int M, int N)
{
    return (1u << 4) | (1u << 7) | (1u << 10) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

constexpr long long kTcSpin = 1LL << 24;
constexpr int kTcMaxR = 512;  // window rows (G*w) the tensor-core passes take
constexpr int kTmemCols = 512;

__device__ __forceinline__ bool wait_or_flag(uint32_t bar, uint32_t parity, volatile int *abort_flag,
                                             unsigned *err)
{
    for (long long i = 0; i < kTcSpin; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 1023) == 1023 && *abort_flag) return false;
    }
    *abort_flag = 1;
    raise_error(err, ERR_INTERNAL);
    return false;
}

// TMEM columns between pass-2 accumulator buffers: a block's width rounded up to 32.
__host__ __device__ constexpr int p2_stride(int cb) { return (cb + 31) & ~31; }

// ---------------------------------------------------------------- work items
// A CTA walks a contiguous range of (unit, 2048-key chunk) items in unit order, so its
// window queries change only when the unit does.  Item i covers unit i / n_chunks, or,
// when a unit list is given (a masked call), unit ulist[i / n_chunks]: the ranges are
// then cut from the scored units only, which keeps the CTAs evenly loaded.
struct ChunkItem {
    long u;
    int chunk, L, j0, j1, ntiles;
    bool valid;  // the unit's length is in range
};

__device__ __forceinline__ ChunkItem chunk_item(int i, int n_chunks, const int32_t *ulist, const int32_t *lens,
                                               int w, int L_cap, bool candidates_only, int tile)
{
    ChunkItem it;
    it.u = ulist ? ulist[i / n_chunks] : i / n_chunks;
    it.chunk = i % n_chunks;
    it.L = lens[it.u];
    it.valid = it.L >= w && it.L <= L_cap;
    const int end = it.valid ? (candidates_only ? it.L - w : it.L) : 0;
    it.j0 = it.chunk * kScoreChunk;
    it.j1 = min(it.j0 + kScoreChunk, end);
    it.ntiles = it.j0 < it.j1 ? (it.j1 - it.j0 + tile - 1) / tile : 0;
    return it;
}

// ---------------------------------------------------------------- column ranges
// 8 consecutive fp32 columns of the calling thread's TMEM lane (no wait).
__device__ __forceinline__ void tmem_ld8_nowait(uint32_t taddr, float *v)
{
    uint32_t r[8];
    asm volatile("tcgen05.ld.sync.aligned.32x32b.x8.b32 {%0,%1,%2,%3,%4,%5,%6,%7}, [%8];"
                 : "=r"(r[0]), "=r"(r[1]), "=r"(r[2]), "=r"(r[3]), "=r"(r[4]), "=r"(r[5]), "=r"(r[6]), "=r"(r[7])
                 : "r"(taddr));
#pragma unroll
    for (int i = 0; i < 8; ++i) v[i] = __uint_as_float(r[i]);
}
// Split n columns (a multiple of 8) into `parts` contiguous ranges of multiples of 8.
__host__ __device__ __forceinline__ int split8_lo(int n, int parts, int g) { return ((n / 8) * g / parts) * 8; }

// ---------------------------------------------------------------- pass 1: row statistics
// A piece is the accumulator of one 128-row query tile mt against one tile of N keys; the
// pieces of a key tile gt are p = gt * MT + mt, in a ring of NR TMEM regions of N columns.
// The 4 * EG epilogue warps of query tile mt split the N columns into EG ranges.
template <int D, int MT, int N, int EG>
struct Pass1Cfg {
    static constexpr int HALVES = D / 64;
    static constexpr int QBOX = 128 * 128;  // 128 rows x 128 bytes
    static constexpr int KBOX = N * 128;
    static constexpr int KSTAGE = HALVES * KBOX;
    static constexpr int NR = kTmemCols / N;  // TMEM regions
    static constexpr int CW = N / EG;         // columns per epilogue group
    static constexpr int QBYTES = MT * HALVES * QBOX;
    static constexpr int NS0 = (200 * 1024 - QBYTES) / KSTAGE;
    static constexpr int NS = NS0 > 8 ? 8 : NS0;
    static constexpr size_t SMEM = 1024 + (size_t)QBYTES + (size_t)NS * KSTAGE;
    static_assert(NR >= MT || NR >= 2, "accumulator ring too short");
    static constexpr int THREADS = 128 + 128 * MT * EG;
    static_assert(CW % 32 == 0, "epilogue group width");
    static_assert(NS >= 2, "K ring too short");
    static_assert(THREADS <= 1024, "too many warps");
};

// Exponent of a normal positive float, as an integer power of two.
__device__ __forceinline__ int exp2_of(float z) { return ((__float_as_int(z) >> 23) & 0xff) - 127; }

// One row's running (reference m, sum z) over 32 accumulator columns v (logit = v * c2 in
// log2 units), of which columns 0..lim are visible.  A full batch is exponentiated against
// the current reference with no max pass; the row's first batch, a masked batch, or one
// whose sum could overflow takes its max first.  z is kept below 2^64 by moving m up.
__device__ __forceinline__ void rowstats_batch(const float (&v)[32], int lim, float c2, float &m, float &z)
{
    const bool full = lim >= 31;
    bool exact = !full || m == -INFINITY;
    if (!exact) {
        const float nb = -m;
        float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int q = 0; q < 32; ++q) a4[q & 3] += fast_exp2(fmaf(v[q], c2, nb));
        const float sum = (a4[0] + a4[1]) + (a4[2] + a4[3]);
        if (sum <= 0x1p96f)
            z += sum;
        else
            exact = true;  // a term too far above the reference (or NaN): redo exactly
    }
    if (exact) {
        float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
#pragma unroll
        for (int q = 0; q < 32; ++q)
            if (full || q <= lim) mx4[q & 3] = fmaxf(mx4[q & 3], v[q]);
        const float mx = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
        const float mn = fmaxf(m, mx * c2);
        if (mn == -INFINITY) return;
        const float nb = -mn;
        float a4[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
        for (int q = 0; q < 32; ++q) a4[q & 3] += (full || q <= lim) ? fast_exp2(fmaf(v[q], c2, nb)) : 0.f;
        z = z * fast_exp2(m - mn) + ((a4[0] + a4[1]) + (a4[2] + a4[3]));
        m = mn;
    }
    if (z > 0x1p64f) {  // move the reference up by a power of two: exact rescale
        const int k = exp2_of(z);
        z = __int_as_float(__float_as_int(z) - (k << 23));
        m += (float)k;
    }
}

template <int D, int MT, int N, int EG>
__global__ void __launch_bounds__(Pass1Cfg<D, MT, N, EG>::THREADS, 1)
    score_rowstats_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const int32_t *__restrict__ lens, int w, int G, int Hq, int Hkv, int L_cap, int R,
                      int n_chunks, int n_items, const int32_t *__restrict__ ulist, const int32_t *__restrict__ ucount,
                      float c2, float *__restrict__ part_m, float *__restrict__ part_z, unsigned *err)
{
    using C = Pass1Cfg<D, MT, N, EG>;
    constexpr int HALVES = C::HALVES, QBOX = C::QBOX, KBOX = C::KBOX, KSTAGE = C::KSTAGE;
    constexpr int NR = C::NR, NS = C::NS, CW = C::CW, NBT = CW / 32;
    constexpr bool PIPE = C::THREADS <= 640;  // registers for two column batches per thread
    constexpr uint32_t IDESC = idesc_bf16(128, N);
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bar_qfull, bar_qempty, bar_kfull[NS], bar_kempty[NS], bar_afull[NR],
        bar_aempty[NR];
    __shared__ uint32_t tmem_sh;
    __shared__ int abort_sh;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const uint32_t raw0 = smem_addr(smem_raw);
    const uint32_t base = (raw0 + 1023u) & ~1023u;
    const uint32_t Qs = base;                // MT x HALVES x QBOX
    const uint32_t Ks = base + C::QBYTES;  // NS x KSTAGE
    if (tid == 0) {
        mbar_init(smem_addr(&bar_qfull), 1);
        mbar_init(smem_addr(&bar_qempty), 1);
        for (int s = 0; s < NS; ++s) {
            mbar_init(smem_addr(&bar_kfull[s]), 1);
            mbar_init(smem_addr(&bar_kempty[s]), 1);
        }
        for (int b = 0; b < NR; ++b) {
            mbar_init(smem_addr(&bar_afull[b]), 1);
            mbar_init(smem_addr(&bar_aempty[b]), 4 * EG);
        }
        abort_sh = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        fence_async_shared();
    }
    if (warp == 1) {
        tmem_alloc(smem_addr(&tmem_sh), kTmemCols);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;
    volatile int *abort_flag = &abort_sh;
    // everything above runs while the previous kernel drains; from here on its outputs
    // (the unit list, the row normalisers, the window queries) are read
    wait_prior_grid();
    const int n_it = ucount ? *ucount * n_chunks : n_items;  // items of the scored units
    const int i_begin = (int)((long long)blockIdx.x * n_it / gridDim.x);
    const int i_end = (int)((long long)(blockIdx.x + 1) * n_it / gridDim.x);

    if (warp == 0) {
        if (lane == 0) {  // producer: queries when the unit changes, then the chunk's K tiles
            int gt = 0, nq = 0;
            long prev_u = -1;
            bool ok = true;
            for (int i = i_begin; ok && i < i_end; ++i) {
                const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, false, N);
                if (it.ntiles == 0) continue;
                if (it.u != prev_u) {
                    if (nq > 0 && !wait_or_flag(smem_addr(&bar_qempty), (nq - 1) & 1, abort_flag, err)) break;
                    const long lb = it.u / Hkv;
                    const int q_row0 = (int)((lb * Hq + (it.u % Hkv) * G) * w);
                    mbar_expect_tx(smem_addr(&bar_qfull), (uint32_t)C::QBYTES);
                    for (int mt = 0; mt < MT; ++mt)
                        for (int hh = 0; hh < HALVES; ++hh)
                            tma_load_2d(Qs + (mt * HALVES + hh) * QBOX, &tmQ, 64 * hh, q_row0 + 128 * mt,
                                        smem_addr(&bar_qfull));
                    ++nq;
                    prev_u = it.u;
                }
                const int k_row0 = (int)(it.u * L_cap + it.j0);
                for (int t = 0; t < it.ntiles; ++t, ++gt) {
                    const int s = gt % NS;
                    if (!wait_or_flag(smem_addr(&bar_kempty[s]), ((gt / NS) & 1) ^ 1, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(smem_addr(&bar_kfull[s]), KSTAGE);
                    for (int hh = 0; hh < HALVES; ++hh)
                        tma_load_2d(Ks + s * KSTAGE + hh * KBOX, &tmK, 64 * hh, k_row0 + t * N,
                                    smem_addr(&bar_kfull[s]));
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {  // MMA issuer
            int gt = 0, nq = 0;
            long prev_u = -1;
            bool ok = true;
            for (int i = i_begin; ok && i < i_end; ++i) {
                const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, false, N);
                if (it.ntiles == 0) continue;
                if (it.u != prev_u) {
                    if (nq > 0) tc_commit(smem_addr(&bar_qempty));  // queries free once prior MMAs land
                    if (!wait_or_flag(smem_addr(&bar_qfull), nq & 1, abort_flag, err)) break;
                    ++nq;
                    prev_u = it.u;
                }
                for (int t = 0; ok && t < it.ntiles; ++t, ++gt) {
                    const int s = gt % NS;
                    if (!wait_or_flag(smem_addr(&bar_kfull[s]), (gt / NS) & 1, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    for (int mt = 0; mt < MT; ++mt) {
                        const int p = gt * MT + mt, b = p % NR;
                        if (!wait_or_flag(smem_addr(&bar_aempty[b]), ((p / NR) & 1) ^ 1, abort_flag, err)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t d = tmem + (uint32_t)(b * N);
                        // descriptors of the first K slice; later slices add their offset / 16
                        const uint64_t ad0 = sw128_desc(Qs + mt * HALVES * QBOX);
                        const uint64_t bd0 = sw128_desc(Ks + s * KSTAGE);
#pragma unroll
                        for (int k = 0; k < D / 16; ++k) {
                            const int hh = k >> 2, kk = k & 3;
                            tc_mma(d, ad0 + (uint64_t)((hh * QBOX + kk * 32) >> 4),
                                   bd0 + (uint64_t)((hh * KBOX + kk * 32) >> 4), IDESC, k > 0 ? 1u : 0u);
                        }
                        tc_commit(smem_addr(&bar_afull[b]));
                    }
                    if (ok) tc_commit(smem_addr(&bar_kempty[s]));
                }
            }
        }
    } else if (warp >= 4) {  // epilogue: query tile mt, column group g, one window row per thread
        const int idx = (warp - 4) >> 2, mt = idx / EG, g = idx % EG, quarter = warp & 3;
        const int r = mt * 128 + quarter * 32 + lane;
        const bool warp_rows = mt * 128 + quarter * 32 < R;  // this warp holds real window rows
        const int t_row = r % w;
        const int c_lo = g * CW;
        int gt = 0;
        for (int i = i_begin; i < i_end; ++i) {
            const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, false, N);
            if (!it.valid) {
                if (it.chunk == 0 && r == 0 && g == 0) raise_error(err, ERR_LEN);
                continue;
            }
            const int jmax = it.L - w + t_row;  // last key this window row sees
            float m = -INFINITY, z = 0.f;       // reference (log2 units) and sum relative to it
            bool ok = true;
            for (int t = 0; t < it.ntiles; ++t, ++gt) {
                const int p = gt * MT + mt, b = p % NR;
                if (!wait_or_flag(smem_addr(&bar_afull[b]), (p / NR) & 1, abort_flag, err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t ta = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(b * N + c_lo);
                // batches of 32 columns; with PIPE the next batch's TMEM load is in flight while
                // one is summed (two register batches), else each batch is loaded, then summed
                float v[PIPE ? 2 : 1][32];
                if (warp_rows) {
                    tmem_ld32_nowait(ta, v[0]);
                    tmem_ld_wait_regs<32>(v[0]);
                }
#pragma unroll
                for (int k = 0; k < NBT; ++k) {
                    float(&cur)[32] = v[PIPE ? (k & 1) : 0];
                    if (k + 1 < NBT) {
                        if (PIPE && warp_rows) tmem_ld32_nowait(ta + 32 * (k + 1), v[PIPE ? ((k + 1) & 1) : 0]);
                    } else {  // every column of the piece read: release the region
                        tc_fence_before();
                        __syncwarp();
                        if (lane == 0) mbar_arrive(smem_addr(&bar_aempty[b]));
                    }
                    const int jb = it.j0 + t * N + c_lo + 32 * k;
                    const int lim = min(it.j1 - 1, jmax) - jb;  // columns 0..lim of this batch are visible
                    if (warp_rows && lim >= 0) rowstats_batch(cur, lim, c2, m, z);
                    if (k + 1 < NBT && warp_rows) {
                        if (!PIPE) tmem_ld32_nowait(ta + 32 * (k + 1), v[0]);
                        tmem_ld_wait_regs<32>(v[PIPE ? ((k + 1) & 1) : 0]);
                    }
                }
            }
            if (!ok) break;
            if (r < R) {
                const size_t o = (((size_t)it.u * n_chunks + it.chunk) * EG + g) * R + r;
                part_m[o] = m;
                part_z[o] = z;
            }
        }
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------- pass 2: column sums
// The NQ query columns of a key tile are one MMA chain (NP = 1, N = NQ <= 256) or two
// (NP = 2, N = NQ / 2); each chain's accumulator is a piece in a ring of NR TMEM regions.
// The four epilogue groups split every piece's columns into ranges of multiples of 8, so
// all 16 epilogue warps work on the same tile; warps 2-3 add the groups' partials.
constexpr int kP2Groups = 4;
constexpr int kP2Slots = 4;  // tiles whose partials may wait for the combining warps

// n (a multiple of 8, at most 32) columns into fixed register slots of v.
__device__ __forceinline__ void tmem_ld_upto32(uint32_t taddr, int n, float (&v)[32])
{
    if (n == 32) {
        tmem_ld32_nowait(taddr, v);
        return;
    }
#pragma unroll
    for (int k = 0; k < 4; ++k)
        if (8 * k < n) tmem_ld8_nowait(taddr + 8 * k, v + 8 * k);
}

// Release a TMEM region after this warp's last load of it.
__device__ __forceinline__ void colsum_release(int lane, uint64_t &bar)
{
    tc_fence_before();
    __syncwarp();
    if (lane == 0) mbar_arrive(smem_addr(&bar));
}

// a4 += sum over n columns (a multiple of 8) of 2^(v * c2 - b); b holds the rows'
// log2 normalisers (16-byte aligned), +inf for padding columns.
__device__ __forceinline__ void colsum_batch(const float (&v)[32], int n, const float *b, float c2, float (&a4)[4])
{
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        if (8 * k < n) {
            const float4 b0 = *reinterpret_cast<const float4 *>(b + 8 * k);
            const float4 b1 = *reinterpret_cast<const float4 *>(b + 8 * k + 4);
            a4[0] += fast_exp2(fmaf(v[8 * k + 0], c2, -b0.x));
            a4[1] += fast_exp2(fmaf(v[8 * k + 1], c2, -b0.y));
            a4[2] += fast_exp2(fmaf(v[8 * k + 2], c2, -b0.z));
            a4[3] += fast_exp2(fmaf(v[8 * k + 3], c2, -b0.w));
            a4[0] += fast_exp2(fmaf(v[8 * k + 4], c2, -b1.x));
            a4[1] += fast_exp2(fmaf(v[8 * k + 5], c2, -b1.y));
            a4[2] += fast_exp2(fmaf(v[8 * k + 6], c2, -b1.z));
            a4[3] += fast_exp2(fmaf(v[8 * k + 7], c2, -b1.w));
        }
    }
}

template <int D>
__global__ void __launch_bounds__(128 + 128 * kP2Groups, 1)
    score_colsum_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    const int32_t *__restrict__ lens, int w, int G, int Hq, int Hkv, int L_cap, int R, int NQ, int NP,
                    int NR, int NS, int n_chunks, int n_items, const int32_t *__restrict__ ulist,
                    const int32_t *__restrict__ ucount, float c2, const float *__restrict__ rowb,
                    const float *__restrict__ row_lse, long rows_q, float *__restrict__ raw, unsigned *err)
{
    constexpr int HALVES = D / 64;
    constexpr int KBOX = 128 * 128;  // 128 keys x 128 bytes
    constexpr int KSTAGE = HALVES * KBOX;
    constexpr int EG = kP2Groups, S = kP2Slots;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bar_qfull, bar_qempty, bar_kfull[4], bar_kempty[4], bar_afull[4],
        bar_aempty[4], bar_cfull[S], bar_cempty[S];
    __shared__ uint32_t tmem_sh;
    __shared__ int abort_sh;
    __shared__ __align__(16) float bsh[4 * EG][128];  // per epilogue warp: normalisers of its columns
    __shared__ float cpart[S][EG][128];  // per tile slot: each group's partial column sums

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int NW = NQ / NP;                     // columns of one piece
    const int stride = (NW + 31) & ~31;         // TMEM columns between regions
    const uint32_t raw0 = smem_addr(smem_raw);
    const uint32_t base = (raw0 + 1023u) & ~1023u;
    const uint32_t QBOXB = (uint32_t)NQ * 128;  // one half (64 columns) of all NQ query rows
    const uint32_t Qs = base;
    const uint32_t Ks = base + HALVES * QBOXB;
    if (tid == 0) {
        mbar_init(smem_addr(&bar_qfull), 1);
        mbar_init(smem_addr(&bar_qempty), 1);
        for (int s = 0; s < NS; ++s) {
            mbar_init(smem_addr(&bar_kfull[s]), 1);
            mbar_init(smem_addr(&bar_kempty[s]), 1);
        }
        for (int b = 0; b < NR; ++b) {
            mbar_init(smem_addr(&bar_afull[b]), 1);
            mbar_init(smem_addr(&bar_aempty[b]), 4 * EG);
        }
        for (int s = 0; s < S; ++s) {
            mbar_init(smem_addr(&bar_cfull[s]), 4 * EG);
            mbar_init(smem_addr(&bar_cempty[s]), 2);
        }
        abort_sh = 0;
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        fence_async_shared();
    }
    if (warp == 1) {
        tmem_alloc(smem_addr(&tmem_sh), kTmemCols);
        tmem_relinquish();
    }
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = tmem_sh;
    volatile int *abort_flag = &abort_sh;
    // everything above runs while the previous kernel drains; from here on its outputs
    // (the unit list, the row normalisers, the window queries) are read
    wait_prior_grid();
    const int n_it = ucount ? *ucount * n_chunks : n_items;  // items of the scored units
    const int i_begin = (int)((long long)blockIdx.x * n_it / gridDim.x);
    const int i_end = (int)((long long)(blockIdx.x + 1) * n_it / gridDim.x);

    if (warp == 0) {
        if (lane == 0) {  // producer
            const int qbox_rows = NQ > 256 ? NQ / 2 : NQ;
            int s = 0, kph = 0, nq = 0;  // K stage and the parity of its round
            long prev_u = -1;
            bool ok = true;
            for (int i = i_begin; ok && i < i_end; ++i) {
                const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, true, 128);
                if (it.ntiles == 0) continue;
                if (it.u != prev_u) {
                    if (nq > 0 && !wait_or_flag(smem_addr(&bar_qempty), (nq - 1) & 1, abort_flag, err)) break;
                    const long lb = it.u / Hkv;
                    const int q_row0 = (int)((lb * Hq + (it.u % Hkv) * G) * w);
                    mbar_expect_tx(smem_addr(&bar_qfull), HALVES * QBOXB);
                    for (int hh = 0; hh < HALVES; ++hh)
                        for (int r0 = 0; r0 < NQ; r0 += qbox_rows)
                            tma_load_2d(Qs + hh * QBOXB + r0 * 128, &tmQ, 64 * hh, q_row0 + r0, smem_addr(&bar_qfull));
                    ++nq;
                    prev_u = it.u;
                }
                const int k_row0 = (int)(it.u * L_cap + it.j0);
                for (int t = 0; t < it.ntiles; ++t) {
                    if (!wait_or_flag(smem_addr(&bar_kempty[s]), kph ^ 1, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(smem_addr(&bar_kfull[s]), KSTAGE);
                    for (int hh = 0; hh < HALVES; ++hh)
                        tma_load_2d(Ks + s * KSTAGE + hh * KBOX, &tmK, 64 * hh, k_row0 + t * 128,
                                    smem_addr(&bar_kfull[s]));
                    if (++s == NS) {
                        s = 0;
                        kph ^= 1;
                    }
                }
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {  // MMA issuer: one chain per piece
            const uint32_t idesc = idesc_bf16(128, NW);
            int s = 0, kph = 0, b = 0, aph = 0, nq = 0;  // K stage, accumulator region, their parities
            long prev_u = -1;
            bool ok = true;
            for (int i = i_begin; ok && i < i_end; ++i) {
                const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, true, 128);
                if (it.ntiles == 0) continue;
                if (it.u != prev_u) {
                    if (nq > 0) tc_commit(smem_addr(&bar_qempty));
                    if (!wait_or_flag(smem_addr(&bar_qfull), nq & 1, abort_flag, err)) break;
                    ++nq;
                    prev_u = it.u;
                }
                for (int t = 0; ok && t < it.ntiles; ++t) {
                    if (!wait_or_flag(smem_addr(&bar_kfull[s]), kph, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    for (int h = 0; h < NP; ++h) {
                        if (!wait_or_flag(smem_addr(&bar_aempty[b]), aph ^ 1, abort_flag, err)) {
                            ok = false;
                            break;
                        }
                        tc_fence_after();
                        const uint32_t d = tmem + (uint32_t)(b * stride);
                        // descriptors of the first K slice; later slices add their offset / 16
                        const uint64_t ad0 = sw128_desc(Ks + s * KSTAGE);
                        const uint64_t bd0 = sw128_desc(Qs + h * NW * 128);
                        const uint64_t bh16 = (uint64_t)(QBOXB >> 4);
#pragma unroll
                        for (int k = 0; k < D / 16; ++k) {
                            const int hh = k >> 2, kk = k & 3;
                            tc_mma(d, ad0 + (uint64_t)((hh * KBOX + kk * 32) >> 4), bd0 + hh * bh16 + (uint64_t)(kk * 2),
                                   idesc, k > 0 ? 1u : 0u);
                        }
                        tc_commit(smem_addr(&bar_afull[b]));
                        if (++b == NR) {
                            b = 0;
                            aph ^= 1;
                        }
                    }
                    if (ok) tc_commit(smem_addr(&bar_kempty[s]));
                    if (++s == NS) {
                        s = 0;
                        kph ^= 1;
                    }
                }
            }
        }
    } else if (warp == 2 || warp == 3) {  // combine the groups' partials of each tile, in group order
        const int k0 = (warp - 2) * 32 + lane;  // keys k0 and k0 + 64 of the tile
        const float invG = 1.f / (float)G;
        int gt = 0;
        bool ok = true;
        for (int i = i_begin; ok && i < i_end; ++i) {
            const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, true, 128);
            for (int t = 0; t < it.ntiles; ++t, ++gt) {
                const int sl = gt % S;
                if (!wait_or_flag(smem_addr(&bar_cfull[sl]), (gt / S) & 1, abort_flag, err)) {
                    ok = false;
                    break;
                }
#pragma unroll
                for (int h = 0; h < 2; ++h) {
                    const int k = k0 + 64 * h;
                    const float acc = ((cpart[sl][0][k] + cpart[sl][1][k]) + cpart[sl][2][k]) + cpart[sl][3][k];
                    const int j = it.j0 + t * 128 + k;
                    if (j < it.j1) raw[it.u * L_cap + j] = acc * invG;
                }
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&bar_cempty[sl]));
            }
        }
    } else if (warp >= 4) {  // epilogue: group g sums its column range of every piece, one key per thread
        const int g = (warp - 4) >> 2, quarter = warp & 3;
        const int row = quarter * 32 + lane;  // key within the tile
        const int c_lo = split8_lo(NW, EG, g), nc = split8_lo(NW, EG, g + 1) - c_lo;
        float *bs = bsh[warp - 4];
        int gt = 0, b = 0, aph = 0;  // tile count; accumulator region and its parity
        long prev_u = -1;
        bool ok = true;
        for (int i = i_begin; ok && i < i_end; ++i) {
            const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, true, 128);
            if (it.ntiles == 0) continue;
            if (it.u != prev_u) {  // this unit's row normalisers of the group's columns (warp-private);
                __syncwarp();          // +inf for padding columns, which then add exp2(-inf) = 0
                for (int q = lane; q < NP * 64; q += 32) {
                    const int h = q >> 6, c = q & 63, rr = h * NW + c_lo + c;
                    float b = INFINITY;
                    if (c < nc && rr < R) {
                        if (row_lse != nullptr) {  // row (g, t) of the window: the decode's lse of that query
                            const long qi = (it.u / Hkv) * Hq + (it.u % Hkv) * G + rr / w;
                            const float l = row_lse[(long)(rr % w) * rows_q + qi];
                            if (isfinite(l)) {
                                b = l * kLog2e;
                            } else {  // the row adds nothing; the device error word says why
                                raise_error(err, ERR_NORM);
                            }
                        } else {
                            b = rowb[it.u * R + rr];
                        }
                    }
                    bs[q] = b;
                }
                __syncwarp();
                prev_u = it.u;
            }
            for (int t = 0; t < it.ntiles; ++t, ++gt) {
                float a4[4] = {0.f, 0.f, 0.f, 0.f};
                for (int h = 0; h < NP; ++h) {
                    if (!wait_or_flag(smem_addr(&bar_afull[b]), aph, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    const uint32_t ta = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(b * stride + c_lo);
                    const float *bh = bs + h * 64;
                    // up to two batches of 32 columns; the second one's load overlaps the first's sums
                    float v[2][32];
                    const int n0 = min(nc, 32), n1 = nc - n0;
                    tmem_ld_upto32(ta, n0, v[0]);
                    tmem_ld_wait_regs<32>(v[0]);
                    if (n1 > 0) tmem_ld_upto32(ta + 32, n1, v[1]);
                    else colsum_release(lane, bar_aempty[b]);
                    colsum_batch(v[0], n0, bh, c2, a4);
                    if (n1 > 0) {
                        tmem_ld_wait_regs<32>(v[1]);
                        colsum_release(lane, bar_aempty[b]);
                        colsum_batch(v[1], n1, bh + 32, c2, a4);
                    }
                    if (++b == NR) {
                        b = 0;
                        aph ^= 1;
                    }
                }
                if (!ok) break;
                const int sl = gt % S;
                if (!wait_or_flag(smem_addr(&bar_cempty[sl]), ((gt / S) & 1) ^ 1, abort_flag, err)) {
                    ok = false;
                    break;
                }
                cpart[sl][g][row] = (a4[0] + a4[1]) + (a4[2] + a4[3]);
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&bar_cfull[sl]));
            }
        }
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------- host side

// Pass 2's pieces: NQ = R rounded up to 16 (to 32 above 256 rows), one MMA chain of N = NQ
// per key tile, or two of N = NQ / 2 above 256 rows; NR TMEM regions of those columns.
struct P2Shape {
    int NQ, NP, NR;
};
static P2Shape p2_shape(int R)
{
    P2Shape p;
    p.NQ = R > 256 ? ((R + 31) / 32) * 32 : ((R + 15) / 16) * 16;
    p.NP = p.NQ > 256 ? 2 : 1;
    const int nw = p.NQ / p.NP;
    p.NR = min(4, kTmemCols / p2_stride(nw));
    return p;
}

bool score_tc_supported(const reco_kv &kv, int w)
{
    const long long R = (long long)(kv.H_q / kv.H_kv) * w;
    const unsigned long long k_rows = (unsigned long long)kv.n_layers * kv.B * kv.H_kv * kv.L_cap;
    const unsigned long long q_rows = (unsigned long long)kv.n_layers * kv.B * kv.H_q * w;
    return kv.dtype == RECO_BF16 && (kv.d == 64 || kv.d == 128) && R <= kTcMaxR && k_rows < (1ull << 31) &&
           q_rows < (1ull << 31);
}

// Pass-1 epilogue groups for R window rows (partials per chunk: the combine merges them).
int score_tc_pass1_groups(int R) { return (R + 127) / 128 >= 4 ? 1 : 2; }

template <int D, int MT, int N, int EG>
static cudaError_t run_pass1(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                             float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool *ok)
{
    using C = Pass1Cfg<D, MT, N, EG>;
    const long units = (long)kv.n_layers * kv.B * kv.H_kv;
    const int R = (kv.H_q / kv.H_kv) * w;
    const int nch = (kv.L_cap + kScoreChunk - 1) / kScoreChunk;
    const unsigned long long k_rows = (unsigned long long)units * kv.L_cap;
    const unsigned long long q_rows = (unsigned long long)kv.n_layers * kv.B * kv.H_q * w;
    CUtensorMap mq, mk;
    if (!encode_bf16_2d(&mq, q_win, q_rows, D, 64, 128) || !encode_bf16_2d(&mk, kv.k, k_rows, D, 64, N)) {
        *ok = false;
        return cudaSuccess;
    }
    cudaError_t e = cudaFuncSetAttribute(score_rowstats_tc<D, MT, N, EG>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)C::SMEM);
    if (e != cudaSuccess) return e;
    const int n_items = (int)(units * nch);
    const int grid = min(n_items, device_sm_count());
    e = launch_pdl(score_rowstats_tc<D, MT, N, EG>, dim3(grid), dim3(C::THREADS), C::SMEM, s, mq, mk, lens, w,
                   kv.H_q / kv.H_kv, kv.H_q, kv.H_kv, kv.L_cap, R, nch, n_items, masked ? ws.ulist : nullptr,
                   masked ? ws.ucount : nullptr, c2, ws.part_m, ws.part_z, err);
    *ok = true;
    return e != cudaSuccess ? e : cudaGetLastError();
}

// Key tiles of 256 for two query tiles: half the MMA instructions per key of 128-key tiles
// (the single issuing thread is the pass's bottleneck; 7B-class heads, both passes 2.03 ->
// 1.85 ms), with two 256-column TMEM regions and two K stages in shared memory.  Three or
// four query tiles leave shared memory for one such stage only and keep 128-key tiles.
template <int D>
static cudaError_t pass1_by_mt(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                               float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool *ok)
{
    const int MT = ((kv.H_q / kv.H_kv) * w + 127) / 128;
    switch (MT) {
    case 1: return run_pass1<D, 1, 128, 2>(kv, q_win, lens, masked, w, c2, ws, err, s, ok);
    case 2: return run_pass1<D, 2, 256, 2>(kv, q_win, lens, masked, w, c2, ws, err, s, ok);  // 256-key tiles
    case 3: return run_pass1<D, 3, 128, 2>(kv, q_win, lens, masked, w, c2, ws, err, s, ok);
    default: return run_pass1<D, 4, 128, 1>(kv, q_win, lens, masked, w, c2, ws, err, s, ok);
    }
}

cudaError_t launch_score_tc_pass1(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                                  float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool *used)
{
    *used = false;
    if (!score_tc_supported(kv, w)) return cudaSuccess;
    return kv.d == 128 ? pass1_by_mt<128>(kv, q_win, lens, masked, w, c2, ws, err, s, used)
                       : pass1_by_mt<64>(kv, q_win, lens, masked, w, c2, ws, err, s, used);
}

template <int D>
static cudaError_t run_pass2(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                             float c2, const ScoreWs &ws, const float *row_lse, unsigned *err, cudaStream_t s,
                             bool *ok)
{
    const long units = (long)kv.n_layers * kv.B * kv.H_kv;
    const int R = (kv.H_q / kv.H_kv) * w;
    const P2Shape ps = p2_shape(R);
    const int nch = (kv.L_cap + kScoreChunk - 1) / kScoreChunk;
    const unsigned long long k_rows = (unsigned long long)units * kv.L_cap;
    const unsigned long long q_rows = (unsigned long long)kv.n_layers * kv.B * kv.H_q * w;
    CUtensorMap mq, mk;
    const int qbox = ps.NQ > 256 ? ps.NQ / 2 : ps.NQ;
    if (!encode_bf16_2d(&mq, q_win, q_rows, D, 64, qbox) || !encode_bf16_2d(&mk, kv.k, k_rows, D, 64, 128)) {
        *ok = false;
        return cudaSuccess;
    }
    const size_t qbytes = (size_t)(D / 64) * ps.NQ * 128, kstage = (size_t)(D / 64) * 128 * 128;
    const size_t static_smem = sizeof(float) * (4 * kP2Groups * 128 + kP2Slots * kP2Groups * 128) + 1024;
    const size_t budget = 227 * 1024 - static_smem - 1024;
    const int NS = (int)min((size_t)4, (budget - qbytes) / kstage);
    if (qbytes >= budget || NS < 2) {
        *ok = false;
        return cudaSuccess;
    }
    const size_t smem = 1024 + qbytes + (size_t)NS * kstage;
    cudaError_t e = cudaFuncSetAttribute(score_colsum_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int n_items = (int)(units * nch);
    const int grid = min(n_items, device_sm_count());
    e = launch_pdl(score_colsum_tc<D>, dim3(grid), dim3(128 + 128 * kP2Groups), smem, s, mq, mk, lens, w,
                   kv.H_q / kv.H_kv, kv.H_q, kv.H_kv, kv.L_cap, R, ps.NQ, ps.NP, ps.NR, NS, nch, n_items,
                   masked ? ws.ulist : nullptr, masked ? ws.ucount : nullptr, c2, (const float *)ws.rowb, row_lse,
                   (long)kv.n_layers * kv.B * kv.H_q, ws.raw, err);
    *ok = true;
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_score_tc_pass2(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                                  float c2, const ScoreWs &ws, const float *row_lse, unsigned *err, cudaStream_t s,
                                  bool *used)
{
    *used = false;
    if (!score_tc_supported(kv, w)) return cudaSuccess;
    return kv.d == 128 ? run_pass2<128>(kv, q_win, lens, masked, w, c2, ws, row_lse, err, s, used)
                       : run_pass2<64>(kv, q_win, lens, masked, w, c2, ws, row_lse, err, s, used);
}

}  // namespace reco
