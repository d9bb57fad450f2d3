// score_tc.cu -- tensor-core (tcgen05) passes of the Eq. 2 cache scores for bf16 caches.
//
// Both passes are persistent (one CTA per SM walking a contiguous range of (unit,
// 2048-key chunk) items, barrier phases running on across items) with the same roles:
//   warp 0  lane 0 : TMA producer (window queries once, then a ring of K tiles)
//   warp 1         : allocates 512 TMEM columns; lane 0 issues tcgen05.mma (bf16 in,
//                    fp32 accumulate in TMEM) and commits to mbarriers
//   warps 4.. 	    : epilogue, reading accumulators with tcgen05.ld (one TMEM lane
//                    per thread) into the softmax arithmetic
// Operands sit in shared memory in the 128-byte-swizzled K-major layout the TMA writes
// (rows of 64 bf16, 8-row atoms of 1024 bytes); each MMA takes a K=16 slice.
//
// Pass 1 (row statistics): queries on M (128-row tiles), keys on N, so each thread
//   owns one window row and keeps its running max / sum over the chunk's keys.
// Pass 2 (column sums): keys on M (128 per tile), queries on N, so each thread owns
//   one key and sums 2^(c*l - b_r) over the window rows with b_r from pass 1.
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
// 1024 bytes (stride byte offset 1024), descriptor version 1.
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
constexpr int kTcMaxR = 384;  // window rows (G*w) the tensor-core passes take; pass 2 smem stays < 227 KB
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

// ---------------------------------------------------------------- pass 1: row statistics
template <int D, int N, int MT>
__global__ void __launch_bounds__(128 + 128 * MT, 1)
    score_rowstats_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                      const int32_t *__restrict__ lens, int w, int G, int Hq, int Hkv, int L_cap, int R,
                      int n_chunks, int n_items, const int32_t *__restrict__ ulist, const int32_t *__restrict__ ucount,
                      float c2, float *__restrict__ part_m, float *__restrict__ part_z,
                      unsigned *err)
{
    constexpr int HALVES = D / 64;
    constexpr int QBOX = 128 * 128;  // 128 rows x 128 bytes
    constexpr int KBOX = N * 128;
    constexpr int KSTAGE = HALVES * KBOX;
    constexpr int NS = 4;
    constexpr uint32_t IDESC = idesc_bf16(128, N);
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bar_qfull, bar_qempty, bar_kfull[NS], bar_kempty[NS], bar_afull[2],
        bar_aempty[2];
    __shared__ uint32_t tmem_sh;
    __shared__ int abort_sh;

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n_it = ucount ? *ucount * n_chunks : n_items;  // items of the scored units
    const int i_begin = (int)((long long)blockIdx.x * n_it / gridDim.x);
    const int i_end = (int)((long long)(blockIdx.x + 1) * n_it / gridDim.x);
    const uint32_t raw0 = smem_addr(smem_raw);
    const uint32_t base = (raw0 + 1023u) & ~1023u;
    const uint32_t Qs = base;                                  // MT x HALVES x QBOX
    const uint32_t Ks = base + (uint32_t)MT * HALVES * QBOX;  // NS x KSTAGE
    if (tid == 0) {
        mbar_init(smem_addr(&bar_qfull), 1);
        mbar_init(smem_addr(&bar_qempty), 1);
        for (int s = 0; s < NS; ++s) {
            mbar_init(smem_addr(&bar_kfull[s]), 1);
            mbar_init(smem_addr(&bar_kempty[s]), 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&bar_afull[b]), 1);
            mbar_init(smem_addr(&bar_aempty[b]), 4 * MT);
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
                    mbar_expect_tx(smem_addr(&bar_qfull), (uint32_t)MT * HALVES * QBOX);
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
                        tma_load_2d(Ks + s * KSTAGE + hh * KBOX, &tmK, 64 * hh, k_row0 + t * N, smem_addr(&bar_kfull[s]));
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
                for (int t = 0; t < it.ntiles; ++t, ++gt) {
                    const int s = gt % NS, b = gt & 1;
                    if (!wait_or_flag(smem_addr(&bar_kfull[s]), (gt / NS) & 1, abort_flag, err) ||
                        !wait_or_flag(smem_addr(&bar_aempty[b]), ((gt >> 1) & 1) ^ 1, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    for (int mt = 0; mt < MT; ++mt) {
                        const uint32_t d = tmem + (uint32_t)((b * MT + mt) * N);
#pragma unroll
                        for (int k = 0; k < D / 16; ++k) {
                            const int hh = k >> 2, kk = k & 3;
                            const uint64_t ad = sw128_desc(Qs + (mt * HALVES + hh) * QBOX + kk * 32);
                            const uint64_t bd = sw128_desc(Ks + s * KSTAGE + hh * KBOX + kk * 32);
                            tc_mma(d, ad, bd, IDESC, k > 0 ? 1u : 0u);
                        }
                    }
                    tc_commit(smem_addr(&bar_kempty[s]));
                    tc_commit(smem_addr(&bar_afull[b]));
                }
            }
        }
    } else if (warp >= 4 && warp < 4 + 4 * MT) {  // epilogue: one window row per thread
        const int e = warp - 4, mt = e >> 2, quarter = warp & 3;
        const int r = mt * 128 + quarter * 32 + lane;
        const int t_row = r % w;
        int gt = 0;
        for (int i = i_begin; i < i_end; ++i) {
            const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, false, N);
            if (!it.valid) {
                if (it.chunk == 0 && r == 0) raise_error(err, ERR_LEN);
                continue;
            }
            const int jmax = it.L - w + t_row;  // last key this window row sees
            float m = -INFINITY, z = 0.f;
            bool ok = true;
            for (int t = 0; t < it.ntiles; ++t, ++gt) {
                const int b = gt & 1;
                if (!wait_or_flag(smem_addr(&bar_afull[b]), (gt >> 1) & 1, abort_flag, err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t ta = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)((b * MT + mt) * N);
                const int jb = it.j0 + t * N;
                const int lim = min(it.j1 - 1, jmax) - jb;  // columns 0..lim are visible to this row
                float v[N];  // the whole tile row: all TMEM loads issued before one wait
#pragma unroll
                for (int cc = 0; cc < N; cc += 32) tmem_ld32_nowait(ta + cc, *reinterpret_cast<float(*)[32]>(v + cc));
                tmem_ld_wait();
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&bar_aempty[b]));
                // logits are v * c2 with c2 > 0: take the max on v, exponentiate fma(v, c2, -m)
                float mx4[4] = {-INFINITY, -INFINITY, -INFINITY, -INFINITY};
                const bool full_tile = lim >= N - 1;  // no masking needed (most tiles)
                if (full_tile) {
#pragma unroll
                    for (int q = 0; q < N; ++q) mx4[q & 3] = fmaxf(mx4[q & 3], v[q]);
                } else {
#pragma unroll
                    for (int q = 0; q < N; ++q)
                        if (q <= lim) mx4[q & 3] = fmaxf(mx4[q & 3], v[q]);
                }
                const float mx = fmaxf(fmaxf(mx4[0], mx4[1]), fmaxf(mx4[2], mx4[3]));
                const float mn = fmaxf(m, mx * c2);
                if (mn == -INFINITY) continue;
                const float nb = -mn;
                float a4[4] = {0.f, 0.f, 0.f, 0.f};
                if (full_tile) {
#pragma unroll
                    for (int q = 0; q < N; ++q) a4[q & 3] += fast_exp2(fmaf(v[q], c2, nb));
                } else {
#pragma unroll
                    for (int q = 0; q < N; ++q) a4[q & 3] += (q <= lim) ? fast_exp2(fmaf(v[q], c2, nb)) : 0.f;
                }
                z = z * fast_exp2(m - mn) + ((a4[0] + a4[1]) + (a4[2] + a4[3]));
                m = mn;
            }
            if (!ok) break;
            if (r < R) {
                part_m[((size_t)it.u * n_chunks + it.chunk) * R + r] = m;
                part_z[((size_t)it.u * n_chunks + it.chunk) * R + r] = z;
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
// NQ (runtime, multiple of 16, <= 384) query columns per tile.  With NQ <= 256 the two
// epilogue warpgroups take alternate tiles (two TMEM buffers); above 256 one buffer is
// shared and each warpgroup sums half of the columns.
template <int D>
__global__ void __launch_bounds__(128 + 256, 1)
    score_colsum_tc(const __grid_constant__ CUtensorMap tmQ, const __grid_constant__ CUtensorMap tmK,
                    const int32_t *__restrict__ lens, int w, int G, int Hq, int Hkv, int L_cap, int R, int NQ,
                    int n_chunks, int n_items, const int32_t *__restrict__ ulist, const int32_t *__restrict__ ucount,
                    float c2, const float *__restrict__ rowb, float *__restrict__ raw,
                    unsigned *err)
{
    constexpr int HALVES = D / 64;
    constexpr int KBOX = 128 * 128;  // 128 keys x 128 bytes
    constexpr int KSTAGE = HALVES * KBOX;
    constexpr int NS = 3;
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bar_qfull, bar_qempty, bar_kfull[NS], bar_kempty[NS], bar_afull[2],
        bar_aempty[2];
    __shared__ uint32_t tmem_sh;
    __shared__ int abort_sh;
    __shared__ float bsh[8][kTcMaxR];  // per epilogue warp: row normalisers of its current unit

    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int n_it = ucount ? *ucount * n_chunks : n_items;  // items of the scored units
    const int i_begin = (int)((long long)blockIdx.x * n_it / gridDim.x);
    const int i_end = (int)((long long)(blockIdx.x + 1) * n_it / gridDim.x);
    const bool split_cols = NQ > 256;
    const int NBUF = split_cols ? 1 : 2;
    const int nmma = split_cols ? 2 : 1;
    const int NM = NQ / nmma;  // MMA N
    const uint32_t idesc = idesc_bf16(128, NM);
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
        for (int b = 0; b < 2; ++b) {
            mbar_init(smem_addr(&bar_afull[b]), 1);
            mbar_init(smem_addr(&bar_aempty[b]), split_cols ? 8 : 4);
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

    if (warp == 0) {
        if (lane == 0) {  // producer
            const int qbox_rows = NQ > 256 ? NQ / 2 : NQ;
            int gt = 0, nq = 0;
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
                for (int t = 0; t < it.ntiles; ++t, ++gt) {
                    const int s = gt % NS;
                    if (!wait_or_flag(smem_addr(&bar_kempty[s]), ((gt / NS) & 1) ^ 1, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    mbar_expect_tx(smem_addr(&bar_kfull[s]), KSTAGE);
                    for (int hh = 0; hh < HALVES; ++hh)
                        tma_load_2d(Ks + s * KSTAGE + hh * KBOX, &tmK, 64 * hh, k_row0 + t * 128,
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
                const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, true, 128);
                if (it.ntiles == 0) continue;
                if (it.u != prev_u) {
                    if (nq > 0) tc_commit(smem_addr(&bar_qempty));
                    if (!wait_or_flag(smem_addr(&bar_qfull), nq & 1, abort_flag, err)) break;
                    ++nq;
                    prev_u = it.u;
                }
                for (int t = 0; t < it.ntiles; ++t, ++gt) {
                    const int s = gt % NS, b = NBUF == 2 ? (gt & 1) : 0;
                    const uint32_t bph = NBUF == 2 ? ((gt >> 1) & 1) : (gt & 1);
                    if (!wait_or_flag(smem_addr(&bar_kfull[s]), (gt / NS) & 1, abort_flag, err) ||
                        !wait_or_flag(smem_addr(&bar_aempty[b]), bph ^ 1, abort_flag, err)) {
                        ok = false;
                        break;
                    }
                    tc_fence_after();
                    for (int nb = 0; nb < nmma; ++nb) {
                        const uint32_t d = tmem + (uint32_t)(b * 256 + nb * NM);
                        for (int k = 0; k < D / 16; ++k) {
                            const int hh = k >> 2, kk = k & 3;
                            const uint64_t ad = sw128_desc(Ks + s * KSTAGE + hh * KBOX + kk * 32);
                            const uint64_t bd = sw128_desc(Qs + hh * QBOXB + nb * NM * 128 + kk * 32);
                            tc_mma(d, ad, bd, idesc, k > 0 ? 1u : 0u);
                        }
                    }
                    tc_commit(smem_addr(&bar_kempty[s]));
                    tc_commit(smem_addr(&bar_afull[b]));
                }
            }
        }
    } else if (warp >= 4) {  // epilogue: one key per thread
        const int eg = (warp - 4) >> 2, quarter = warp & 3;
        const int row = quarter * 32 + lane;  // key within the tile
        const int c_lo = split_cols ? eg * (NQ / 2) : 0;
        const int c_hi = split_cols ? c_lo + NQ / 2 : NQ;
        const float invG = 1.f / (float)G;
        float *bs = bsh[warp - 4];
        int gt = 0;
        long prev_u = -1;
        for (int i = i_begin; i < i_end; ++i) {
            const ChunkItem it = chunk_item(i, n_chunks, ulist, lens, w, L_cap, true, 128);
            if (it.ntiles == 0) continue;
            if (it.u != prev_u) {  // this unit's row normalisers (warp-private copy)
                __syncwarp();
                for (int rr = lane; rr < kTcMaxR; rr += 32) bs[rr] = rr < R ? rowb[it.u * R + rr] : 0.f;
                __syncwarp();
                prev_u = it.u;
            }
            bool ok = true;
            for (int t = 0; t < it.ntiles; ++t, ++gt) {
                const bool mine = split_cols || ((gt & 1) == eg);
                if (!mine) continue;
                const int b = NBUF == 2 ? (gt & 1) : 0;
                const uint32_t bph = NBUF == 2 ? ((gt >> 1) & 1) : (gt & 1);
                if (!wait_or_flag(smem_addr(&bar_afull[b]), bph, abort_flag, err)) {
                    ok = false;
                    break;
                }
                tc_fence_after();
                const uint32_t ta = tmem + ((uint32_t)(quarter * 32) << 16) + (uint32_t)(b * 256);
                float a4[4] = {0.f, 0.f, 0.f, 0.f};
                for (int cb = c_lo; cb < c_hi; cb += 64) {
                    float v[64];
                    const bool two = cb + 32 < c_hi;
                    tmem_ld32_nowait(ta + cb, *reinterpret_cast<float(*)[32]>(v));
                    if (two) tmem_ld32_nowait(ta + cb + 32, *reinterpret_cast<float(*)[32]>(v + 32));
                    tmem_ld_wait();
                    const int nv = two ? 64 : 32;
                    if (cb + nv <= R) {  // every column is a real window row
#pragma unroll
                        for (int q = 0; q < 64; ++q)
                            if (q < nv) a4[q & 3] += fast_exp2(fmaf(v[q], c2, -bs[cb + q]));
                    } else {
#pragma unroll
                        for (int q = 0; q < 64; ++q)
                            if (q < nv && cb + q < R) a4[q & 3] += fast_exp2(fmaf(v[q], c2, -bs[cb + q]));
                    }
                }
                const float acc = (a4[0] + a4[1]) + (a4[2] + a4[3]);
                tc_fence_before();
                __syncwarp();
                if (lane == 0) mbar_arrive(smem_addr(&bar_aempty[b]));
                const int j = it.j0 + t * 128 + row;
                if (j < it.j1) {
                    if (split_cols)  // two halves land on a zeroed entry: 0 + a + b, order-independent
                        atomicAdd(raw + it.u * L_cap + j, acc * invG);
                    else
                        raw[it.u * L_cap + j] = acc * invG;
                }
            }
            if (!ok) break;
        }
    }
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------- host side

int score_tc_nq(int R) { return R <= 256 ? ((R + 15) / 16) * 16 : ((R + 31) / 32) * 32; }

bool score_tc_supported(const reco_kv &kv, int w)
{
    const long long R = (long long)(kv.H_q / kv.H_kv) * w;
    const unsigned long long k_rows = (unsigned long long)kv.n_layers * kv.B * kv.H_kv * kv.L_cap;
    const unsigned long long q_rows = (unsigned long long)kv.n_layers * kv.B * kv.H_q * w;
    return kv.dtype == RECO_BF16 && (kv.d == 64 || kv.d == 128) && R <= kTcMaxR && k_rows < (1ull << 31) &&
           q_rows < (1ull << 31);
}

template <int D, int N, int MT>
static cudaError_t run_pass1(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                             float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool *ok)
{
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
    const size_t smem = 1024 + (size_t)MT * (D / 64) * 128 * 128 + 4 * (size_t)(D / 64) * N * 128;
    cudaError_t e = cudaFuncSetAttribute(score_rowstats_tc<D, N, MT>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    const int n_items = (int)(units * nch);
    const int grid = min(n_items, device_sm_count());
    score_rowstats_tc<D, N, MT><<<grid, 128 + 128 * MT, smem, s>>>(mq, mk, lens, w, kv.H_q / kv.H_kv, kv.H_q,
                                                                  kv.H_kv, kv.L_cap, R, nch, n_items,
                                                                  masked ? ws.ulist : nullptr,
                                                                  masked ? ws.ucount : nullptr, c2, ws.part_m,
                                                                  ws.part_z, err);
    *ok = true;
    return cudaGetLastError();
}

template <int D>
static cudaError_t pass1_by_mt(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                               float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool *ok)
{
    const int MT = ((kv.H_q / kv.H_kv) * w + 127) / 128;
    switch (MT) {
    case 1: return run_pass1<D, 128, 1>(kv, q_win, lens, masked, w, c2, ws, err, s, ok);
    case 2: return run_pass1<D, 128, 2>(kv, q_win, lens, masked, w, c2, ws, err, s, ok);
    case 3: return run_pass1<D, 64, 3>(kv, q_win, lens, masked, w, c2, ws, err, s, ok);
    default: return run_pass1<D, 64, 4>(kv, q_win, lens, masked, w, c2, ws, err, s, ok);
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
                             float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool *ok)
{
    const long units = (long)kv.n_layers * kv.B * kv.H_kv;
    const int R = (kv.H_q / kv.H_kv) * w;
    const int NQ = score_tc_nq(R);
    const int nch = (kv.L_cap + kScoreChunk - 1) / kScoreChunk;
    const unsigned long long k_rows = (unsigned long long)units * kv.L_cap;
    const unsigned long long q_rows = (unsigned long long)kv.n_layers * kv.B * kv.H_q * w;
    CUtensorMap mq, mk;
    const int qbox = NQ > 256 ? NQ / 2 : NQ;
    if (!encode_bf16_2d(&mq, q_win, q_rows, D, 64, qbox) || !encode_bf16_2d(&mk, kv.k, k_rows, D, 64, 128)) {
        *ok = false;
        return cudaSuccess;
    }
    cudaError_t e;
    if (NQ > 256 && (e = cudaMemsetAsync(ws.raw, 0, (size_t)units * kv.L_cap * sizeof(float), s)) != cudaSuccess)
        return e;
    const size_t smem = 1024 + (size_t)(D / 64) * NQ * 128 + 3 * (size_t)(D / 64) * 128 * 128;
    e = cudaFuncSetAttribute(score_colsum_tc<D>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    const int n_items = (int)(units * nch);
    const int grid = min(n_items, device_sm_count());
    score_colsum_tc<D><<<grid, 128 + 256, smem, s>>>(mq, mk, lens, w, kv.H_q / kv.H_kv, kv.H_q, kv.H_kv, kv.L_cap, R,
                                                     NQ, nch, n_items, masked ? ws.ulist : nullptr,
                                                     masked ? ws.ucount : nullptr, c2, ws.rowb, ws.raw, err);
    *ok = true;
    return cudaGetLastError();
}

cudaError_t launch_score_tc_pass2(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                                  float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool *used)
{
    *used = false;
    if (!score_tc_supported(kv, w)) return cudaSuccess;
    return kv.d == 128 ? run_pass2<128>(kv, q_win, lens, masked, w, c2, ws, err, s, used)
                       : run_pass2<64>(kv, q_win, lens, masked, w, c2, ws, err, s, used);
}

}  // namespace reco
