// decode.cu -- decode attention over the ragged compacted cache, the per-token
// attention whose cost the compression lowers (Sec. 1; Sec. 2.2; Sec. 4.2).
//
// bf16 path (decode_tma): a persistent split-K flash-decode, one CTA of 8 warps per
// SM (for long work 4 of them, each with a ring twice as deep).  Every CTA first
// builds the same work plan from lens: the prefix sum of 16-key blocks per unit, with
// the blocks of all units laid end to end and cut into one equal contiguous range per
// warp (a stream-K split: balanced to one block, no work queue).  A call with more units
// than one plan holds runs as consecutive launches over contiguous unit ranges.
// When no unit is long enough to be cut, the units are instead sorted by length and
// dealt whole to the warps in snake order (longest first).
// An item's keys stream from HBM in 16-key blocks: one lane issues TMA tensor copies
// (128-byte swizzled 16 x 64 tiles of K and V) into the warp's 3-stage ring and the
// warp waits on the stage's mbarrier (bounded).  QK^T and PV run on mma.sync
// m16n8k16 (bf16 in, fp32 accumulate) with the G <= 8 query heads of the KV head
// packed into one MMA tile.  The head dimension is permuted consistently on the Q
// and K sides (and on the V and output sides) so that each thread's fragments are
// whole 16-byte chunks, and the swizzle makes every fragment read conflict-free.  A
// unit split over several items writes partial (max, sum, output) triples; the last
// item to finish (atomic ticket, no waiting) merges them.  The counters live in the
// caller's workspace, zero-filled before its first use; each launch clears what it
// counted, so no reset runs between launches.  The appended token (k_new, v_new) is
// read from the inputs and written into the cache by the warp that covers its index;
// the last warp of the grid to finish advances lens.
//
// float32 path (decode_simt): one CTA per unit, four warps over the keys, G <= 16.
#include <cuda.h>

#include <algorithm>

#include "common.cuh"
#include "internal.h"
#include "tma.cuh"

namespace reco {

DecodeWs decode_ws_layout(const reco_kv &kv, void *base)
{
    size_t units = (size_t)kv.n_layers * kv.B * kv.H_kv;
    size_t G = kv.H_q / kv.H_kv;
    char *p = (char *)base;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *r = p ? p + off : nullptr;
        off += align256(bytes);
        return r;
    };
    DecodeWs ws;
    ws.part_slots = kDecodePartSlots;
    // merge tickets per unit of the TMA path, which splits a unit of G > 8 heads in two
    ws.counters = (int32_t *)take((2 + units * (G > 8 ? 2 : 1)) * 4);
    ws.part_ml = (float *)take((size_t)ws.part_slots * G * 2 * 4);
    ws.part_o = (float *)take((size_t)ws.part_slots * G * kv.d * 4);
    ws.bytes = off;
    return ws;
}

struct DecodeArgs {
    void *K;
    void *V;
    const void *q;
    const void *k_new;
    const void *v_new;
    int32_t *lens;
    void *out;
    float *lse;
    int32_t *counters;
    float *part_ml;
    float *part_o;
    int units, Hq, Hkv, G, L_cap, append, out_bf16;
    float c2;  // scale * log2(e)
    unsigned *err;
    int hs, gv;       // TMA path: hs virtual units of gv (<= 8) query heads per unit (G > 8: hs = 2)
    float *ring;      // or nullptr: lse rows ring[*slot] and ring[*slot + slots], each [nq]
    long long *slot;  // device ring row, advanced by one (mod slots) per launch
    int slots;
    long long nq;     // query heads of the launch (layers * B * H_q)
    void *qring;      // or nullptr: [nq][slots][D] of q's dtype, row *slot of every head gets its query
    int q_bytes;      // bytes per element of q
    long long nq_rows;  // query heads of this launch (nq, or a part of it when the units are split)
    int advance;        // this launch advances *slot (the last of a split launch's parts)
};

// The ring row this launch writes (read once the previous kernel's writes are visible),
// or -1 without a ring; a slot outside [0, slots) writes nothing and sets the error word.
__device__ __forceinline__ long long ring_row(const DecodeArgs &a)
{
    if (!a.ring) return -1;
    const long long s = *a.slot;
    if (s < 0 || s >= a.slots) {
        raise_error(a.err, ERR_INTERNAL);
        return -1;
    }
    return s;
}

// lse of query row i: to the lse output and, with a ring, to ring rows rs and rs + slots.
__device__ __forceinline__ void put_lse(const DecodeArgs &a, long long rs, size_t i, float v)
{
    if (a.lse) a.lse[i] = v;
    if (rs >= 0) {
        a.ring[rs * a.nq + (long long)i] = v;
        a.ring[(rs + a.slots) * a.nq + (long long)i] = v;
    }
}

// atomicAdd with acquire-release semantics at GPU scope.
__device__ __forceinline__ int atom_add_acq_rel(int *p, int v)
{
    int old;
    asm volatile("atom.acq_rel.gpu.global.add.s32 %0, [%1], %2;" : "=r"(old) : "l"(p), "r"(v) : "memory");
    return old;
}

__device__ __forceinline__ unsigned long long atom_add_acq_rel_u64(unsigned long long *p, unsigned long long v)
{
    unsigned long long old;
    asm volatile("atom.acq_rel.gpu.global.add.u64 %0, [%1], %2;" : "=l"(old) : "l"(p), "l"(v) : "memory");
    return old;
}

__device__ __forceinline__ bool unit_ok(int L, int L_cap, int append)
{
    return L >= 0 && L <= L_cap && (!append || L < L_cap);
}

template <typename T> __device__ __forceinline__ void store_out(void *out, bool bf16, size_t i, float v)
{
    if (bf16)
        reinterpret_cast<__nv_bfloat16 *>(out)[i] = __float2bfloat16_rn(v);
    else
        reinterpret_cast<float *>(out)[i] = v;
}

// ---------------------------------------------------------------- SIMT path
template <typename T, int D>
__global__ void __launch_bounds__(128) decode_simt(DecodeArgs a)
{
    constexpr int NW = 4, PER = D / 32, GM = 16;
    __shared__ float sm_m[NW][GM], sm_l[NW][GM];
    __shared__ float sm_o[NW][GM][D];
    const long u = blockIdx.x;
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const int L = a.lens[u];
    const long long rs = ring_row(a);
    const bool ok = unit_ok(L, a.L_cap, a.append);
    if (!ok && threadIdx.x == 0) raise_error(a.err, (a.append && L == a.L_cap) ? ERR_ROOM : ERR_LEN);
    const int Le = ok ? L + a.append : 0;
    const long lb = u / a.Hkv;
    const int h = (int)(u % a.Hkv);
    const int G = a.G;
    T *Kp = reinterpret_cast<T *>(a.K) + u * (long)a.L_cap * D;
    T *Vp = reinterpret_cast<T *>(a.V) + u * (long)a.L_cap * D;
    const T *kn = a.append ? reinterpret_cast<const T *>(a.k_new) + u * D : nullptr;
    const T *vn = a.append ? reinterpret_cast<const T *>(a.v_new) + u * D : nullptr;
    const T *qp = reinterpret_cast<const T *>(a.q) + (lb * a.Hq + (long)h * G) * D;
    float q[GM][PER], o[GM][PER], m[GM], l[GM];
#pragma unroll
    for (int g = 0; g < GM; ++g) {
        m[g] = -INFINITY;
        l[g] = 0.f;
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            q[g][i] = g < G ? to_float(qp[(long)g * D + lane * PER + i]) : 0.f;
            o[g][i] = 0.f;
        }
    }
    for (int j = wid; j < Le; j += NW) {
        const T *kr = (a.append && j == L) ? kn : Kp + (long)j * D;
        const T *vr = (a.append && j == L) ? vn : Vp + (long)j * D;
        float kk[PER], vv[PER];
#pragma unroll
        for (int i = 0; i < PER; ++i) {
            kk[i] = to_float(kr[lane * PER + i]);
            vv[i] = to_float(vr[lane * PER + i]);
        }
#pragma unroll
        for (int g = 0; g < GM; ++g) {
            if (g < G) {
                float s = 0.f;
#pragma unroll
                for (int i = 0; i < PER; ++i) s = fmaf(q[g][i], kk[i], s);
                s = warp_sum(s) * a.c2;
                const float mn = fmaxf(m[g], s);
                const float al = fast_exp2(m[g] - mn);
                const float p = fast_exp2(s - mn);
                l[g] = l[g] * al + p;
#pragma unroll
                for (int i = 0; i < PER; ++i) o[g][i] = fmaf(o[g][i], al, p * vv[i]);
                m[g] = mn;
            }
        }
    }
#pragma unroll
    for (int g = 0; g < GM; ++g) {
        if (g < G) {
            if (lane == 0) {
                sm_m[wid][g] = m[g];
                sm_l[wid][g] = l[g];
            }
#pragma unroll
            for (int i = 0; i < PER; ++i) sm_o[wid][g][lane * PER + i] = o[g][i];
        }
    }
    __syncthreads();
    for (int e = threadIdx.x; e < G * D; e += blockDim.x) {
        const int g = e / D, dd = e % D;
        float M = -INFINITY;
        for (int w = 0; w < NW; ++w) M = fmaxf(M, sm_m[w][g]);
        float Ls = 0.f, O = 0.f;
        if (M != -INFINITY) {
            for (int w = 0; w < NW; ++w) {
                const float wt = fast_exp2(sm_m[w][g] - M);
                Ls += sm_l[w][g] * wt;
                O += sm_o[w][g][dd] * wt;
            }
        }
        const size_t row = (size_t)(lb * a.Hq + (long)h * G + g);
        store_out<T>(a.out, a.out_bf16, row * D + dd, Ls > 0.f ? O / Ls : 0.f);
        if (dd == 0) put_lse(a, rs, row, Ls > 0.f ? (M + log2f(Ls)) * kLn2 : -INFINITY);
    }
    if (ok && a.append) {
        for (int e = threadIdx.x; e < D; e += blockDim.x) {
            Kp[(long)L * D + e] = kn[e];
            Vp[(long)L * D + e] = vn[e];
        }
        if (threadIdx.x == 0) a.lens[u] = L + 1;
    }
}

// ---------------------------------------------------------------- tensor-core path
__device__ __forceinline__ void mma_bf16(float (&c)[4], uint32_t a0, uint32_t a1, uint32_t a2, uint32_t a3,
                                         uint32_t b0, uint32_t b1)
{
    asm volatile(
        "mma.sync.aligned.m16n8k16.row.col.f32.bf16.bf16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
        "{%0,%1,%2,%3};"
        : "+f"(c[0]), "+f"(c[1]), "+f"(c[2]), "+f"(c[3])
        : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

__device__ __forceinline__ uint32_t pack_bf16(float lo, float hi)
{
    __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
    return *reinterpret_cast<uint32_t *>(&v);
}

// (a, b) -> bf16x2 hi = round(a, b) and lo = round((a, b) - hi).
__device__ __forceinline__ void split_bf16(float a, float b, uint32_t &hi, uint32_t &lo)
{
    __nv_bfloat162 h = __floats2bfloat162_rn(a, b);
    const float2 f = __bfloat1622float2(h);
    hi = *reinterpret_cast<uint32_t *>(&h);
    lo = pack_bf16(a - f.x, b - f.y);
}

__device__ __forceinline__ uint32_t word(const uint4 &v, int x)
{
    return x == 0 ? v.x : (x == 1 ? v.y : (x == 2 ? v.z : v.w));
}

constexpr int kDecodeWarps = 8;       // warps per CTA (one CTA per SM)
constexpr int kDecodeStages = 3;      // ring stages per warp
constexpr int kMaxTmaUnits = 8192;    // one plan entry per unit kept in shared memory
constexpr long long kSpinLimit = 1LL << 24;  // bounded mbarrier waits (about a second)
constexpr float kLazyLog2 = 8.f;             // output rescale threshold (log2 units)
constexpr int kMinBlocksPerWarp = 4;         // fewer working warps rather than shorter ranges
constexpr int kMaxWholeBlocks = 16;          // units of at most this many blocks are never cut
constexpr int kDeepBlocksPerWarp = 64;       // from this many blocks per warp, half the warps with deep rings

template <int D> struct TmaLayout {
    static constexpr int HALVES = D / 64;             // 128-byte boxes per row
    static constexpr int TILE = 16 * 128;             // one 16-row box
    static constexpr int STAGE = 4 * HALVES * 16 * 64; // K boxes then V boxes (bytes)
    static constexpr int RING = kDecodeWarps * kDecodeStages * STAGE;
};

// the largest plan fits beside the d = 128 ring (227 KB per CTA, about 1 KB of it static)
static_assert(1024 + TmaLayout<128>::RING + (kMaxTmaUnits + 1) * 4 + 1024 <= 227 * 1024, "decode smem budget");
static_assert((kMaxTmaUnits + 32 + (kMaxWholeBlocks + 1) * kDecodeWarps * 32) * 4 <= TmaLayout<64>::RING,
              "lengths and the sort counters are staged in the ring");

template <int D>
size_t tma_smem_bytes(int units)
{
    return 1024 + (size_t)TmaLayout<D>::RING + (size_t)(units + 1) * sizeof(int);
}

// Byte offset of 16-byte chunk ch (0..7) of row rr inside a 128B-swizzled 16-row box.
__device__ __forceinline__ uint32_t swz(int rr, int ch) { return rr * 128 + ((ch ^ (rr & 7)) << 4); }

template <int D, int HS>
__global__ void __launch_bounds__(kDecodeWarps * 32, 1)
    decode_tma(const __grid_constant__ CUtensorMap tmK, const __grid_constant__ CUtensorMap tmV, DecodeArgs a)
{
    using LY = TmaLayout<D>;
    constexpr int NW = kDecodeWarps, S = kDecodeStages, HALVES = LY::HALVES, TILE = LY::TILE;
    constexpr int STAGE = LY::STAGE;
    constexpr int MT = D / 16;  // m-tiles of PV (d on M)
    extern __shared__ __align__(1024) unsigned char smem_raw[];
    __shared__ __align__(8) uint64_t bars[NW * S];  // ring stages of all warps (either partition)
    __shared__ int sm_scan[NW];
    __shared__ int sm_red[2 * NW];  // per warp: most blocks of a unit, units with keys
    const uint32_t raw0 = (uint32_t)__cvta_generic_to_shared(smem_raw);
    const uint32_t ring0 = (raw0 + 1023u) & ~1023u;
    int *sm_pre = reinterpret_cast<int *>(smem_raw + (ring0 - raw0) + LY::RING);  // [units + 1]
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int units = a.units;
    if (tid == 0) {  // fetch both tensor-map descriptors (kernel parameters) while the previous kernel drains
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmK)) : "memory");
        asm volatile("prefetch.tensormap [%0];" ::"l"(reinterpret_cast<uint64_t>(&tmV)) : "memory");
    }
    if (lane == 0) {
        for (int s2 = 0; s2 < S; ++s2) mbar_init((uint32_t)__cvta_generic_to_shared(&bars[wid * S + s2]), 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        fence_async_shared();
    }
    __syncwarp();
    wait_prior_grid();  // lens, q and the new rows may come from the previous kernels
    const long long rs = ring_row(a);  // the ring row this launch writes (-1: none)

    // ---- plan: identical in every CTA (lens are not modified until every warp is done).
    // Each unit's keys form nb_u = ceil(le_u / 16) blocks; the blocks of all units are laid
    // end to end (prefix pb) and every working warp takes one contiguous range of equal
    // length, cut across unit boundaries (a stream-K split).  A unit cut between warps
    // leaves partial (max, sum, output) triples that its last piece merges.  Short units
    // (<= kMaxWholeBlocks blocks) are never cut: a range start inside one moves to the
    // unit's nearer end, since there a merge costs more than the imbalance it removes.
    int *pb = sm_pre;  // [units + 1] prefix of blocks
    const int seg = (units + blockDim.x - 1) / blockDim.x;
    const int u_lo = min(units, tid * seg), u_hi = min(units, u_lo + seg);
    // Units here are virtual: unit u covers query heads [(u / P) * gv, ...) of the cache
    // unit u % P (P cache units).  With two halves (G > 8) all first halves come first in
    // the plan, then all second halves in the same order, so warps w and w + W/2 stream
    // the same rows at about the same time and the second read mostly hits L2.
    const int GS = a.gv, P = units / HS;
    auto cache_unit = [&](int u) { return HS == 1 ? u : u % P; };
    auto head_part = [&](int u) { return HS == 1 ? 0 : u / P; };
    auto eff_len = [&](int u) {
        const int L = a.lens[cache_unit(u)];
        return unit_ok(L, a.L_cap, a.append) ? L + a.append : -1;
    };
    // stage the lengths in the (still idle) ring memory with one coalesced sweep; the
    // plan below reads them from there (the ring is first written by TMA after the plan)
    int *len_sm = reinterpret_cast<int *>(smem_raw + (ring0 - raw0));
    for (int u0 = 0; u0 < units; u0 += 8 * (int)blockDim.x) {
        int Lr[8];  // all loads of the batch in flight before any store or error report
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int u = u0 + k * (int)blockDim.x + tid;
            Lr[k] = u < units ? __ldcg(a.lens + cache_unit(u)) : 0;
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const int u = u0 + k * (int)blockDim.x + tid;
            if (u < units) {
                const bool ok = unit_ok(Lr[k], a.L_cap, a.append);
                if (!ok && blockIdx.x == 0)
                    raise_error(a.err, (a.append && Lr[k] == a.L_cap) ? ERR_ROOM : ERR_LEN);
                len_sm[u] = ok ? Lr[k] + a.append : 0;
            }
        }
    }
    __syncthreads();
    {
        int my_b = 0, my_max = 0, my_ne = 0;
        for (int u = u_lo; u < u_hi; ++u) {
            const int nb = (len_sm[u] + 15) >> 4;
            my_b += nb;
            my_max = max(my_max, nb);
            my_ne += nb > 0;
        }
        int f = my_b;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int nf = __shfl_up_sync(0xffffffffu, f, o);
            if (lane >= o) f += nf;
        }
        my_max = __reduce_max_sync(0xffffffffu, (unsigned)my_max);
        my_ne = __reduce_add_sync(0xffffffffu, (unsigned)my_ne);
        if (lane == 31) sm_scan[wid] = f;
        if (lane == 0) {
            sm_red[wid] = my_max;
            sm_red[NW + wid] = my_ne;
        }
        __syncthreads();
        int rb = f - my_b;
        for (int w2 = 0; w2 < wid; ++w2) rb += sm_scan[w2];
        for (int u = u_lo; u < u_hi; ++u) {
            pb[u] = rb;
            rb += (len_sm[u] + 15) >> 4;
        }
        if (tid == blockDim.x - 1) pb[units] = rb;
    }
    __syncthreads();
    const int NB = pb[units];
    const int total_warps = gridDim.x * NW;
    // Long work (at least kDeepBlocksPerWarp blocks per warp) runs on half the warps, each
    // with a ring twice as deep: more bytes in flight per warp keep HBM busier once every
    // warp has many blocks; short work keeps all warps for latency.  The CTA's ring is the
    // same either way (NW * S stages).
    // Fewer than half as many units as warps (with at least 8 blocks per warp) also
    // takes the deep partition: there the 8-warp split would cut every unit into many
    // pieces, whose merges cost more than the shallower rings save.
    const bool deep =
        NB >= kDeepBlocksPerWarp * total_warps || (NB >= 8 * total_warps && total_warps > 2 * units);
    int max_nb = 0, n_ne = 0;  // most blocks of one unit; units with keys
#pragma unroll
    for (int w2 = 0; w2 < NW; ++w2) {
        max_nb = max(max_nb, sm_red[w2]);
        n_ne += sm_red[NW + w2];
    }
    // Only short units (none is ever cut): the contiguous deal below would leave some warps
    // two whole units where others have one.  Instead the units are sorted by blocks, most
    // first (ties by index, so every CTA builds the same order), and dealt in snake order:
    // warp w takes sorted units w, 2W-1-w, 2W+w, ... of W = min(warps, units with keys),
    // so a warp holding one of the longest units in a round holds one of the shortest in
    // the next.  The order replaces the block prefix in shared memory; units without keys
    // sort last.
    const bool snake = !deep && max_nb <= kMaxWholeBlocks;
    int *order = sm_pre;
    if (snake) {
        constexpr int NBK = kMaxWholeBlocks + 1;  // buckets: 16 - blocks, so most blocks first
        int *cnt = len_sm + ((units + 31) & ~31);  // [NBK][blockDim.x], also in the idle ring
        for (int k = 0; k < NBK; ++k) cnt[k * blockDim.x + tid] = 0;
        for (int u = u_lo; u < u_hi; ++u) ++cnt[(kMaxWholeBlocks - ((len_sm[u] + 15) >> 4)) * blockDim.x + tid];
        __syncthreads();
        // exclusive scan of cnt in memory order (bucket-major, then thread): thread t takes
        // entries [NBK t, NBK (t + 1))
        int loc = 0;
        for (int k = 0; k < NBK; ++k) loc += cnt[tid * NBK + k];
        int f = loc;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            const int nf = __shfl_up_sync(0xffffffffu, f, o);
            if (lane >= o) f += nf;
        }
        __syncthreads();  // every thread has read its entries (and NB, before the order overwrites pb)
        if (lane == 31) sm_scan[wid] = f;
        __syncthreads();
        int run = f - loc;
        for (int w2 = 0; w2 < wid; ++w2) run += sm_scan[w2];
        for (int k = 0; k < NBK; ++k) {
            const int c2 = cnt[tid * NBK + k];
            cnt[tid * NBK + k] = run;
            run += c2;
        }
        __syncthreads();
        // each thread places its own units, in index order, from its own column of cnt
        for (int u = u_lo; u < u_hi; ++u) order[cnt[(kMaxWholeBlocks - ((len_sm[u] + 15) >> 4)) * blockDim.x + tid]++] = u;
        __syncthreads();
    }
    bool aborted = false;
    {
    const int NWm = deep ? NW / 2 : NW, Sm = deep ? 2 * S : S;  // NWm * Sm == NW * S either way
    const uint32_t my_ring = ring0 + (uint32_t)wid * Sm * STAGE;
    // working warps: every one gets at least kMinBlocksPerWarp blocks (or all warps work)
    const int W = max(1, min(NWm * (int)gridDim.x, NB / kMinBlocksPerWarp));
    const int g = lane >> 2, c = lane & 3;
    const bool out_bf16 = a.out_bf16 != 0;
    auto wstart = [&](int w) { return (int)((long long)w * NB / W); };  // ideal first block of warp w
    auto owner = [&](int b) { return (int)(((long long)(b + 1) * W - 1) / NB); };  // ideal owner of block b

    // A piece: the part of unit u inside one warp's block range.  A unit cut between warps
    // wf .. wf+nsplit-1 keeps warp w's partial in slot 2w (the warp's first piece) or 2w+1
    // (its last piece): only those two pieces of a warp can be partial.  Only long units
    // are cut, and no range start moves inside a long unit, so there the ideal owners hold.
    struct Item {
        int u, pu, hp, ub, wf, nsplit, slot, slot0, le, k0, k1, Lapp, nblk;  // pu, hp: cache unit, head part
    };
    auto last_le = [](const int *pre, int units_, int d) {  // largest u with pre[u] <= d
        int lo = 0, hi = units_ - 1;
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (pre[mid] <= d) lo = mid; else hi = mid - 1;
        }
        return lo;
    };
    auto snap = [&](int b) {  // a range start inside a short unit moves to its nearer end
        if (b >= NB) return NB;
        const int u = last_le(pb, units, b);
        const int ub = pb[u], ue = pb[u + 1];
        if (ue - ub > kMaxWholeBlocks) return b;
        return b - ub <= ue - b ? ub : ue;
    };
    // static deal interleaved across CTAs (warp wid of every CTA before warp wid+1 of
    // any): with fewer working warps than warps the work still spreads over all SMs
    const int gw = wid * (int)gridDim.x + (int)blockIdx.x;
    const bool working = gw < W && !snake;
    const int b_end = working ? snap(wstart(gw + 1)) : 0;
    int b_next = working ? snap(wstart(gw)) : 0;
    int eu = gw;  // next unit this warp checks for emptiness (empty units: no blocks)
    const int Ws = min(NW * (int)gridDim.x, n_ne);  // snake deal: warps with units
    int sk = 0, spos = gw < Ws ? gw : n_ne;          // round and sorted position of the next unit
    auto next_item = [&]() {
        Item it;
        it.nblk = -1;  // no item
        if (snake) {
            if (spos < n_ne) {
                const int u = order[spos];
                const int le_raw = eff_len(u);
                it.u = u;
                it.pu = cache_unit(u);
                it.hp = head_part(u);
                it.ub = 0;
                it.le = le_raw >= 0 ? le_raw : 0;
                it.Lapp = (le_raw >= 0 && a.append) ? it.le - 1 : -1;
                it.k0 = 0;
                it.k1 = it.le;
                it.nblk = (it.le + 15) >> 4;
                it.wf = gw;
                it.nsplit = 1;
                it.slot = it.slot0 = 0;
                ++sk;
                spos = sk * Ws + ((sk & 1) ? Ws - 1 - gw : gw);
                return it;
            }
            while (n_ne + eu < units) {  // units without keys: zero output, lse = -inf
                const int u = order[n_ne + eu];
                eu += total_warps;
                it.u = u;
                it.pu = cache_unit(u);
                it.hp = head_part(u);
                it.ub = 0;
                it.le = 0;
                it.Lapp = -1;
                it.k0 = it.k1 = 0;
                it.nblk = 0;
                it.wf = 0;
                it.nsplit = 1;
                it.slot = it.slot0 = 0;
                return it;
            }
            return it;
        }
        if (b_next < b_end) {
            const int u = last_le(pb, units, b_next);  // the nonempty unit holding block b_next
            const int ub = pb[u], ue = pb[u + 1];
            const int bend = min(b_end, ue);
            const int le_raw = eff_len(u);
            it.u = u;
            it.pu = cache_unit(u);
            it.hp = head_part(u);
            it.ub = ub;
            it.le = le_raw >= 0 ? le_raw : 0;
            it.Lapp = (le_raw >= 0 && a.append) ? it.le - 1 : -1;
            it.k0 = (b_next - ub) * 16;
            it.k1 = min((bend - ub) * 16, it.le);
            it.nblk = bend - b_next;
            if (ue - ub <= kMaxWholeBlocks) {  // a short unit: always whole
                it.wf = gw;
                it.nsplit = 1;
                it.slot = it.slot0 = 0;
            } else {
                it.wf = owner(ub);
                it.nsplit = owner(ue - 1) - it.wf + 1;
                it.slot0 = 2 * it.wf + (snap(wstart(it.wf)) < ub ? 1 : 0);  // warp wf's slot
                it.slot = gw == it.wf ? it.slot0 : 2 * gw;
            }
            b_next = bend;
            return it;
        }
        while (eu < units) {  // units without keys: zero output, lse = -inf
            const int u = eu;
            eu += total_warps;
            if (pb[u + 1] == pb[u]) {
                const int le_raw = eff_len(u);
                it.u = u;
                it.pu = cache_unit(u);
                it.hp = head_part(u);
                it.ub = pb[u];
                it.le = 0;
                it.Lapp = -1;
                it.k0 = it.k1 = 0;
                it.nblk = 0;
                it.wf = 0;
                it.nsplit = 1;
                it.slot = it.slot0 = 0;
                (void)le_raw;
                return it;
            }
        }
        return it;
    };

    // Q fragments of an item (rows g < G), head dim permuted to match the K chunks:
    // k-step j = 4*hh + 2*e + half takes elements 64*hh + 16c + 8e + 4*half + {0,1} (a0)
    // and + {2,3} (a2).
    auto load_q = [&](const Item &it, uint32_t (&qa)[D / 16][2]) {
        const long qrow = (long)(it.pu / a.Hkv) * a.Hq + (long)(it.pu % a.Hkv) * a.G + it.hp * GS;
        const int nh = min(GS, a.G - it.hp * GS);
        const __nv_bfloat16 *qp = reinterpret_cast<const __nv_bfloat16 *>(a.q) + (qrow + g) * D;
#pragma unroll
        for (int hh = 0; hh < HALVES; ++hh)
#pragma unroll
            for (int e = 0; e < 2; ++e) {
                uint4 wv = make_uint4(0, 0, 0, 0);
                if (g < nh) wv = *reinterpret_cast<const uint4 *>(qp + 64 * hh + 16 * c + 8 * e);
                const int j = 4 * hh + 2 * e;
                qa[j][0] = wv.x;
                qa[j][1] = wv.y;
                qa[j + 1][0] = wv.z;
                qa[j + 1][1] = wv.w;
            }
    };

    // K and V rows are read once per launch: evict them first, so they do not displace the
    // queries, the outputs, the partials or the next kernels' inputs from L2 (a medium cache,
    // 1792 units of 200-400 rows, went from 62.1 to 56.6 us; the 7B-class launch 1.5% faster)
    const uint64_t kv_policy = l2_evict_first_policy();
    // ---- block stream: lane 0 keeps up to S blocks in flight, running from the current
    // item into the next one (grabbed one item ahead) so no refill bubble opens between
    // items; the warp consumes blocks in issue order.
    uint32_t issued = 0, consumed = 0;
    uint32_t p_slot = 0, c_slot = 0, c_par = 0;  // ring slot of the next issue / next wait, wait phase
    Item cur = next_item();
    Item nxt;
    nxt.nblk = -1;  // looked up below, after the first copies are out
    Item pit = cur;  // item the producer is issuing from
    int pblk = 0;
    bool p_on_next = false;
    auto can_issue = [&]() {
        if (pblk < pit.nblk) return true;
        if (!p_on_next && nxt.nblk > 0) {
            pit = nxt;
            pblk = 0;
            p_on_next = true;
            return true;
        }
        return false;
    };
    auto issue = [&]() {
        const uint32_t slot = p_slot;
        if (lane == 0) {
            const uint32_t bar = (uint32_t)__cvta_generic_to_shared(&bars[wid * Sm + slot]);
            const uint32_t dst = my_ring + slot * STAGE;
            const int y = pit.pu * a.L_cap + pit.k0 + 16 * pblk;
            fence_async_shared();
            mbar_expect_tx(bar, STAGE);
#pragma unroll
            for (int hh = 0; hh < HALVES; ++hh) {
                tma_load_2d_hint(dst + hh * TILE, &tmK, 64 * hh, y, bar, kv_policy);
                tma_load_2d_hint(dst + (HALVES + hh) * TILE, &tmV, 64 * hh, y, bar, kv_policy);
            }
        }
        ++pblk;
        ++issued;
        if (++p_slot == (uint32_t)Sm) p_slot = 0;
    };
    // the first piece's copies go out before the next piece is looked up (that lookup
    // reads a length from global memory)
    __syncwarp();
    while (issued < (uint32_t)Sm && pblk < pit.nblk) issue();
    uint32_t qa_n[D / 16][2];  // query fragments of the next item to start
    if (cur.nblk >= 0) load_q(cur, qa_n);
    nxt = cur.nblk >= 0 ? next_item() : cur;
    // the launch's queries into the window ring (row rs of every query head's `slots`
    // rows): each warp copies an equal share of 16-byte chunks while its first copies
    // are in flight
    if (a.qring != nullptr && rs >= 0) {
        constexpr int CH = D / 8;  // 16-byte chunks of a bf16 query row
        const long long n16 = a.nq_rows * CH;
        const int tw = (int)gridDim.x * NW, me = (int)blockIdx.x * NW + wid;
        const long long per = (n16 + tw - 1) / tw;
        const long long c0 = min(n16, (long long)me * per), c1 = min(n16, c0 + per);
        const uint4 *src = reinterpret_cast<const uint4 *>(a.q);
        uint4 *dst = reinterpret_cast<uint4 *>(a.qring);
        for (long long cb = c0; cb < c1; cb += 32 * 8) {
            uint4 v[8];  // all loads in flight before the stores
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const long long c = cb + 32 * k + lane;
                if (c < c1) v[k] = __ldcg(src + c);
            }
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const long long c = cb + 32 * k + lane;
                if (c < c1) dst[(c / CH * a.slots + rs) * CH + c % CH] = v[k];
            }
        }
    }

    while (cur.nblk >= 0) {
        const int u = cur.u, k0 = cur.k0, k1 = cur.k1, Lapp = cur.Lapp;
        const int nsplit = cur.nsplit, item = cur.slot, wf = cur.wf, slot0 = cur.slot0;  // partial slots
        const int pu = cur.pu;  // the cache unit
        const long lb = pu / a.Hkv;
        const int h = pu % a.Hkv;
        const int G = min(GS, a.G - cur.hp * GS);
        const __nv_bfloat16 *kn = a.append ? reinterpret_cast<const __nv_bfloat16 *>(a.k_new) + (long)pu * D : nullptr;
        const __nv_bfloat16 *vn = a.append ? reinterpret_cast<const __nv_bfloat16 *>(a.v_new) + (long)pu * D : nullptr;
        const long qrow0 = lb * a.Hq + (long)h * a.G + cur.hp * GS;
        const int row0 = pu * a.L_cap;  // first tensor-map row of this unit
        // this lane's 16-byte chunk of the appended row (K for lanes < D/8, V for the next
        // D/8), loaded now so that neither the stage patch nor the cache write below waits
        // on global memory
        uint4 app = make_uint4(0, 0, 0, 0);
        if (Lapp >= k0 && Lapp < k1 && lane < 2 * (D / 8)) {
            const bool isv = lane >= D / 8;
            app = *reinterpret_cast<const uint4 *>((isv ? vn : kn) + (isv ? lane - D / 8 : lane) * 8);
        }

        // start this item's copies before the wait on its query registers below
        __syncwarp();
        while (issued - consumed < (uint32_t)Sm && can_issue()) issue();
        uint32_t qa[D / 16][2];
#pragma unroll
        for (int j = 0; j < D / 16; ++j) {
            qa[j][0] = qa_n[j][0];
            qa[j][1] = qa_n[j][1];
        }
        if (nxt.nblk >= 0) load_q(nxt, qa_n);  // the next item's queries load while this one streams
        float o[MT][4];
#pragma unroll
        for (int t = 0; t < MT; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
        float m = -INFINITY, l = 0.f;

        for (int bi = 0; bi < cur.nblk; ++bi) {
            __syncwarp();
            while (issued - consumed < (uint32_t)Sm && can_issue()) issue();
            const uint32_t slot = c_slot, parity = c_par;
            const uint32_t bar = (uint32_t)__cvta_generic_to_shared(&bars[wid * Sm + slot]);
            if (!mbar_wait_bounded(bar, parity, kSpinLimit)) {  // a copy never landed: report, drain, stop
                if (lane == 0) raise_error(a.err, ERR_INTERNAL);
                for (uint32_t q2 = consumed + 1; q2 < issued; ++q2)
                    mbar_wait_bounded((uint32_t)__cvta_generic_to_shared(&bars[wid * Sm + q2 % Sm]), (q2 / Sm) & 1u,
                                      kSpinLimit);
                aborted = true;
                break;
            }
            const int kb = k0 + 16 * bi;
            const uint32_t Ks = my_ring + slot * STAGE, Vs = Ks + HALVES * TILE;
            // patch the stage: zero V rows past the item (K rows there are masked), and
            // put the appended row (not yet in the cache) in place
            if (kb + 16 > k1 || (Lapp >= kb && Lapp < kb + 16)) {
                const int zr = max(k1 - kb, 0);
                for (int p = lane; p < (16 - zr) * HALVES * 8; p += 32) {
                    const int rr = zr + p / (HALVES * 8), ch = p % (HALVES * 8);
                    sts_u4(Vs + (ch >> 3) * TILE + swz(rr, ch & 7), make_uint4(0, 0, 0, 0));
                }
                if (Lapp >= kb && Lapp < kb + 16 && lane < 2 * HALVES * 8) {
                    const int rr = Lapp - kb;
                    const bool isv = lane >= HALVES * 8;
                    const int ch = isv ? lane - HALVES * 8 : lane;
                    sts_u4((isv ? Vs : Ks) + (ch >> 3) * TILE + swz(rr, ch & 7), app);
                }
                __syncwarp();
            }
            // four accumulators (keys 0-7 / 8-15, even / odd k-steps): dependent MMA chains
            // of D/32 instead of D/16
            float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
            float t0[4] = {0.f, 0.f, 0.f, 0.f}, t1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int hh = 0; hh < HALVES; ++hh)
#pragma unroll
                for (int e = 0; e < 2; ++e) {
                    const uint4 ka = lds_u4(Ks + hh * TILE + swz(g, 2 * c + e));
                    const uint4 kc = lds_u4(Ks + hh * TILE + swz(8 + g, 2 * c + e));
                    const int j = 4 * hh + 2 * e;
                    mma_bf16(s0, qa[j][0], 0u, qa[j][1], 0u, ka.x, ka.y);
                    mma_bf16(s1, qa[j][0], 0u, qa[j][1], 0u, kc.x, kc.y);
                    mma_bf16(t0, qa[j + 1][0], 0u, qa[j + 1][1], 0u, ka.z, ka.w);
                    mma_bf16(t1, qa[j + 1][0], 0u, qa[j + 1][1], 0u, kc.z, kc.w);
                }
#pragma unroll
            for (int i = 0; i < 2; ++i) {
                s0[i] += t0[i];
                s1[i] += t1[i];
            }
            // scores of query g for keys kb+2c, kb+2c+1, kb+8+2c, kb+9+2c
            const int kA = kb + 2 * c, kB = kb + 8 + 2 * c;
            const float x0 = (kA < k1) ? s0[0] * a.c2 : -INFINITY;
            const float x1 = (kA + 1 < k1) ? s0[1] * a.c2 : -INFINITY;
            const float x2 = (kB < k1) ? s1[0] * a.c2 : -INFINITY;
            const float x3 = (kB + 1 < k1) ? s1[1] * a.c2 : -INFINITY;
            float mb = fmaxf(fmaxf(x0, x1), fmaxf(x2, x3));
            mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, 1));
            mb = fmaxf(mb, __shfl_xor_sync(0xffffffffu, mb, 2));
            // Lazy rescale: a row's reference max m moves only when a block max exceeds it
            // by more than 2^kLazyLog2, so probabilities against a stale m stay <= 2^8
            // (exact in fp32, and the bf16 hi + lo split keeps 16 bits of them); the
            // output rescale below then runs on few blocks.  m, l and o stay consistent, so
            // o / l and lse = m + log2 l are the same quantities as with an exact max.
            const bool grow = mb > m + kLazyLog2;
            if (__any_sync(0xffffffffu, grow)) {
                const float mn = grow ? mb : m;
                const float alpha = grow ? fast_exp2(m - mn) : 1.f;  // m = -inf gives 0
                l *= alpha;
                m = mn;
                const float a0 = __shfl_sync(0xffffffffu, alpha, (2 * c) * 4);
                const float a1 = __shfl_sync(0xffffffffu, alpha, (2 * c + 1) * 4);
#pragma unroll
                for (int t = 0; t < MT; ++t) {
                    o[t][0] *= a0;
                    o[t][1] *= a1;
                    o[t][2] *= a0;
                    o[t][3] *= a1;
                }
            }
            const float base = (m == -INFINITY) ? 0.f : m;
            const float p0 = fast_exp2(x0 - base), p1 = fast_exp2(x1 - base);
            const float p2 = fast_exp2(x2 - base), p3 = fast_exp2(x3 - base);
            l += (p0 + p1) + (p2 + p3);
            // P enters the PV product as bf16 hi + lo parts (two MMAs), which keeps about
            // 16 significant bits of each probability instead of 8.
            uint32_t ph0, ph1, pl0, pl1;
            split_bf16(p0, p1, ph0, pl0);
            split_bf16(p2, p3, ph1, pl1);
#pragma unroll
            for (int hh = 0; hh < HALVES; ++hh) {
                const uint4 v0 = lds_u4(Vs + hh * TILE + swz(2 * c, g));
                const uint4 v1 = lds_u4(Vs + hh * TILE + swz(2 * c + 1, g));
                const uint4 v2 = lds_u4(Vs + hh * TILE + swz(2 * c + 8, g));
                const uint4 v3 = lds_u4(Vs + hh * TILE + swz(2 * c + 9, g));
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    const uint32_t W0 = word(v0, x), W1 = word(v1, x), W2 = word(v2, x), W3 = word(v3, x);
                    const uint32_t A0 = __byte_perm(W0, W1, 0x5410), A1 = __byte_perm(W0, W1, 0x7632);
                    const uint32_t A2 = __byte_perm(W2, W3, 0x5410), A3 = __byte_perm(W2, W3, 0x7632);
                    mma_bf16(o[4 * hh + x], A0, A1, A2, A3, ph0, ph1);
                    mma_bf16(o[4 * hh + x], A0, A1, A2, A3, pl0, pl1);
                }
            }
            ++consumed;
            if (++c_slot == (uint32_t)Sm) {
                c_slot = 0;
                c_par ^= 1u;
            }
        }
        if (aborted) break;

        l += __shfl_xor_sync(0xffffffffu, l, 1);
        l += __shfl_xor_sync(0xffffffffu, l, 2);

        // the warp that covers the appended index writes the new row into the cache
        if (Lapp >= k0 && Lapp < k1 && lane < 2 * (D / 8) && cur.hp == 0) {
            const bool isv = lane >= D / 8;
            const int pc = isv ? lane - D / 8 : lane;
            __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(isv ? a.V : a.K) + ((long)row0 + Lapp) * D + pc * 8;
            *reinterpret_cast<uint4 *>(dst) = app;
        }

        const int q0 = 2 * c, q1 = 2 * c + 1;
        const float l0 = __shfl_sync(0xffffffffu, l, q0 * 4), l1 = __shfl_sync(0xffffffffu, l, q1 * 4);
        if (nsplit == 1) {
            const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f, inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
            for (int hh = 0; hh < HALVES; ++hh) {
                const long d0 = 64 * hh + 8 * g;
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    if (q0 < G) {
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + q0) * D + d0 + 2 * x, o[4 * hh + x][0] * inv0);
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + q0) * D + d0 + 2 * x + 1, o[4 * hh + x][2] * inv0);
                    }
                    if (q1 < G) {
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + q1) * D + d0 + 2 * x, o[4 * hh + x][1] * inv1);
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + q1) * D + d0 + 2 * x + 1, o[4 * hh + x][3] * inv1);
                    }
                }
            }
            if (c == 0 && g < G) put_lse(a, rs, qrow0 + g, l > 0.f ? (m + log2f(l)) * kLn2 : -INFINITY);
        } else {
            float *po = a.part_o + (size_t)item * GS * D;
#pragma unroll
            for (int hh = 0; hh < HALVES; ++hh) {
                const int d0 = 64 * hh + 8 * g;
                if (q0 < G) {
                    float4 *dst = reinterpret_cast<float4 *>(po + (size_t)q0 * D + d0);
                    dst[0] = make_float4(o[4 * hh + 0][0], o[4 * hh + 0][2], o[4 * hh + 1][0], o[4 * hh + 1][2]);
                    dst[1] = make_float4(o[4 * hh + 2][0], o[4 * hh + 2][2], o[4 * hh + 3][0], o[4 * hh + 3][2]);
                }
                if (q1 < G) {
                    float4 *dst = reinterpret_cast<float4 *>(po + (size_t)q1 * D + d0);
                    dst[0] = make_float4(o[4 * hh + 0][1], o[4 * hh + 0][3], o[4 * hh + 1][1], o[4 * hh + 1][3]);
                    dst[1] = make_float4(o[4 * hh + 2][1], o[4 * hh + 2][3], o[4 * hh + 3][1], o[4 * hh + 3][3]);
                }
            }
            if (c == 0 && g < G) {
                a.part_ml[((size_t)item * GS + g) * 2 + 0] = m;
                a.part_ml[((size_t)item * GS + g) * 2 + 1] = l;
            }
            // publish: the warp barrier orders every lane's partial writes before lane 0's
            // release; the last arriver's acquire (and the barrier after it) orders its reads
            __syncwarp();
            int old = 0;
            if (lane == 0) old = atom_add_acq_rel(&a.counters[2 + u], 1);
            old = __shfl_sync(0xffffffffu, old, 0);
            __syncwarp();
            if (old == nsplit - 1) {  // last item of this unit: merge the partials
                if (lane == 0) a.counters[2 + u] = 0;  // every piece has counted: clear for the next launch
                // pass 1: per-query-head maxima, lanes over splits (independent loads)
                float Mq[8];
#pragma unroll
                for (int qq = 0; qq < 8; ++qq) Mq[qq] = -INFINITY;
                for (int sb = 0; sb < nsplit; sb += 32) {
                    const int s2 = sb + lane;
                    if (s2 < nsplit) {
#pragma unroll
                        for (int qq = 0; qq < 8; ++qq)
                            if (qq < G)
                                Mq[qq] = fmaxf(Mq[qq], __ldcg(a.part_ml + ((size_t)(s2 ? 2 * (wf + s2) : slot0) * GS + qq) * 2));
                    }
                }
#pragma unroll
                for (int qq = 0; qq < 8; ++qq) Mq[qq] = warp_max(Mq[qq]);
                // pass 2: every lane owns 4 head-dim elements of all G heads; one sweep over
                // the splits with all of a split's loads issued together
                constexpr int PER = D / 32;
                float acc[8][PER], Lq[8];
#pragma unroll
                for (int qq = 0; qq < 8; ++qq) {
                    Lq[qq] = 0.f;
#pragma unroll
                    for (int e = 0; e < PER; ++e) acc[qq][e] = 0.f;
                }
#pragma unroll 2
                for (int s2 = 0; s2 < nsplit; ++s2) {
                    const size_t it0 = (size_t)(s2 ? 2 * (wf + s2) : slot0) * GS;
#pragma unroll
                    for (int qq = 0; qq < 8; ++qq) {
                        if (qq < G && Mq[qq] != -INFINITY) {
                            const float2 ml = __ldcg(reinterpret_cast<const float2 *>(a.part_ml) + it0 + qq);
                            const float wt = fast_exp2(ml.x - Mq[qq]);
                            Lq[qq] += ml.y * wt;
                            const float *src = a.part_o + (it0 + qq) * D + lane * PER;
                            if constexpr (PER == 4) {
                                const float4 ov = __ldcg(reinterpret_cast<const float4 *>(src));
                                acc[qq][0] += ov.x * wt;
                                acc[qq][1] += ov.y * wt;
                                acc[qq][2] += ov.z * wt;
                                acc[qq][3] += ov.w * wt;
                            } else {
#pragma unroll
                                for (int e = 0; e < PER; ++e) acc[qq][e] += __ldcg(src + e) * wt;
                            }
                        }
                    }
                }
#pragma unroll
                for (int qq = 0; qq < 8; ++qq) {
                    if (qq < G) {
                        const float inv = Lq[qq] > 0.f ? 1.f / Lq[qq] : 0.f;
#pragma unroll
                        for (int e = 0; e < PER; ++e)
                            store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + qq) * D + lane * PER + e,
                                                     acc[qq][e] * inv);
                        if (lane == 0)
                            put_lse(a, rs, qrow0 + qq, Lq[qq] > 0.f ? (Mq[qq] + log2f(Lq[qq])) * kLn2 : -INFINITY);
                    }
                }
            }
        }
        // advance: the producer may already be streaming the next item's blocks
        cur = nxt;
        nxt = cur.nblk >= 0 ? next_item() : cur;
        if (p_on_next) {
            p_on_next = false;
        } else {
            pit = cur;
            pblk = 0;
        }
    }
    }

    // Every warp, stopped early or not, counts itself done with one 64-bit add on the
    // pair counters[0..1]: +1 on counters[1] (warps done) and, for a stopped warp, +1 on
    // counters[0] (warps stopped), so the value the add returns tells the last warp of
    // every stop before it, with no further read.  The last one has every other warp
    // behind it: it advances the lengths (every plan has been read by then) and clears
    // the counters, so a launch leaves the workspace's counters zero as it found them,
    // also after a stop.
    unsigned long long dc = 0;
    const bool stopped = __shfl_sync(0xffffffffu, aborted, 0);
    __syncwarp();
    if (lane == 0)
        dc = atom_add_acq_rel_u64(reinterpret_cast<unsigned long long *>(a.counters),
                                  (1ull << 32) | (stopped ? 1ull : 0ull));
    dc = __shfl_sync(0xffffffffu, dc, 0);
    __syncwarp();
    if ((int)(dc >> 32) == total_warps - 1) {
        const bool any_stop = stopped || (uint32_t)dc != 0u;
        if (any_stop) {  // tickets of units whose pieces stopped early may still count
            for (int u = lane; u < units; u += 32) a.counters[2 + u] = 0;
        } else if (a.append) {
            // 16 independent loads per lane in flight before any store, of 4 lengths each
            // when lens is 16-byte aligned: one L2 round trip for up to 2048 units
            constexpr int BATCH = 16;
            const int cu = units / HS;  // cache units
            const int n4 = (reinterpret_cast<uintptr_t>(a.lens) & 15u) == 0 ? cu / 4 : 0;
            int4 *l4 = reinterpret_cast<int4 *>(a.lens);
            for (int i0 = 0; i0 < n4; i0 += 32 * BATCH) {
                int4 L[BATCH];
#pragma unroll
                for (int k = 0; k < BATCH; ++k) {
                    const int i = i0 + 32 * k + lane;
                    L[k] = i < n4 ? __ldcg(l4 + i) : make_int4(-1, -1, -1, -1);
                }
#pragma unroll
                for (int k = 0; k < BATCH; ++k) {
                    const int i = i0 + 32 * k + lane;
                    if (i < n4) {
                        int4 v = L[k];
                        v.x += unit_ok(v.x, a.L_cap, a.append) ? 1 : 0;
                        v.y += unit_ok(v.y, a.L_cap, a.append) ? 1 : 0;
                        v.z += unit_ok(v.z, a.L_cap, a.append) ? 1 : 0;
                        v.w += unit_ok(v.w, a.L_cap, a.append) ? 1 : 0;
                        l4[i] = v;
                    }
                }
            }
            for (int u0 = 4 * n4; u0 < cu; u0 += 32 * BATCH) {  // the rest (or all) one length at a time
                int L[BATCH];
#pragma unroll
                for (int k = 0; k < BATCH; ++k) {
                    const int u = u0 + 32 * k + lane;
                    L[k] = u < cu ? __ldcg(a.lens + u) : -1;
                }
#pragma unroll
                for (int k = 0; k < BATCH; ++k) {
                    const int u = u0 + 32 * k + lane;
                    if (u < cu && unit_ok(L[k], a.L_cap, a.append)) a.lens[u] = L[k] + 1;
                }
            }
        }
        __syncwarp();
        if (lane == 0) {
            *reinterpret_cast<unsigned long long *>(a.counters) = 0ull;
            if (rs >= 0 && a.advance) *a.slot = (rs + 1) % a.slots;  // every warp has read the row by now
        }
    }
}

// The launch's queries into the window ring after the SIMT decode: chunk c (16 bytes)
// of query row c / ch goes to row *slot of that head's `slots` rows.
__global__ void qring_copy(const uint4 *__restrict__ q, uint4 *__restrict__ qring, long long n16, int ch, int slots,
                           const long long *slot)
{
    const long long s = *slot;
    if (s < 0 || s >= slots) return;  // the decode has reported the slot
    for (long long c = (long long)blockIdx.x * blockDim.x + threadIdx.x; c < n16; c += (long long)gridDim.x * blockDim.x)
        qring[(c / ch * slots + s) * ch + c % ch] = q[c];
}

// The ring slot's advance after the SIMT decode (its CTAs have no last-warp step).
__global__ void ring_advance(long long *slot, int slots)
{
    const long long s = *slot;
    if (s >= 0 && s < slots) *slot = (s + 1) % slots;
}

// ---------------------------------------------------------------- host side
// [rows, d] bf16 view of a cache tensor, 16-row x 64-column boxes, 128-byte swizzle.
static bool encode_cache_map(CUtensorMap *map, const void *base, unsigned long long rows, int d)
{
    return encode_bf16_2d(map, base, rows, d, 64, 16);
}

cudaError_t launch_decode(const reco_kv &kv, const void *q, const void *k_new, const void *v_new,
                          int32_t *lens, float scale, void *out, reco_dtype out_dtype, float *lse,
                          const DecodeWs &ws, unsigned *err, cudaStream_t s, float *ring, int slots,
                          long long *slot, void *qring)
{
    DecodeArgs a;
    a.K = kv.k;
    a.V = kv.v;
    a.q = q;
    a.k_new = k_new;
    a.v_new = v_new;
    a.lens = lens;
    a.out = out;
    a.lse = lse;
    a.counters = ws.counters;
    a.part_ml = ws.part_ml;
    a.part_o = ws.part_o;
    a.units = kv.n_layers * kv.B * kv.H_kv;
    a.Hq = kv.H_q;
    a.Hkv = kv.H_kv;
    a.G = kv.H_q / kv.H_kv;
    a.L_cap = kv.L_cap;
    a.append = (k_new && v_new) ? 1 : 0;
    a.out_bf16 = out_dtype == RECO_BF16 ? 1 : 0;
    a.c2 = scale * kLog2e;
    a.err = err;
    a.ring = ring;
    a.slot = slot;
    a.slots = slots;
    a.nq = (long long)kv.n_layers * kv.B * kv.H_q;
    a.qring = ring ? qring : nullptr;
    a.q_bytes = kv.dtype == RECO_F32 ? 4 : 2;
    a.nq_rows = a.nq;
    a.advance = 1;
    // partial slots: two per warp of the grid
    const bool slots_fit = 2LL * device_sm_count() * kDecodeWarps <= (long long)ws.part_slots;
    // the TMA path takes up to 8 query heads per unit; a unit of G <= 16 heads is two
    // virtual units of ceil(G / 2) heads each
    a.hs = a.G > 8 ? 2 : 1;
    a.gv = (a.G + a.hs - 1) / a.hs;
    // More units than one plan holds in shared memory run as consecutive launches over
    // contiguous unit ranges (every unit is independent): each part gets its own K/V, q,
    // output, lens and ring pointers, and only the last part advances the ring slot.
    const long long part_units = kMaxTmaUnits / a.hs;  // cache units per launch
    if (kv.dtype == RECO_BF16 && a.G <= 16 && (unsigned long long)std::min<long long>(a.units, part_units) * kv.L_cap <
                                                   (1ull << 31) && slots_fit) {
        const bool two = a.hs == 2;
        const void *fn = kv.d == 64 ? (two ? (const void *)decode_tma<64, 2> : (const void *)decode_tma<64, 1>)
                                    : (two ? (const void *)decode_tma<128, 2> : (const void *)decode_tma<128, 1>);
        const size_t row_b = (size_t)kv.d * 2;  // bf16 cache and query rows
        const size_t out_b = (size_t)kv.d * (out_dtype == RECO_BF16 ? 2 : 4);
        for (long long u0 = 0; u0 < a.units; u0 += part_units) {
            const long long cu = std::min(part_units, (long long)a.units - u0);
            const long long q0 = u0 * a.G;  // first query head of the part
            const unsigned long long rows = (unsigned long long)cu * kv.L_cap;
            CUtensorMap mk, mv;
            const char *kb = static_cast<const char *>(kv.k) + (size_t)u0 * kv.L_cap * row_b;
            const char *vb = static_cast<const char *>(kv.v) + (size_t)u0 * kv.L_cap * row_b;
            if (!encode_cache_map(&mk, kb, rows, kv.d) || !encode_cache_map(&mv, vb, rows, kv.d)) {
                if (u0 == 0) break;  // the SIMT path below takes the whole call
                return cudaErrorInvalidValue;
            }
            DecodeArgs at = a;  // virtual units of this part
            at.units = (int)(cu * a.hs);
            at.K = const_cast<char *>(kb);
            at.V = const_cast<char *>(vb);
            at.q = static_cast<const char *>(q) + (size_t)q0 * row_b;
            at.k_new = k_new ? static_cast<const char *>(k_new) + (size_t)u0 * row_b : nullptr;
            at.v_new = v_new ? static_cast<const char *>(v_new) + (size_t)u0 * row_b : nullptr;
            at.lens = lens + u0;
            at.out = static_cast<char *>(out) + (size_t)q0 * out_b;
            at.lse = lse ? lse + q0 : nullptr;
            at.ring = ring ? ring + q0 : nullptr;  // ring rows keep their full stride nq
            at.qring = a.qring ? static_cast<char *>(a.qring) + (size_t)q0 * slots * row_b : nullptr;
            at.nq_rows = cu * a.G;
            at.advance = u0 + cu >= a.units ? 1 : 0;
            // the counters are zero on entry (zero-filled workspace) and every launch leaves them so
            const size_t smem = kv.d == 64 ? tma_smem_bytes<64>(at.units) : tma_smem_bytes<128>(at.units);
            cudaError_t e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
            if (e != cudaSuccess) return e;
            const int grid = device_sm_count();
            const dim3 blk(kDecodeWarps * 32);
            if (kv.d == 64)
                e = two ? launch_pdl(decode_tma<64, 2>, dim3(grid), blk, smem, s, mk, mv, at)
                        : launch_pdl(decode_tma<64, 1>, dim3(grid), blk, smem, s, mk, mv, at);
            else
                e = two ? launch_pdl(decode_tma<128, 2>, dim3(grid), blk, smem, s, mk, mv, at)
                        : launch_pdl(decode_tma<128, 1>, dim3(grid), blk, smem, s, mk, mv, at);
            if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
            if (u0 + cu >= a.units) return cudaSuccess;
        }
    }
    a.hs = 1;
    a.gv = a.G;
    const unsigned grid = (unsigned)a.units;
    if (kv.dtype == RECO_F32) {
        if (kv.d == 64) decode_simt<float, 64><<<grid, 128, 0, s>>>(a);
        else decode_simt<float, 128><<<grid, 128, 0, s>>>(a);
    } else {
        if (kv.d == 64) decode_simt<__nv_bfloat16, 64><<<grid, 128, 0, s>>>(a);
        else decode_simt<__nv_bfloat16, 128><<<grid, 128, 0, s>>>(a);
    }
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess || !ring) return e;
    if (a.qring) {
        const int ch = kv.d * a.q_bytes / 16;
        const long long n16 = a.nq * ch;
        const unsigned blocks = (unsigned)std::min<long long>((n16 + 255) / 256, 4LL * device_sm_count());
        qring_copy<<<blocks, 256, 0, s>>>(reinterpret_cast<const uint4 *>(q), reinterpret_cast<uint4 *>(a.qring), n16,
                                          ch, slots, slot);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    ring_advance<<<1, 1, 0, s>>>(slot, slots);
    return cudaGetLastError();
}

}  // namespace reco
