// select.cu -- top-m selection and in-place compaction (Sec. 3.2: keep the m_i
// highest-scoring tokens with the latest w always retained, then compress the L
// cached tokens down to m_i).
//
// select_topm: CTAs that walk the (layer, sequence, KV head) units, one unit at a time
// (a unit whose sequence keeps its whole cache is an identity, skipped by the
// compaction).  A 4 x 8-bit radix select
// over order-preserving uint32 keys of the float32 scores finds the (m-w)-th
// largest key T and how many keys equal to T are still needed; one ordered pass
// then emits every candidate with key > T plus the first `need` with key == T in
// index order.  The result is sorted and ties go to the lower index, with no sort.
// select_topm_smem does the same from keys staged in shared memory (units of up to
// kSelectSmemKeys candidates).
//
// compact_rows: CTAs per (K|V, 128-byte column slice) that walk the units, one at a
// time.  kept[] is strictly increasing, so kept[r] >= r (the kernel refuses any index that is not): the source
// of destination r is never a row that an earlier destination overwrote.  Each CTA walks
// its destinations in chunks, in order: a chunk's reads, a barrier, then its writes;
// the next chunk's reads are issued before the current chunk's writes, since their
// sources lie above every row written so far.  Rows with kept[r] == r are not moved.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace reco {

SelectWs select_ws_layout(const reco_kv &kv, void *base)
{
    size_t units = (size_t)kv.n_layers * kv.B * kv.H_kv;
    char *p = (char *)base;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *r = p ? p + off : nullptr;
        off += align256(bytes);
        return r;
    };
    SelectWs ws;
    ws.idx = (int32_t *)take(units * (size_t)kv.L_cap * 4);
    ws.count = (int32_t *)take(units * 4);
    ws.bytes = off;
    return ws;
}

// Most candidates a unit may have for the shared-memory selection (192 KB of keys).
constexpr int kSelectSmemKeys = 48 * 1024;

// Units a walking CTA reads the headers of up front, all loads in flight together (a CTA
// of a boundary call holds a few units, most of which it only skips or copies).
constexpr int kWalkAhead = 64;

// (L, m) of the CTA's units (at most kWalkAhead) into `lm`; the caller synchronises.
__device__ __forceinline__ void walk_headers(int2 *lm, const int32_t *lens, const int32_t *keep, long units, int B,
                                             int Hkv)
{
    for (int i = threadIdx.x; i < kWalkAhead; i += blockDim.x) {
        const long u = blockIdx.x + (long)i * gridDim.x;
        if (u < units) lm[i] = make_int2(lens[u], keep[(int)((u / Hkv) % B)]);
    }
}

__device__ __forceinline__ uint32_t order_key(float f)
{
    uint32_t u = __float_as_uint(f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}

// Exclusive block scan of a 0/1 flag.  `tot` must hold NT/32 + 1 ints.
template <int NT>
__device__ __forceinline__ int block_scan_flag(bool flag, int *tot, int &total)
{
    const unsigned lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    const unsigned bal = __ballot_sync(0xffffffffu, flag);
    const int in_warp = __popc(bal & ((1u << lane) - 1u));
    if (lane == 0) tot[wid] = __popc(bal);
    __syncthreads();
    if (wid == 0) {
        int v = lane < NT / 32 ? tot[lane] : 0;
        int incl = v;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int n = __shfl_up_sync(0xffffffffu, incl, o);
            if ((int)lane >= o) incl += n;
        }
        if (lane < NT / 32) tot[lane] = incl - v;
        if (lane == 31) tot[NT / 32] = incl;
    }
    __syncthreads();
    const int res = tot[wid] + in_warp;
    total = tot[NT / 32];
    __syncthreads();
    return res;
}

template <int NT>
__global__ void __launch_bounds__(NT) select_topm(const float *__restrict__ scores, const int32_t *lens,
                                                  int32_t *lens_out, const int32_t *__restrict__ keep, int w, int B, int Hkv,
                                                  int L_cap, int32_t *__restrict__ idx_out,
                                                  int32_t *__restrict__ count, long units, unsigned *err)
{
    __shared__ int hist[256];
    __shared__ int tot[NT / 32 + 1];
    __shared__ uint32_t s_prefix;
    __shared__ int s_remaining;
    __shared__ int2 s_lm[kWalkAhead];
    wait_prior_grid();  // scores, lens and keep may come from the previous kernels
    walk_headers(s_lm, lens, keep, units, B, Hkv);
    __syncthreads();
    int it = 0;
    for (long u = blockIdx.x; u < units; u += gridDim.x, ++it) {  // a few CTAs per SM walk the units
        const int tid = threadIdx.x, lane = tid & 31;
        const int L = s_lm[it].x, m = s_lm[it].y;  // the grid gives no CTA more than kWalkAhead units
        if (L < w || L > L_cap || m < w || m > L) {
            if (tid == 0) {
                count[u] = 0;
                raise_error(err, (L < w || L > L_cap) ? ERR_LEN : ERR_KEEP);
            }
            continue;
        }
        const int nc = L - w, kc = m - w;
        const float *s = scores + u * L_cap;
        int32_t *idx = idx_out + u * L_cap;
        if (kc == nc) {  // keep everything: identity, nothing moves (the compaction skips it)
            for (int j = tid; j < L; j += NT) idx[j] = j;
            if (tid == 0) count[u] = 0;
            continue;
        }
        uint32_t T = 0xffffffffu;
        int need = 0;
        if (kc > 0) {
            if (tid == 0) {
                s_prefix = 0;
                s_remaining = kc;
            }
            uint32_t mask = 0;
            for (int shift = 24; shift >= 0; shift -= 8) {
                for (int i = tid; i < 256; i += NT) hist[i] = 0;
                __syncthreads();
                const uint32_t prefix = s_prefix;
                const int remaining = s_remaining;
                for (int jb = 0; jb < nc; jb += NT) {
                    const int j = jb + tid;
                    const bool valid = j < nc;
                    const uint32_t key = valid ? order_key(s[j]) : 0u;
                    const bool match = valid && (key & mask) == prefix;
                    const uint32_t bin = (key >> shift) & 255u;
                    if (match) atomicAdd(&hist[bin], 1);
                }
                __syncthreads();
                if (tid < 32) {  // find the bin holding the remaining-th largest key
                    int c8[8], sum = 0;
    #pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        c8[i] = hist[255 - 8 * lane - i];
                        sum += c8[i];
                    }
                    int incl = sum;
    #pragma unroll
                    for (int o = 1; o < 32; o <<= 1) {
                        int n = __shfl_up_sync(0xffffffffu, incl, o);
                        if (lane >= o) incl += n;
                    }
                    int cum = incl - sum;
                    if (cum < remaining && remaining <= incl) {
    #pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            if (cum + c8[i] >= remaining) {
                                s_prefix = prefix | ((uint32_t)(255 - 8 * lane - i) << shift);
                                s_remaining = remaining - cum;
                                break;
                            }
                            cum += c8[i];
                        }
                    }
                }
                mask |= 255u << shift;
                __syncthreads();
            }
            T = s_prefix;
            need = s_remaining;
        }
        int base_pos = 0, base_eq = 0;
        for (int jb = 0; jb < nc; jb += NT) {
            const int j = jb + tid;
            const bool valid = j < nc;
            const uint32_t key = valid ? order_key(s[j]) : 0u;
            const bool gt = valid && key > T;
            const bool eq = valid && key == T;
            int eq_tot, f_tot;
            const int eq_rank = block_scan_flag<NT>(eq, tot, eq_tot) + base_eq;
            const bool flag = gt || (eq && eq_rank < need);
            const int pos = block_scan_flag<NT>(flag, tot, f_tot) + base_pos;
            if (flag) idx[pos] = j;
            base_eq += eq_tot;
            base_pos += f_tot;
        }
        for (int t = tid; t < w; t += NT) idx[kc + t] = nc + t;
        if (tid == 0) {
            count[u] = m;
            if (lens_out) lens_out[u] = m;
        }
        __syncthreads();  // this unit's shared memory is read out before the next unit's fill
    }
}

// The same selection with the unit's keys staged in shared memory once (all loads in
// flight), the radix passes run from there, and the ordered emit done by warp-contiguous
// segments: one counting sweep, one scan of the 32 warps' counts, one writing sweep.
template <int NT>
__global__ void __launch_bounds__(NT) select_topm_smem(const float *__restrict__ scores, const int32_t *lens,
                                                       int32_t *lens_out, const int32_t *__restrict__ keep, int w, int B, int Hkv,
                                                       int L_cap, int32_t *__restrict__ idx_out,
                                                       int32_t *__restrict__ count, long units, unsigned *err)
{
    static_assert(NT == 1024, "one warp per lane of the warp-count scan");
    constexpr int NW = NT / 32;
    extern __shared__ uint32_t keys[];  // [L - w]
    __shared__ int hist[256];
    __shared__ int w_gt[NW], w_eq[NW];
    __shared__ uint32_t s_prefix;
    __shared__ int s_remaining;
    __shared__ int2 s_lm[kWalkAhead];
    wait_prior_grid();  // scores, lens and keep may come from the previous kernels
    walk_headers(s_lm, lens, keep, units, B, Hkv);
    __syncthreads();
    int it = 0;
    for (long u = blockIdx.x; u < units; u += gridDim.x, ++it) {  // a few CTAs per SM walk the units
        const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
        const int L = s_lm[it].x, m = s_lm[it].y;  // the grid gives no CTA more than kWalkAhead units
        if (L < w || L > L_cap || m < w || m > L) {
            if (tid == 0) {
                count[u] = 0;
                raise_error(err, (L < w || L > L_cap) ? ERR_LEN : ERR_KEEP);
            }
            continue;
        }
        const int nc = L - w, kc = m - w;
        const float *s = scores + u * L_cap;
        int32_t *idx = idx_out + u * L_cap;
        if (kc == nc) {  // keep everything: identity, nothing moves (the compaction skips it)
            for (int j = tid; j < L; j += NT) idx[j] = j;
            if (tid == 0) count[u] = 0;
            continue;
        }
    #pragma unroll 8
        for (int j = tid; j < nc; j += NT) keys[j] = order_key(__ldcg(s + j));
        if (tid == 0) {
            s_prefix = 0;
            s_remaining = kc;
        }
        __syncthreads();
        uint32_t T = 0xffffffffu;
        int need = 0;
        if (kc > 0) {
            uint32_t mask = 0;
            for (int shift = 24; shift >= 0; shift -= 8) {
                for (int i = tid; i < 256; i += NT) hist[i] = 0;
                __syncthreads();
                const uint32_t prefix = s_prefix;
                const int remaining = s_remaining;
                for (int jb = 0; jb < nc; jb += NT) {
                    const int j = jb + tid;
                    const bool valid = j < nc;
                    const uint32_t key = valid ? keys[j] : 0u;
                    const bool match = valid && (key & mask) == prefix;
                    const uint32_t bin = (key >> shift) & 255u;
                    // plain shared-memory atomics: grouping a warp's equal bins first
                    // (__match_any_sync) cost more than the conflicts it saves (7B-class
                    // selection 109 -> 79 us)
                    if (match) atomicAdd(&hist[bin], 1);
                }
                __syncthreads();
                if (tid < 32) {  // find the bin holding the remaining-th largest key
                    int c8[8], sum = 0;
    #pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        c8[i] = hist[255 - 8 * lane - i];
                        sum += c8[i];
                    }
                    int incl = sum;
    #pragma unroll
                    for (int o = 1; o < 32; o <<= 1) {
                        int n = __shfl_up_sync(0xffffffffu, incl, o);
                        if (lane >= o) incl += n;
                    }
                    int cum = incl - sum;
                    if (cum < remaining && remaining <= incl) {
    #pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            if (cum + c8[i] >= remaining) {
                                s_prefix = prefix | ((uint32_t)(255 - 8 * lane - i) << shift);
                                s_remaining = remaining - cum;
                                break;
                            }
                            cum += c8[i];
                        }
                    }
                }
                mask |= 255u << shift;
                __syncthreads();
            }
            T = s_prefix;
            need = s_remaining;
        }
        // emit in index order: keys > T, then the first `need` keys == T
        const int seg = (nc + NW - 1) / NW;
        const int j0 = min(nc, wid * seg), j1 = min(nc, j0 + seg);
        int n_gt = 0, n_eq = 0;
        for (int jb = j0; jb < j1; jb += 32) {
            const int j = jb + lane;
            const uint32_t key = j < j1 ? keys[j] : 0u;
            n_gt += __popc(__ballot_sync(0xffffffffu, j < j1 && key > T));
            n_eq += __popc(__ballot_sync(0xffffffffu, j < j1 && key == T));
        }
        if (lane == 0) {
            w_gt[wid] = n_gt;
            w_eq[wid] = n_eq;
        }
        __syncthreads();
        if (wid == 0) {  // per warp: equal keys before its segment, and output rows before it
            const int e = w_eq[lane], g = w_gt[lane];
            int e_inc = e;
    #pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int n = __shfl_up_sync(0xffffffffu, e_inc, o);
                if (lane >= o) e_inc += n;
            }
            const int e_base = e_inc - e;
            const int f = g + min(max(need - e_base, 0), e);
            int f_inc = f;
    #pragma unroll
            for (int o = 1; o < 32; o <<= 1) {
                const int n = __shfl_up_sync(0xffffffffu, f_inc, o);
                if (lane >= o) f_inc += n;
            }
            w_eq[lane] = e_base;
            w_gt[lane] = f_inc - f;
        }
        __syncthreads();
        int e_run = w_eq[wid], pos = w_gt[wid];
        const unsigned below = (1u << lane) - 1u;
        for (int jb = j0; jb < j1; jb += 32) {
            const int j = jb + lane;
            const bool valid = j < j1;
            const uint32_t key = valid ? keys[j] : 0u;
            const bool is_eq = valid && key == T;
            const unsigned eb = __ballot_sync(0xffffffffu, is_eq);
            const bool flag = (valid && key > T) || (is_eq && e_run + __popc(eb & below) < need);
            const unsigned fb = __ballot_sync(0xffffffffu, flag);
            if (flag) idx[pos + __popc(fb & below)] = j;
            e_run += __popc(eb);
            pos += __popc(fb);
        }
        for (int t = tid; t < w; t += NT) idx[kc + t] = nc + t;
        if (tid == 0) {
            count[u] = m;
            if (lens_out) lens_out[u] = m;
        }
        __syncthreads();  // this unit's shared memory is read out before the next unit's fill
    }
}

// Rows to move for unit u.  From the selection: its count (0 = leave the unit alone).
// From the caller's keep counts: m = keep[b] when w <= m < L <= L_cap; m == L is the
// no-op; anything else leaves the unit alone and sets the error word.
// `lim` receives the end of the rows a source index may name.
struct CountFromSelect {
    const int32_t *count;
    int L_cap;
    __device__ __forceinline__ int rows(long u, unsigned *, int &lim) const
    {
        lim = L_cap;
        return count[u];
    }
};
struct CountFromKeep {
    const int32_t *lens, *keep;
    int w, B, Hkv, L_cap;
    __device__ __forceinline__ int rows(long u, unsigned *err, int &lim) const
    {
        const int L = lens[u], m = keep[(u / Hkv) % B];
        lim = L;
        if (L < w || L > L_cap || m < w || m > L) {
            if (blockIdx.y == 0 && blockIdx.z == 0)  // one column slice reports (an atomic OR)
                raise_error(err, (L < w || L > L_cap) ? ERR_LEN : ERR_KEEP);
            return 0;
        }
        return m == L ? 0 : m;
    }
};

template <class Count>
__global__ void __launch_bounds__(256, 8) compact_rows(char *K, char *V, const int32_t *__restrict__ idx_all,
                                                    Count cnt, int L_cap, int row_bytes, long units, unsigned *err)
{
    constexpr int P = 8;  // 16-byte pieces per 128-byte slice
    constexpr int U = 2;  // rows per thread in one chunk
    __shared__ int2 s_ml[kWalkAhead];  // (rows to move, source limit) of this CTA's units
    wait_prior_grid();    // kept indices, lens and the cache may belong to the previous kernels
    for (int i = threadIdx.x; i < kWalkAhead; i += blockDim.x) {
        const long u = blockIdx.x + (long)i * gridDim.x;
        if (u < units) {
            int lim;
            const int m = cnt.rows(u, err, lim);
            s_ml[i] = make_int2(m, lim);
        }
    }
    __syncthreads();
    int it = 0;
    for (long u = blockIdx.x; u < units; u += gridDim.x, ++it) {  // a few CTAs per SM walk the units
        const int m = s_ml[it].x, lim = s_ml[it].y;  // the grid gives no CTA more than kWalkAhead units
        if (m == 0) continue;
        char *base = (blockIdx.y == 0 ? K : V) + u * (long)L_cap * row_bytes;
        const int32_t *idx = idx_all + u * L_cap;
        const int rows_per_pass = blockDim.x / P;
        const int my_row = threadIdx.x / P;
        const int off = blockIdx.z * 128 + (threadIdx.x % P) * 16;
        const int step = U * rows_per_pass;  // destinations per chunk
        auto load = [&](int r0, uint4 (&v)[U], int (&dst)[U]) {
    #pragma unroll
            for (int i = 0; i < U; ++i) {
                const int r = r0 + i * rows_per_pass + my_row;
                dst[i] = -1;
                if (r < m) {
                    const int src = idx[r];
                    if (src < r || src >= lim) {  // never trust an index outside [r, lim)
                        raise_error(err, ERR_INTERNAL);
                    } else if (src != r) {
                        v[i] = *reinterpret_cast<const uint4 *>(base + (long)src * row_bytes + off);
                        dst[i] = r;
                    }
                }
            }
        };
        auto store = [&](const uint4 (&v)[U], const int (&dst)[U]) {
    #pragma unroll
            for (int i = 0; i < U; ++i)
                if (dst[i] >= 0) *reinterpret_cast<uint4 *>(base + (long)dst[i] * row_bytes + off) = v[i];
        };
        // Two chunks in registers: the next chunk's reads are issued before this chunk's
        // writes (its sources lie at or above its first destination, above every row this
        // chunk writes); the barrier before a chunk's writes follows every read of it.
        uint4 va[U], vb[U];
        int da[U], db[U];
        load(0, va, da);
        for (int r0 = 0; r0 < m; r0 += 2 * step) {
            load(r0 + step, vb, db);
            __syncthreads();
            store(va, da);
            if (r0 + step >= m) break;
            load(r0 + 2 * step, va, da);
            __syncthreads();
            store(vb, db);
        }
    }
}

// lens[u] = keep[b] for the units reco_compact moved (after every CTA of the unit read lens).
__global__ void compact_set_lens(int32_t *lens, const int32_t *__restrict__ keep, long units, int w, int B,
                                 int Hkv, int L_cap)
{
    wait_prior_grid();
    const long u = (long)blockIdx.x * blockDim.x + threadIdx.x;
    if (u >= units) return;
    const int L = lens[u], m = keep[(u / Hkv) % B];
    if (L >= w && L <= L_cap && m >= w && m < L) lens[u] = m;
}

// CTAs that walk `units` units: as many as the GPU holds at once (`per_unit` CTAs share
// each unit), never more than the units.  Most calls at step boundaries compress a few
// sequences, so most units are skipped at once; a grid of one CTA per unit would spend
// its time scheduling CTAs that exit immediately.
template <typename F>
static unsigned walk_grid(F fn, int threads, size_t smem, long units, int per_unit)
{
    int per_sm = 1;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, fn, threads, smem) != cudaSuccess || per_sm < 1) {
        (void)cudaGetLastError();
        per_sm = 1;
    }
    long ctas = std::max(1L, (long)per_sm * device_sm_count() / per_unit);
    ctas = std::max(ctas, (units + kWalkAhead - 1) / kWalkAhead);  // at most kWalkAhead units per CTA
    return (unsigned)std::min(units, ctas);
}

static cudaError_t launch_select(const reco_kv &kv, const float *scores, const int32_t *lens, int32_t *lens_out,
                                 const int32_t *keep, int w, int32_t *idx, int32_t *count, unsigned *err,
                                 cudaStream_t s)
{
    const long units = (long)kv.n_layers * kv.B * kv.H_kv;
    // keys of a unit staged in shared memory when L_cap - w of them fit
    const size_t key_bytes = (size_t)(kv.L_cap - w) * sizeof(uint32_t);
    if (key_bytes <= kSelectSmemKeys * sizeof(uint32_t)) {
        cudaError_t e = cudaFuncSetAttribute(select_topm_smem<1024>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             (int)kSelectSmemKeys * (int)sizeof(uint32_t));
        if (e != cudaSuccess) return e;
        const unsigned grid = walk_grid(select_topm_smem<1024>, 1024, key_bytes, units, 1);
        e = launch_pdl(select_topm_smem<1024>, dim3(grid), dim3(1024), key_bytes, s, scores, lens, lens_out, keep, w,
                       kv.B, kv.H_kv, kv.L_cap, idx, count, units, err);
        if (e != cudaSuccess) return e;
    } else {
        const unsigned grid = walk_grid(select_topm<1024>, 1024, 0, units, 1);
        cudaError_t e = launch_pdl(select_topm<1024>, dim3(grid), dim3(1024), 0, s, scores, lens, lens_out, keep, w,
                                   kv.B, kv.H_kv, kv.L_cap, idx, count, units, err);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

template <class Count>
static dim3 compact_grid(const reco_kv &kv, int &row_bytes, long &units)
{
    row_bytes = kv.d * (kv.dtype == RECO_F32 ? 4 : 2);
    units = (long)kv.n_layers * kv.B * kv.H_kv;
    const int per_unit = 2 * (row_bytes / 128);  // K and V, 128-byte column slices
    return dim3(walk_grid(compact_rows<Count>, 256, 0, units, per_unit), 2, row_bytes / 128);
}

cudaError_t launch_select_compact(const reco_kv &kv, const float *scores, int32_t *lens,
                                  const int32_t *keep, int w, int32_t *kept_idx, const SelectWs &ws,
                                  unsigned *err, cudaStream_t s)
{
    int32_t *idx = kept_idx ? kept_idx : ws.idx;
    cudaError_t e = launch_select(kv, scores, lens, lens, keep, w, idx, ws.count, err, s);
    if (e != cudaSuccess) return e;
    int row_bytes;
    long units;
    const dim3 grid = compact_grid<CountFromSelect>(kv, row_bytes, units);
    e = launch_pdl(compact_rows<CountFromSelect>, grid, dim3(256), 0, s, (char *)kv.k, (char *)kv.v, (const int32_t *)idx,
                   CountFromSelect{ws.count, kv.L_cap}, kv.L_cap, row_bytes, units, err);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_select_only(const reco_kv &kv, const float *scores, const int32_t *lens, const int32_t *keep,
                               int w, int32_t *kept_idx, const SelectWs &ws, unsigned *err, cudaStream_t s)
{
    return launch_select(kv, scores, lens, nullptr, keep, w, kept_idx, ws.count, err, s);
}

cudaError_t launch_compact(const reco_kv &kv, const int32_t *kept_idx, int32_t *lens, const int32_t *keep, int w,
                           unsigned *err, cudaStream_t s)
{
    int row_bytes;
    long units;
    const dim3 grid = compact_grid<CountFromKeep>(kv, row_bytes, units);
    cudaError_t e = launch_pdl(compact_rows<CountFromKeep>, grid, dim3(256), 0, s, (char *)kv.k, (char *)kv.v,
                               kept_idx, CountFromKeep{lens, keep, w, kv.B, kv.H_kv, kv.L_cap}, kv.L_cap, row_bytes,
                               units, err);
    if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
    e = launch_pdl(compact_set_lens, dim3((unsigned)((units + 255) / 256)), dim3(256), 0, s, lens, keep, units, w, kv.B,
                   kv.H_kv, kv.L_cap);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace reco
