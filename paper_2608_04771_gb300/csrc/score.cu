// score.cu -- Eq. 2 (Sec. 3.2, attention-guided selection): per-KV-head cache scores.
//
// s_j = (1/G) sum_g sum_t softmax_j(scale * q_{g,t} . k_j), window query t at position
// L-w+t seeing keys j <= L-w+t, then a max-pool over the candidate range [0, L-w).
//
// A softmax row needs its max and normaliser over ALL keys before any column can be
// summed, so the scores take two passes over K:
//   pass 1  per (unit, key chunk): per-row running max / sum in the log2 domain
//   combine per (unit, row): merge the chunk partials -> b_r = m_r + log2 Z_r
//   pass 2  per (unit, key chunk): column sums  sum_r 2^(c*l_rj - b_r) / G
//   pool    per (unit, key): max over the clipped window
// This file holds the SIMT passes used for float32 caches (and any shape the tensor-
// core passes do not cover), the combine and pool kernels, and the launcher;
// score_tc.cu holds the bf16 tensor-core (tcgen05) passes.
#include <algorithm>

#include "common.cuh"
#include "internal.h"

namespace reco {

ScoreWs score_ws_layout(const reco_kv &kv, int w, void *base)
{
    size_t units = (size_t)kv.n_layers * kv.B * kv.H_kv;
    size_t R = (size_t)(kv.H_q / kv.H_kv) * w;
    size_t nch = ((size_t)kv.L_cap + kScoreChunk - 1) / kScoreChunk;
    char *p = (char *)base;
    size_t off = 0;
    auto take = [&](size_t bytes) {
        char *r = p ? p + off : nullptr;
        off += align256(bytes);
        return r;
    };
    ScoreWs ws;
    // up to two partials per (unit, chunk, row): the tensor-core pass 1 may split a
    // chunk's key tiles between two epilogue groups
    ws.part_m = (float *)take(units * nch * 2 * R * 4);
    ws.part_z = (float *)take(units * nch * 2 * R * 4);
    ws.rowb = (float *)take(units * R * 4);
    ws.raw = (float *)take(units * (size_t)kv.L_cap * 4);
    ws.ulist = (int32_t *)take(units * 4);
    ws.ucount = (int32_t *)take(4);
    ws.bytes = off;
    return ws;
}

// Pass 1: one thread per window row, its query held in registers; K streamed
// through shared memory 64 rows at a time.
template <typename T, int D>
__global__ void __launch_bounds__(256) score_rowstats_simt(
    const T *__restrict__ q_win, const T *__restrict__ K, const int32_t *__restrict__ lens, ScoreMask mask,
    int w, int G, int Hq, int Hkv, int L_cap, int R, int n_chunks, float c2, float *__restrict__ part_m,
    float *__restrict__ part_z, unsigned *err)
{
    constexpr int KT = 64;
    __shared__ __align__(16) float Ks[KT][D];
    const int chunk = blockIdx.x;
    const long u = blockIdx.y;
    const int r = blockIdx.z * blockDim.x + threadIdx.x;
    const int L = lens[u];
    if (L < w || L > L_cap) {
        if (chunk == 0 && blockIdx.z == 0 && threadIdx.x == 0) raise_error(err, ERR_LEN);
        return;
    }
    if (mask.skip(u, L, w, L_cap)) return;
    const int j0 = chunk * kScoreChunk;
    const int j1 = min(j0 + kScoreChunk, L);
    const long lb = u / Hkv;
    const int h = (int)(u % Hkv);
    const bool row_ok = r < R;
    const int g = row_ok ? r / w : 0, t = row_ok ? r % w : 0;
    const int jmax = L - w + t;
    float q[D];
    {
        const T *qp = q_win + (((lb * Hq) + (long)h * G + g) * w + t) * D;
#pragma unroll
        for (int c = 0; c < D; ++c) q[c] = row_ok ? to_float(qp[c]) : 0.f;
    }
    float m = -INFINITY, z = 0.f;
    const T *Kp = K + u * (long)L_cap * D;
    for (int jt = j0; jt < j1; jt += KT) {
        const int nk = min(KT, j1 - jt);
        __syncthreads();
        for (int e = threadIdx.x; e < KT * D; e += blockDim.x) {
            int jj = e / D, c = e % D;
            Ks[jj][c] = jj < nk ? to_float(Kp[(long)(jt + jj) * D + c]) : 0.f;
        }
        __syncthreads();
        if (row_ok) {
            for (int jj = 0; jj < nk; ++jj) {
                if (jt + jj > jmax) break;
                float s = 0.f;
#pragma unroll
                for (int c = 0; c < D; c += 4) {
                    float4 kv = *reinterpret_cast<const float4 *>(&Ks[jj][c]);
                    s = fmaf(q[c], kv.x, s);
                    s = fmaf(q[c + 1], kv.y, s);
                    s = fmaf(q[c + 2], kv.z, s);
                    s = fmaf(q[c + 3], kv.w, s);
                }
                s *= c2;
                if (s > m) {
                    z = z * fast_exp2(m - s) + 1.f;
                    m = s;
                } else {
                    z += fast_exp2(s - m);
                }
            }
        }
    }
    if (row_ok) {
        size_t o = ((size_t)u * n_chunks + chunk) * R + r;
        part_m[o] = m;
        part_z[o] = z;
    }
}

// Merge the partials of each row (per_chunk of them for each key chunk, laid out
// [unit][chunk][per_chunk][R]) into b_r = m_r + log2(Z_r).
__global__ void score_combine(const int32_t *__restrict__ lens, ScoreMask mask, int w, int L_cap, int R,
                              int n_chunks, int per_chunk, const float *__restrict__ part_m,
                              const float *__restrict__ part_z, float *__restrict__ rowb, long units)
{
    long i = (long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= units * R) return;
    long u = i / R;
    int r = (int)(i % R);
    int L = lens[u];
    if (L < w || L > L_cap || mask.skip(u, L, w, L_cap)) return;
    int used = ((L + kScoreChunk - 1) / kScoreChunk) * per_chunk;
    float m = -INFINITY, z = 0.f;
    for (int c = 0; c < used; ++c) {
        size_t o = ((size_t)u * n_chunks * per_chunk + c) * R + r;
        lse_merge(m, z, part_m[o], part_z[o]);
    }
    rowb[i] = m + log2f(z);
}

// The units a masked call scores, in ascending order (one CTA; a ballot scan per
// blockDim.x units), and their count.
__device__ __forceinline__ void unit_list_block(const int32_t *__restrict__ lens, ScoreMask mask, int w, int L_cap,
                                                int units, int32_t *__restrict__ ulist, int32_t *__restrict__ ucount)
{
    __shared__ int warp_n[32];
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5, nw = blockDim.x >> 5;
    int base = 0;
    for (int u0 = 0; u0 < units; u0 += blockDim.x) {
        const int u = u0 + threadIdx.x;
        const bool take = u < units && !mask.skip(u, lens[u], w, L_cap);
        const unsigned bal = __ballot_sync(0xffffffffu, take);
        if (lane == 0) warp_n[wid] = __popc(bal);
        __syncthreads();
        int off = base, tot = 0;
        for (int k = 0; k < nw; ++k) {
            off += k < wid ? warp_n[k] : 0;
            tot += warp_n[k];
        }
        if (take) ulist[off + __popc(bal & ((1u << lane) - 1u))] = u;
        base += tot;
        __syncthreads();
    }
    if (threadIdx.x == 0) *ucount = base;
}

__global__ void __launch_bounds__(1024) score_unit_list(const int32_t *__restrict__ lens, ScoreMask mask, int w,
                                                        int L_cap, int units, int32_t *__restrict__ ulist,
                                                        int32_t *__restrict__ ucount)
{
    wait_prior_grid();
    unit_list_block(lens, mask, w, L_cap, units, ulist, ucount);
}

// Row normalisers from log-sum-exps the decode already produced (Eq. 2 with one pass over
// K).  Window row (g, t) is query head g of the token at position L - w + t; when that
// token was decoded the cache held exactly the keys j <= L - w + t that Eq. 2's causal
// mask gives the row, so the decode's natural-log normaliser lse of that query head is
// the row's: b_r = lse * log2(e).  row_lse is [w][rows_q] (rows_q = layers * B * H_q,
// query heads in q order).  A non-finite normaliser raises ERR_NORM and leaves the row's
// normaliser at +inf, so the row adds nothing to the scores.  The tensor-core pass 2
// computes the same b_r itself where it loads a row's normaliser; this kernel serves
// the SIMT pass.
__global__ void score_rowb_from_lse(const int32_t *__restrict__ lens, ScoreMask mask, int w, int L_cap, int R, int G,
                                    int Hq, int Hkv, long rows_q, const float *__restrict__ row_lse,
                                    float *__restrict__ rowb, long units, unsigned *err)
{
    wait_prior_grid();  // lens and the ring rows may come from the previous kernels
    const long i = (long)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= units * R) return;
    const long u = i / R;
    const int r = (int)(i % R);
    const int L = lens[u];
    if (L < w || L > L_cap || mask.skip(u, L, w, L_cap)) return;
    const int g = r / w, t = r % w;
    const long qi = (u / Hkv) * Hq + (u % Hkv) * G + g;
    const float lse = row_lse[(long)t * rows_q + qi];
    if (!isfinite(lse)) {
        raise_error(err, ERR_NORM);
        rowb[i] = INFINITY;
        return;
    }
    rowb[i] = lse * kLog2e;
}

// lse ring of 2 * slots rows: rows *slot and *slot + slots both get lse[0:n] (the second
// half mirrors the first, so the rows of any `slots` consecutive pushes are contiguous),
// then *slot = (*slot + 1) % slots.  One block: every thread reads the slot before thread
// 0 advances it.
__global__ void __launch_bounds__(1024) lse_push_kernel(const float *__restrict__ lse, long n, float *__restrict__ ring,
                                                        int slots, long long *slot, unsigned *err)
{
    wait_prior_grid();  // lse (and the slot) may come from the previous kernels
    __shared__ long long s0;
    if (threadIdx.x == 0) s0 = *slot;
    __syncthreads();
    const long long s = s0;
    if (s < 0 || s >= slots) {
        if (threadIdx.x == 0) raise_error(err, ERR_INTERNAL);
        return;
    }
    float *dst = ring + s * n, *mir = ring + (s + slots) * n;
    // four independent loads in flight per thread before their stores
    constexpr int U = 4;
    if (n % 4 == 0 &&
        ((reinterpret_cast<uintptr_t>(lse) | reinterpret_cast<uintptr_t>(dst) | reinterpret_cast<uintptr_t>(mir)) & 15u) == 0) {
        const float4 *src4 = reinterpret_cast<const float4 *>(lse);
        float4 *dst4 = reinterpret_cast<float4 *>(dst), *mir4 = reinterpret_cast<float4 *>(mir);
        const long n4 = n / 4;
        for (long i0 = threadIdx.x; i0 < n4; i0 += (long)U * blockDim.x) {
            float4 v[U];
#pragma unroll
            for (int k = 0; k < U; ++k) {
                const long i = i0 + (long)k * blockDim.x;
                if (i < n4) v[k] = src4[i];
            }
#pragma unroll
            for (int k = 0; k < U; ++k) {
                const long i = i0 + (long)k * blockDim.x;
                if (i < n4) {
                    dst4[i] = v[k];
                    mir4[i] = v[k];
                }
            }
        }
    } else {
        for (long i0 = threadIdx.x; i0 < n; i0 += (long)U * blockDim.x) {
            float v[U];
#pragma unroll
            for (int k = 0; k < U; ++k) {
                const long i = i0 + (long)k * blockDim.x;
                if (i < n) v[k] = lse[i];
            }
#pragma unroll
            for (int k = 0; k < U; ++k) {
                const long i = i0 + (long)k * blockDim.x;
                if (i < n) {
                    dst[i] = v[k];
                    mir[i] = v[k];
                }
            }
        }
    }
    if (threadIdx.x == 0) *slot = (s + 1) % slots;
}

// Pass 2: one thread per candidate key, its key row held in registers; the window
// queries sit in shared memory and are read by broadcast.
template <typename T, int D>
__global__ void __launch_bounds__(128) score_colsum_simt(
    const T *__restrict__ q_win, const T *__restrict__ K, const int32_t *__restrict__ lens, ScoreMask mask,
    int w, int G, int Hq, int Hkv, int L_cap, int R, float c2, const float *__restrict__ rowb,
    float *__restrict__ raw)
{
    extern __shared__ __align__(16) float smem[];
    float *Qs = smem;         // [R][D]
    float *Bs = smem + R * D; // [R]
    const int chunk = blockIdx.x;
    const long u = blockIdx.y;
    const int L = lens[u];
    if (L < w || L > L_cap || mask.skip(u, L, w, L_cap)) return;
    const int nc = L - w;
    const int j0 = chunk * kScoreChunk;
    const int j1 = min(j0 + kScoreChunk, nc);
    if (j0 >= j1) return;
    const long lb = u / Hkv;
    const int h = (int)(u % Hkv);
    for (int e = threadIdx.x; e < R * D; e += blockDim.x) {
        int rr = e / D, c = e % D;
        int g = rr / w, t = rr % w;
        Qs[e] = to_float(q_win[(((lb * Hq) + (long)h * G + g) * w + t) * D + c]);
    }
    for (int rr = threadIdx.x; rr < R; rr += blockDim.x) Bs[rr] = rowb[u * R + rr];
    __syncthreads();
    const T *Kp = K + u * (long)L_cap * D;
    const float invG = 1.f / (float)G;
    for (int j = j0 + threadIdx.x; j < j1; j += blockDim.x) {
        float k[D];
#pragma unroll
        for (int c = 0; c < D; ++c) k[c] = to_float(Kp[(long)j * D + c]);
        float acc = 0.f;
        for (int rr = 0; rr < R; ++rr) {
            const float *qr = Qs + rr * D;
            float s = 0.f;
#pragma unroll
            for (int c = 0; c < D; c += 4) {
                float4 qv = *reinterpret_cast<const float4 *>(qr + c);
                s = fmaf(qv.x, k[c], s);
                s = fmaf(qv.y, k[c + 1], s);
                s = fmaf(qv.z, k[c + 2], s);
                s = fmaf(qv.w, k[c + 3], s);
            }
            acc += fast_exp2(fmaf(s, c2, -Bs[rr]));
        }
        raw[u * L_cap + j] = acc * invG;
    }
}

// Max-pool over the clipped window [j - pool/2, j + pool/2] within [0, L-w).
// score_pool over the units of a masked call's list only: CTAs (blockIdx.x: a 256-key
// chunk) walk the list, so the units left out cost no CTAs.
__global__ void score_pool_list(const float *__restrict__ raw, const int32_t *__restrict__ lens,
                                const int32_t *__restrict__ ulist, const int32_t *__restrict__ ucount, int w,
                                int L_cap, int pool, float *__restrict__ scores)
{
    wait_prior_grid();  // the raw scores and the list come from the previous kernels
    const int n = *ucount;
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    const int half = pool / 2;
    for (int k = blockIdx.y; k < n; k += gridDim.y) {
        const long u = ulist[k];
        const int L = lens[u];
        if (L < w || L > L_cap) continue;
        const int nc = L - w;
        if (j >= nc) continue;
        const int lo = max(0, j - half), hi = min(nc - 1, j + half);
        const float *rp = raw + u * L_cap;
        float m = rp[lo];
        for (int i = lo + 1; i <= hi; ++i) m = fmaxf(m, rp[i]);
        scores[u * L_cap + j] = m;
    }
}

__global__ void score_pool(const float *__restrict__ raw, const int32_t *__restrict__ lens, ScoreMask mask, int w,
                           int L_cap, int pool, float *__restrict__ scores)
{
    wait_prior_grid();  // the raw scores come from the previous kernel
    const int j = blockIdx.x * blockDim.x + threadIdx.x;
    const long u = blockIdx.y;
    const int L = lens[u];
    if (L < w || L > L_cap || mask.skip(u, L, w, L_cap)) return;
    const int nc = L - w;
    if (j >= nc) return;
    const int half = pool / 2;
    const int lo = max(0, j - half), hi = min(nc - 1, j + half);
    const float *rp = raw + u * L_cap;
    float m = rp[lo];
    for (int i = lo + 1; i <= hi; ++i) m = fmaxf(m, rp[i]);
    scores[u * L_cap + j] = m;
}


cudaError_t launch_score_tc_pass1(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                                  float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool *used);
// row_lse (or nullptr: ws.rowb) gives pass 2 its row normalisers: the decode's lse, read
// where each row's normaliser is loaded.
cudaError_t launch_score_tc_pass2(const reco_kv &kv, const void *q_win, const int32_t *lens, bool masked, int w,
                                  float c2, const ScoreWs &ws, const float *row_lse, unsigned *err, cudaStream_t s,
                                  bool *used);
bool score_tc_supported(const reco_kv &kv, int w);
int score_tc_pass1_groups(int R);

// SIMT passes; with pass1 false the row normalisers are already in ws.rowb.
template <typename T, int D>
static cudaError_t score_simt(const reco_kv &kv, const T *q_win, const int32_t *lens, ScoreMask mask, int w,
                              float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool pass1 = true)
{
    const long units = (long)kv.n_layers * kv.B * kv.H_kv;
    const int G = kv.H_q / kv.H_kv, R = G * w;
    const int nch = (kv.L_cap + kScoreChunk - 1) / kScoreChunk;
    const T *K = (const T *)kv.k;
    cudaError_t e = cudaSuccess;
    if (pass1) {
        int bx = R < 256 ? ((R + 31) / 32) * 32 : 256;
        dim3 g1(nch, (unsigned)units, (R + bx - 1) / bx);
        score_rowstats_simt<T, D><<<g1, bx, 0, s>>>(q_win, K, lens, mask, w, G, kv.H_q, kv.H_kv, kv.L_cap, R,
                                                    nch, c2, ws.part_m, ws.part_z, err);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        long n = units * R;
        score_combine<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(lens, mask, w, kv.L_cap, R, nch, 1, ws.part_m,
                                                                  ws.part_z, ws.rowb, units);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    size_t smem = ((size_t)R * D + R) * sizeof(float);
    e = cudaFuncSetAttribute(score_colsum_simt<T, D>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                             (int)smem);
    if (e != cudaSuccess) return e;
    score_colsum_simt<T, D><<<dim3(nch, (unsigned)units), 128, smem, s>>>(
        q_win, K, lens, mask, w, G, kv.H_q, kv.H_kv, kv.L_cap, R, c2, ws.rowb, ws.raw);
    return cudaGetLastError();
}

// Largest R*D the SIMT pass 2 keeps in shared memory.
constexpr size_t kSimtMaxQ = 200 * 1024 / 4;

bool score_shape_supported(const reco_kv &kv, int w)
{
    size_t R = (size_t)(kv.H_q / kv.H_kv) * w;
    if (score_tc_supported(kv, w)) return true;
    return (kv.d == 64 || kv.d == 128) && (R * kv.d + R) <= kSimtMaxQ;
}

static cudaError_t score_simt_any(const reco_kv &kv, const void *q_win, const int32_t *lens, ScoreMask mask, int w,
                                  float c2, const ScoreWs &ws, unsigned *err, cudaStream_t s, bool pass1)
{
    if (kv.dtype == RECO_F32)
        return kv.d == 64 ? score_simt<float, 64>(kv, (const float *)q_win, lens, mask, w, c2, ws, err, s, pass1)
                          : score_simt<float, 128>(kv, (const float *)q_win, lens, mask, w, c2, ws, err, s, pass1);
    return kv.d == 64
               ? score_simt<__nv_bfloat16, 64>(kv, (const __nv_bfloat16 *)q_win, lens, mask, w, c2, ws, err, s, pass1)
               : score_simt<__nv_bfloat16, 128>(kv, (const __nv_bfloat16 *)q_win, lens, mask, w, c2, ws, err, s,
                                                pass1);
}

// Max-pooling of the raw scores into `scores`: over the unit list when the call built one
// (a masked tensor-core call), else one CTA per (unit, 256-key chunk).
static cudaError_t launch_pool(const reco_kv &kv, const int32_t *lens, ScoreMask mask, bool listed, int w, int pool,
                               float *scores, const ScoreWs &ws, cudaStream_t s)
{
    const long units = (long)kv.n_layers * kv.B * kv.H_kv;
    const unsigned chunks = (unsigned)((kv.L_cap + 255) / 256);
    if (listed) {
        const long walkers = std::max(1L, 8L * device_sm_count() / (long)chunks);
        const unsigned ys = (unsigned)std::min(units, std::min(walkers, 65535L));
        cudaError_t e = launch_pdl(score_pool_list, dim3(chunks, ys), dim3(256), 0, s, (const float *)ws.raw, lens,
                                   (const int32_t *)ws.ulist, (const int32_t *)ws.ucount, w, kv.L_cap, pool, scores);
        if (e != cudaSuccess) return e;
    } else {
        cudaError_t e = launch_pdl(score_pool, dim3(chunks, (unsigned)units), dim3(256), 0, s, (const float *)ws.raw, lens,
                                   mask, w, kv.L_cap, pool, scores);
        if (e != cudaSuccess) return e;
    }
    return cudaGetLastError();
}

cudaError_t launch_score(const reco_kv &kv, const void *q_win, const int32_t *lens, const int32_t *keep, int w,
                         int pool, float scale, float *scores, const ScoreWs &ws, unsigned *err, cudaStream_t s)
{
    const float c2 = scale * kLog2e;
    const long units = (long)kv.n_layers * kv.B * kv.H_kv;
    const ScoreMask mask{keep, kv.B, kv.H_kv};
    cudaError_t e = cudaSuccess;
    bool used_tc = false;
    const bool tc = kv.dtype == RECO_BF16 && score_tc_supported(kv, w);
    if (tc) {
        // tensor-core passes: (unit list) -> pass 1 -> combine -> pass 2
        if (keep) {
            e = launch_pdl(score_unit_list, dim3(1), dim3(1024), 0, s, lens, mask, w, kv.L_cap, (int)units, ws.ulist,
                           ws.ucount);
            if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
        }
        e = launch_score_tc_pass1(kv, q_win, lens, keep != nullptr, w, c2, ws, err, s, &used_tc);
        if (e != cudaSuccess) return e;
        if (used_tc) {
            const int R = (kv.H_q / kv.H_kv) * w;
            const int nch = (kv.L_cap + kScoreChunk - 1) / kScoreChunk;
            score_combine<<<(unsigned)((units * R + 255) / 256), 256, 0, s>>>(
                lens, mask, w, kv.L_cap, R, nch, score_tc_pass1_groups(R), ws.part_m, ws.part_z, ws.rowb, units);
            if ((e = cudaGetLastError()) != cudaSuccess) return e;
            bool used2 = false;
            e = launch_score_tc_pass2(kv, q_win, lens, keep != nullptr, w, c2, ws, nullptr, err, s, &used2);
            if (e != cudaSuccess) return e;
            if (!used2) return cudaErrorNotSupported;
        }
    }
    if (!used_tc) {
        e = score_simt_any(kv, q_win, lens, mask, w, c2, ws, err, s, true);
        if (e != cudaSuccess) return e;
    }
    return launch_pool(kv, lens, mask, tc && keep, w, pool, scores, ws, s);
}

cudaError_t launch_lse_push(const float *lse, long n, float *ring, int slots, long long *slot, unsigned *err,
                            cudaStream_t s)
{
    cudaError_t e = launch_pdl(lse_push_kernel, dim3(1), dim3(1024), 0, s, lse, n, ring, slots, slot, err);
    return e != cudaSuccess ? e : cudaGetLastError();
}

// Row *index of a [rows][n16] array of 16-byte chunks into dst, for captured step loops
// whose input row is chosen on the device: a grid of a few CTAs per SM, eight independent
// 16-byte loads per thread in flight before its stores.
__global__ void __launch_bounds__(256) copy_row_kernel(const uint4 *__restrict__ src, long long rows, long long n16,
                                                     const long long *__restrict__ index, uint4 *__restrict__ dst,
                                                     unsigned *err)
{
    wait_prior_grid();  // the index (and the destination's readers) belong to earlier kernels
    const long long r = *index;
    if (r < 0 || r >= rows) {
        if (blockIdx.x == 0 && threadIdx.x == 0) raise_error(err, ERR_INTERNAL);
        return;
    }
    const uint4 *row = src + r * n16;
    const long long stride = (long long)gridDim.x * blockDim.x;
    for (long long i0 = (long long)blockIdx.x * blockDim.x + threadIdx.x; i0 < n16; i0 += 8 * stride) {
        uint4 v[8];
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const long long i = i0 + k * stride;
            if (i < n16) v[k] = ld_stream_u4(row + i);
        }
#pragma unroll
        for (int k = 0; k < 8; ++k) {
            const long long i = i0 + k * stride;
            if (i < n16) dst[i] = v[k];
        }
    }
}

cudaError_t launch_copy_row(const void *src, long long rows, long long row_bytes, const long long *index, void *dst,
                            unsigned *err, cudaStream_t s)
{
    const long long n16 = row_bytes / 16;
    const long long want = (n16 + 256LL * 8 - 1) / (256LL * 8);
    const unsigned grid = (unsigned)std::max(1LL, std::min(want, 4LL * device_sm_count()));
    cudaError_t e = launch_pdl(copy_row_kernel, dim3(grid), dim3(256), 0, s, reinterpret_cast<const uint4 *>(src), rows,
                               n16, index, reinterpret_cast<uint4 *>(dst), err);
    return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_score_lse(const reco_kv &kv, const void *q_win, const int32_t *lens, const int32_t *keep,
                             const float *row_lse, int w, int pool, float scale, float *scores, const ScoreWs &ws,
                             unsigned *err, cudaStream_t s)
{
    const float c2 = scale * kLog2e;
    const long units = (long)kv.n_layers * kv.B * kv.H_kv;
    const ScoreMask mask{keep, kv.B, kv.H_kv};
    const int G = kv.H_q / kv.H_kv, R = G * w;
    const long rows_q = (long)kv.n_layers * kv.B * kv.H_q;
    const bool tc = kv.dtype == RECO_BF16 && score_tc_supported(kv, w);
    cudaError_t e;
    bool used = false;
    if (tc) {  // the tensor-core pass reads each row's normaliser from row_lse itself
        if (keep) {
            e = launch_pdl(score_unit_list, dim3(1), dim3(1024), 0, s, lens, mask, w, kv.L_cap, (int)units, ws.ulist,
                           ws.ucount);
            if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
        }
        e = launch_score_tc_pass2(kv, q_win, lens, keep != nullptr, w, c2, ws, row_lse, err, s, &used);
        if (e != cudaSuccess) return e;
    }
    if (!used) {  // the SIMT pass takes them from ws.rowb
        e = launch_pdl(score_rowb_from_lse, dim3((unsigned)((units * R + 255) / 256)), dim3(256), 0, s, lens, mask, w,
                       kv.L_cap, R, G, kv.H_q, kv.H_kv, rows_q, row_lse, ws.rowb, units, err);
        if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
        e = score_simt_any(kv, q_win, lens, mask, w, c2, ws, err, s, false);
        if (e != cudaSuccess) return e;
    }
    return launch_pool(kv, lens, mask, tc && keep, w, pool, scores, ws, s);
}

}  // namespace reco
