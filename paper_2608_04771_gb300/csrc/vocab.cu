// vocab.cu -- the two vocabulary-side steps of ReCo's generation control (Sec. 3.3).
//
// reflect_penalty: Eq. 3 picks beta_i in {0, beta/2, beta} from the band of the
// step reward (float32 compares); Eq. 4 subtracts it from the logit of every
// reflection token, in place.  R is a set: an id listed twice is penalised once.
//
// sample_cluster (or sample_segments + sample_pick for unaligned or very long rows):
// Eq. 3-4 and then one draw per row from softmax of the penalised logits (Sec. 3.3,
// temperature 1) by inversion at a caller-supplied uniform.
//
// ppl_rows + ppl_finish: Eq. 5 log p(x_t) = z[x_t] - logsumexp(z) per answer row
// (one CTA per row, one streaming pass with an online max/sum), then per sequence
// PPL = exp(-mean log p) and the Eq. 6 stop flag PPL <= tau_p.
#include "common.cuh"
#include "internal.h"
#include "tma.cuh"

namespace reco {

// The ids of R in shared memory (one coalesced read per CTA), so the duplicate check of
// each id against the ones before it runs on shared memory; longer lists are read
// from global memory.
constexpr int kIdsShared = 1024;

__device__ __forceinline__ bool stage_ids(const int32_t *__restrict__ ids, int n_ids, int *sm_ids)
{
    const bool staged = n_ids <= kIdsShared;  // uniform across the CTA
    if (staged) {
        for (int i = threadIdx.x; i < n_ids; i += blockDim.x) sm_ids[i] = ids[i];
        __syncthreads();
    }
    return staged;
}

__device__ __forceinline__ bool seen_before(const int32_t *__restrict__ ids, const int *sm_ids, bool staged, int i,
                                            int id)
{
    bool dup = false;
    if (staged) {
        for (int k = 0; k < i; ++k) dup |= sm_ids[k] == id;
    } else {
        for (int k = 0; k < i && !dup; ++k) dup = ids[k] == id;
    }
    return dup;
}

__global__ void reflect_penalty_kernel(float *logits, int V, const int32_t *__restrict__ ids, int n_ids,
                                       const float *__restrict__ rewards, float tau_l, float tau_h,
                                       float beta, float *beta_out, unsigned *err)
{
    __shared__ int sm_ids[kIdsShared];
    wait_prior_grid();
    const int b = blockIdx.x;
    const float v = rewards[b];
    const float bi = (v <= tau_l) ? 0.f : ((v >= tau_h) ? beta : beta * 0.5f);
    if (threadIdx.x == 0 && beta_out) beta_out[b] = bi;
    const bool staged = stage_ids(ids, n_ids, sm_ids);
    for (int i = threadIdx.x; i < n_ids; i += blockDim.x) {
        const int id = staged ? sm_ids[i] : ids[i];
        if (id < 0 || id >= V) {
            if (b == 0) raise_error(err, ERR_ID);
            continue;
        }
        if (bi == 0.f || seen_before(ids, sm_ids, staged, i, id)) continue;
        float *p = logits + (size_t)b * V + id;
        *p = __fsub_rn(*p, bi);
    }
}

cudaError_t launch_penalty(float *logits, int B, int V, const int32_t *ids, int n_ids,
                           const float *rewards, float tau_l, float tau_h, float beta, float *beta_out,
                           unsigned *err, cudaStream_t s)
{
    int nt = n_ids < 32 ? 32 : (n_ids > 256 ? 256 : ((n_ids + 31) / 32) * 32);
    return launch_pdl(reflect_penalty_kernel, dim3(B), dim3(nt), 0, s, logits, V, ids, n_ids, rewards, tau_l, tau_h,
                      beta, beta_out, err);
}

// ---------------------------------------------------------------- penalty + sampling
// Pass 1, one CTA per (row, segment of kSampleSeg logits): the penalty of Eq. 4 on the
// ids inside the segment (once per distinct id, one correctly rounded float32
// subtract), then one streaming read of the segment for its log2-domain (max, sum).
// Tokens at -inf carry no mass.
template <int NT>
__global__ void __launch_bounds__(NT) sample_segments(float *__restrict__ logits, int V, int nseg,
                                                      const int32_t *__restrict__ ids, int n_ids,
                                                      const float *__restrict__ rewards, float tau_l, float tau_h,
                                                      float beta, float *__restrict__ beta_out,
                                                      float2 *__restrict__ part, unsigned *err)
{
    constexpr int PER = kSampleSeg / NT;
    __shared__ float sm_m[NT / 32], sm_s[NT / 32];
    __shared__ int sm_ids[kIdsShared];
    wait_prior_grid();
    const int sg = blockIdx.x, b = blockIdx.y;
    const int lo = sg * kSampleSeg, hi = min(V, lo + kSampleSeg);
    float *z = logits + (size_t)b * V;
    const float v = rewards[b];
    const float bi = (v <= tau_l) ? 0.f : ((v >= tau_h) ? beta : beta * 0.5f);
    if (sg == 0 && threadIdx.x == 0 && beta_out) beta_out[b] = bi;
    const bool staged = stage_ids(ids, n_ids, sm_ids);
    for (int i = threadIdx.x; i < n_ids; i += NT) {
        const int id = staged ? sm_ids[i] : ids[i];
        if (id < 0 || id >= V) {
            if (b == 0 && sg == 0) raise_error(err, ERR_ID);
            continue;
        }
        if (id < lo || id >= hi || bi == 0.f) continue;
        if (!seen_before(ids, sm_ids, staged, i, id)) z[id] = __fsub_rn(z[id], bi);
    }
    __syncthreads();  // the segment's penalised logits are visible to the whole CTA
    float y[PER];
    float m = -INFINITY;
#pragma unroll
    for (int k = 0; k < PER; ++k) {  // all loads in flight first
        const int j = lo + k * NT + (int)threadIdx.x;
        y[k] = j < hi ? z[j] * kLog2e : -INFINITY;
    }
#pragma unroll
    for (int k = 0; k < PER; ++k) m = fmaxf(m, y[k]);
    float s = 0.f;
    if (m != -INFINITY) {
#pragma unroll
        for (int k = 0; k < PER; ++k) s += fast_exp2(y[k] - m);  // -inf terms add 0
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
        lse_merge(m, s, m2, s2);
    }
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
        sm_m[wid] = m;
        sm_s[wid] = s;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float M = sm_m[0], S = sm_s[0];
        for (int w2 = 1; w2 < NT / 32; ++w2) lse_merge(M, S, sm_m[w2], sm_s[w2]);
        part[(size_t)b * nseg + sg] = make_float2(M, S);
    }
}

// Exclusive block scan of one float per thread (NT threads), in thread order.
template <int NT>
__device__ __forceinline__ float block_scan_excl(float x, float *sm_w)
{
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    float incl = x;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const float y = __shfl_up_sync(0xffffffffu, incl, o);
        if (lane >= o) incl += y;
    }
    if (lane == 31) sm_w[wid] = incl;
    __syncthreads();
    float base = 0.f;
    for (int w2 = 0; w2 < wid; ++w2) base += sm_w[w2];
    __syncthreads();
    return base + (incl - x);
}

// The values v[0..R) of every thread form one sequence in thread order (thread t holds
// indices first + 0 .. first + R-1).  Returns the first index whose running sum exceeds
// T among positive values, with the running sum before it; -1 if none (T at or above
// the total, or NaN).  `last` receives the last index with a positive value (-1: none).
// A thread whose run the block scan says holds the crossing takes its last positive
// value, with the running sum before that value, when its own sequential sum falls a
// rounding short of T (so the search inside a chosen segment then ends at its top).
template <int NT, int R>
__device__ __forceinline__ int find_crossing(const float (&v)[R], int first, float T, float *sm_w, int *sm_i,
                                             float *sm_f, float &before, int &last)
{
    float run = 0.f;
    int my_last = -1;
#pragma unroll
    for (int k = 0; k < R; ++k) {
        run += v[k];
        if (v[k] > 0.f) my_last = first + k;
    }
    const float excl = block_scan_excl<NT>(run, sm_w);
    if (threadIdx.x == 0) {
        sm_i[0] = -1;
        sm_i[1] = -1;
        sm_f[0] = 0.f;
    }
    __syncthreads();
    if (run > 0.f && excl <= T && excl + run > T) {  // at most one thread: the prefix only grows
        float c = excl, prev = excl;  // defaults: the crossing lost to rounding
        int pick = my_last;
        bool hit = false;
#pragma unroll
        for (int k = 0; k < R; ++k) {
            const float c0 = c;
            c += v[k];
            if (!hit && v[k] > 0.f) {
                if (c > T) {
                    hit = true;
                    pick = first + k;
                }
                prev = c0;
            }
        }
        sm_i[0] = pick;
        sm_f[0] = prev;
    }
    if (my_last >= 0) atomicMax(&sm_i[1], my_last);
    __syncthreads();
    const int idx = sm_i[0];
    before = sm_f[0];
    last = sm_i[1];
    __syncthreads();
    return idx;
}

// Pass 2, one CTA per row.  With M the largest segment max, segment k carries the mass
// W_k = S_k 2^(m_k - M) and the row Z = sum W_k; the draw u selects T = u Z.  The
// segment where the running mass first exceeds T is read again and its tokens' masses
// 2^(z log2e - M) locate the token where the running mass first exceeds what is left of
// T.  No crossing (u at the top of [0, 1) after rounding, or NaN) takes the last token
// with mass; a row without mass gets -1.
template <int NT>
__global__ void __launch_bounds__(NT) sample_pick(const float *__restrict__ logits, int V, int nseg,
                                                  const float *__restrict__ uniforms,
                                                  const float2 *__restrict__ part, int32_t *__restrict__ tokens)
{
    constexpr int PER = kSampleSeg / NT;
    constexpr int SR = kSampleMaxSeg / NT;  // segments per thread
    __shared__ float sm_w[NT / 32];
    __shared__ float sm_f[1];
    __shared__ int sm_i[2];
    wait_prior_grid();
    const int b = blockIdx.x, tid = threadIdx.x;
    const float2 *pp = part + (size_t)b * nseg;
    float2 q[SR];
    float M = -INFINITY;
#pragma unroll
    for (int k = 0; k < SR; ++k) {
        const int sg = tid * SR + k;
        q[k] = sg < nseg ? pp[sg] : make_float2(-INFINITY, 0.f);
        M = fmaxf(M, q[k].x);
    }
    M = warp_max(M);
    if ((tid & 31) == 0) sm_w[tid >> 5] = M;
    __syncthreads();
    M = sm_w[0];
    for (int w2 = 1; w2 < NT / 32; ++w2) M = fmaxf(M, sm_w[w2]);
    __syncthreads();
    if (M == -INFINITY) {  // no token has mass
        if (tid == 0) tokens[b] = -1;
        return;
    }
    float w[SR];
    float zsum = 0.f;
#pragma unroll
    for (int k = 0; k < SR; ++k) {
        w[k] = q[k].y > 0.f ? q[k].y * fast_exp2(q[k].x - M) : 0.f;
        zsum += w[k];
    }
    zsum = warp_sum(zsum);
    if ((tid & 31) == 0) sm_w[tid >> 5] = zsum;
    __syncthreads();
    float Z = 0.f;
    for (int w2 = 0; w2 < NT / 32; ++w2) Z += sm_w[w2];
    __syncthreads();
    const float u = uniforms[b];
    const float T = u != u ? u : fmaxf(u, 0.f) * Z;  // a NaN draw finds no crossing
    float before;
    int last_seg;
    int seg = find_crossing<NT, SR>(w, tid * SR, T, sm_w, sm_i, sm_f, before, last_seg);
    const bool found = seg >= 0;
    if (!found) seg = last_seg;
    const float Tr = found ? fmaxf(T - before, 0.f) : INFINITY;  // left of T inside the segment
    const float *z = logits + (size_t)b * V;
    const int first = seg * kSampleSeg + tid * PER;
    float p[PER];
#pragma unroll
    for (int k = 0; k < PER; ++k) {
        const int j = first + k;
        const float y = j < V ? z[j] * kLog2e : -INFINITY;
        p[k] = y == -INFINITY ? 0.f : fast_exp2(y - M);
    }
    float before2;
    int last_tok;
    const int tok = find_crossing<NT, PER>(p, first, Tr, sm_w, sm_i, sm_f, before2, last_tok);
    if (tid == 0) tokens[b] = tok >= 0 ? tok : last_tok;
}

// ---------------------------------------------------------------- penalty + sampling in one launch
// One cluster of C <= 8 CTAs per row, for rows of 16-byte aligned float32 logits (V a
// multiple of 4) of at most C * kSampleClusterRecs records of kSampleRec tokens.  CTA r
// of the cluster brings records [r * rpc, (r + 1) * rpc) of its row into shared memory
// with bulk copies, applies the Eq. 4 penalty to the ids inside them (in shared memory
// and in place in global memory, the same correctly rounded subtract as above), and
// writes each record's log2-domain (max, sum) into CTA 0's shared memory.  After a
// cluster barrier CTA 0 draws exactly as sample_pick does, with records in place of
// segments, reading the chosen record from its owner CTA's shared memory; a second
// cluster barrier keeps every CTA's shared memory alive until that read is done.  The
// row is read from HBM once and no workspace is used.
constexpr int kSampleRec = 1024;          // tokens per record
constexpr int kSampleClusterRecs = 48;    // records per CTA at most (192 KB of shared memory)
constexpr int kSampleCluster = 8;         // CTAs per row at most (the portable cluster size)
constexpr long long kSampleSpin = 1LL << 24;  // bounded wait on the bulk copies (about a second)

__device__ __forceinline__ uint32_t cluster_rank()
{
    uint32_t r;
    asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
    return r;
}

// Address of the same shared-memory location in CTA `rank` of the cluster.
__device__ __forceinline__ uint32_t cluster_addr(uint32_t addr, uint32_t rank)
{
    uint32_t r;
    asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(r) : "r"(addr), "r"(rank));
    return r;
}

__device__ __forceinline__ void st_cluster_f2(uint32_t addr, float x, float y)
{
    asm volatile("st.shared::cluster.v2.f32 [%0], {%1, %2};" ::"r"(addr), "f"(x), "f"(y) : "memory");
}

__device__ __forceinline__ float4 ld_cluster_f4(uint32_t addr)
{
    float4 v;
    asm volatile("ld.shared::cluster.v4.f32 {%0, %1, %2, %3}, [%4];"
                 : "=f"(v.x), "=f"(v.y), "=f"(v.z), "=f"(v.w)
                 : "r"(addr)
                 : "memory");
    return v;
}

// All threads of all CTAs of the cluster; shared-memory writes before it (local or
// remote) are visible to every CTA after it.
__device__ __forceinline__ void cluster_sync()
{
    asm volatile("barrier.cluster.arrive.release.aligned;\n\tbarrier.cluster.wait.acquire.aligned;" ::: "memory");
}

// Untiled bulk copy global -> shared (both 16-byte aligned, bytes a multiple of 16).
__device__ __forceinline__ void bulk_load(uint32_t dst, const void *src, uint32_t bytes, uint32_t bar)
{
    asm volatile("cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];"
                 ::"r"(dst), "l"(reinterpret_cast<uint64_t>(src)), "r"(bytes), "r"(bar)
                 : "memory");
}

template <int NT>
__global__ void __launch_bounds__(NT) sample_cluster(float *__restrict__ logits, int V, int rpc,
                                                     const int32_t *__restrict__ ids, int n_ids,
                                                     const float *__restrict__ rewards, float tau_l, float tau_h,
                                                     float beta, float *__restrict__ beta_out,
                                                     const float *__restrict__ uniforms,
                                                     int32_t *__restrict__ tokens, unsigned *err)
{
    constexpr int NWARP = NT / 32;
    constexpr int SR = (kSampleCluster * kSampleClusterRecs + NT - 1) / NT;  // records per thread (pick)
    constexpr int PER = kSampleRec / NT;                                     // tokens per thread (pick)
    constexpr int RL = kSampleRec / 32;                                      // tokens per lane (records)
    static_assert(PER == 4, "the pick reads one float4 of the chosen record per thread");
    extern __shared__ __align__(128) float sm_z[];  // [rpc * kSampleRec] this CTA's part of the row
    __shared__ float2 sm_rec[NT * SR];               // (max, sum) of every record of the row (CTA 0)
    __shared__ int sm_ids[kIdsShared];
    __shared__ float sm_w[NWARP];
    __shared__ float sm_f[1];
    __shared__ int sm_i[2];
    __shared__ __align__(8) uint64_t bar;
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const uint32_t r = cluster_rank();
    const int b = blockIdx.y;
    const int nrec = (V + kSampleRec - 1) / kSampleRec;
    const int lo = (int)r * rpc * kSampleRec;  // first token held here
    const int hi = min(V, lo + rpc * kSampleRec);
    const int nr = hi > lo ? (hi - lo + kSampleRec - 1) / kSampleRec : 0;  // records held here
    const uint32_t bar_a = smem_addr(&bar), z_a = smem_addr(sm_z);
    if (tid == 0) {
        mbar_init(bar_a, 1);
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        fence_async_shared();
    }
    __syncthreads();
    wait_prior_grid();
    float *z = logits + (size_t)b * V;
    if (tid == 0 && nr > 0) {  // the copies run while the ids and the reward load
        const uint32_t bytes = (uint32_t)(hi - lo) * 4u;
        mbar_expect_tx(bar_a, bytes);
        for (uint32_t off = 0; off < bytes; off += 16384u)
            bulk_load(z_a + off, z + lo + off / 4u, min(16384u, bytes - off), bar_a);
    }
    const float v = rewards[b];
    const float bi = (v <= tau_l) ? 0.f : ((v >= tau_h) ? beta : beta * 0.5f);
    if (r == 0 && tid == 0 && beta_out) beta_out[b] = bi;
    const bool staged = stage_ids(ids, n_ids, sm_ids);
    bool landed = true;
    if (nr > 0) {
        landed = mbar_wait_bounded(bar_a, 0, kSampleSpin);
        if (!landed && tid == 0) raise_error(err, ERR_INTERNAL);
    }
    for (int i = tid; i < n_ids; i += NT) {
        const int id = staged ? sm_ids[i] : ids[i];
        if (id < 0 || id >= V) {
            if (b == 0 && r == 0) raise_error(err, ERR_ID);
            continue;
        }
        if (id < lo || id >= hi || bi == 0.f || !landed) continue;
        if (!seen_before(ids, sm_ids, staged, i, id)) {
            const float pz = __fsub_rn(sm_z[id - lo], bi);
            sm_z[id - lo] = pz;
            z[id] = pz;
        }
    }
    __syncthreads();  // the penalised records are visible to the whole CTA

    // one warp per record: its log2-domain (max, sum), into CTA 0's table
    const uint32_t rec0 = cluster_addr(smem_addr(sm_rec), 0);
    for (int k = wid; k < nr; k += NWARP) {
        float y[RL];
        float m = -INFINITY;
#pragma unroll
        for (int i = 0; i < RL; ++i) {
            const int j = k * kSampleRec + i * 32 + lane;
            y[i] = lo + j < hi ? sm_z[j] * kLog2e : -INFINITY;
            m = fmaxf(m, y[i]);
        }
        float s = 0.f;
        if (m != -INFINITY) {
#pragma unroll
            for (int i = 0; i < RL; ++i) s += fast_exp2(y[i] - m);  // -inf terms add 0
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) {
            const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
            const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
            lse_merge(m, s, m2, s2);
        }
        if (lane == 0) st_cluster_f2(rec0 + (uint32_t)((int)r * rpc + k) * 8u, m, s);
    }
    cluster_sync();

    if (r == 0) {  // uniform across the CTA
        float2 q[SR];
        float M = -INFINITY;
#pragma unroll
        for (int k = 0; k < SR; ++k) {
            const int g = tid * SR + k;
            q[k] = g < nrec ? sm_rec[g] : make_float2(-INFINITY, 0.f);
            M = fmaxf(M, q[k].x);
        }
        M = warp_max(M);
        if (lane == 0) sm_w[wid] = M;
        __syncthreads();
        M = sm_w[0];
        for (int w2 = 1; w2 < NWARP; ++w2) M = fmaxf(M, sm_w[w2]);
        __syncthreads();
        if (M == -INFINITY) {  // no token has mass
            if (tid == 0) tokens[b] = -1;
        } else {
            float w[SR];
            float zsum = 0.f;
#pragma unroll
            for (int k = 0; k < SR; ++k) {
                w[k] = q[k].y > 0.f ? q[k].y * fast_exp2(q[k].x - M) : 0.f;
                zsum += w[k];
            }
            zsum = warp_sum(zsum);
            if (lane == 0) sm_w[wid] = zsum;
            __syncthreads();
            float Z = 0.f;
            for (int w2 = 0; w2 < NWARP; ++w2) Z += sm_w[w2];
            __syncthreads();
            const float u = uniforms[b];
            const float T = u != u ? u : fmaxf(u, 0.f) * Z;  // a NaN draw finds no crossing
            float before;
            int last_rec;
            int rec = find_crossing<NT, SR>(w, tid * SR, T, sm_w, sm_i, sm_f, before, last_rec);
            const bool found = rec >= 0;
            if (!found) rec = last_rec;
            const float Tr = found ? fmaxf(T - before, 0.f) : INFINITY;
            // the chosen record, from the shared memory of the CTA that holds it
            const int first = rec * kSampleRec + tid * PER;
            const float4 zz = ld_cluster_f4(
                cluster_addr(z_a + (uint32_t)((rec % rpc) * kSampleRec + tid * PER) * 4u, (uint32_t)(rec / rpc)));
            const float zv[PER] = {zz.x, zz.y, zz.z, zz.w};
            float p[PER];
#pragma unroll
            for (int k = 0; k < PER; ++k) {
                const float y = first + k < V ? zv[k] * kLog2e : -INFINITY;
                p[k] = y == -INFINITY ? 0.f : fast_exp2(y - M);
            }
            float before2;
            int last_tok;
            const int tok = find_crossing<NT, PER>(p, first, Tr, sm_w, sm_i, sm_f, before2, last_tok);
            if (tid == 0) tokens[b] = tok >= 0 ? tok : last_tok;
        }
    }
    cluster_sync();  // CTA 0 has read the chosen record
}

cudaError_t launch_penalty_sample(float *logits, int B, int V, const int32_t *ids, int n_ids, const float *rewards,
                                  float tau_l, float tau_h, float beta, const float *uniforms, int32_t *tokens,
                                  float *beta_out, float2 *part, unsigned *err, cudaStream_t s)
{
    const int nrec = (V + kSampleRec - 1) / kSampleRec;
    const int C = nrec < kSampleCluster ? nrec : kSampleCluster;
    const int rpc = (nrec + C - 1) / C;
    if ((V & 3) == 0 && ((uintptr_t)logits & 15u) == 0 && rpc <= kSampleClusterRecs) {
        const size_t smem = (size_t)rpc * kSampleRec * sizeof(float);
        cudaError_t e = cudaFuncSetAttribute(sample_cluster<256>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                             kSampleClusterRecs * kSampleRec * (int)sizeof(float));
        if (e != cudaSuccess) return e;
        cudaLaunchConfig_t cfg = {};
        cfg.gridDim = dim3(C, B);
        cfg.blockDim = dim3(256);
        cfg.dynamicSmemBytes = smem;
        cfg.stream = s;
        cudaLaunchAttribute attr[2];
        attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[0].val.programmaticStreamSerializationAllowed = 1;
        attr[1].id = cudaLaunchAttributeClusterDimension;
        attr[1].val.clusterDim.x = C;
        attr[1].val.clusterDim.y = 1;
        attr[1].val.clusterDim.z = 1;
        cfg.attrs = attr;
        cfg.numAttrs = 2;
        return cudaLaunchKernelEx(&cfg, sample_cluster<256>, logits, V, rpc, ids, n_ids, rewards, tau_l, tau_h, beta,
                                  beta_out, uniforms, tokens, err);
    }
    // other rows: two launches through the workspace
    const int nseg = (V + kSampleSeg - 1) / kSampleSeg;
    cudaError_t e = launch_pdl(sample_segments<256>, dim3(nseg, B), dim3(256), 0, s, logits, V, nseg, ids, n_ids,
                               rewards, tau_l, tau_h, beta, beta_out, part, err);
    if (e != cudaSuccess) return e;
    return launch_pdl(sample_pick<256>, dim3(B), dim3(256), 0, s, (const float *)logits, V, nseg, uniforms,
                      (const float2 *)part, tokens);
}

// One row's Eq. 5 term per CTA: one streaming pass over the row's logits for their
// log2-domain (max, sum), then lp = z[x] - logsumexp(z).  (Four CTAs per row in a cluster,
// merged through CTA 0's shared memory, measured slower: 38.9 against 31.1 us at 8 x 32 rows
// of 152064 logits.)
template <int NT>
__global__ void __launch_bounds__(NT) ppl_rows(const float *__restrict__ logits,
                                               const int32_t *__restrict__ tokens,
                                               const int32_t *__restrict__ n_valid, int n, int V,
                                               float *__restrict__ lp, unsigned *err)
{
    __shared__ float sm_m[NT / 32], sm_s[NT / 32];
    wait_prior_grid();  // the logits may come from the previous kernel
    const int t = blockIdx.x, b = blockIdx.y;
    const int nb = n_valid ? min(n_valid[b], n) : n;
    if (t >= nb) return;
    const float *z = logits + ((size_t)b * n + t) * V;
    float m = -INFINITY, s = 0.f;
    // Vector loads only when every row starts on a 16-byte boundary: the base is
    // 16-byte aligned and rows are a multiple of 4 floats long.
    if ((V & 3) == 0 && ((uintptr_t)logits & 15u) == 0) {
        // eight 16-byte loads per thread in flight, then one max and 32 exponentials
        const float4 *z4 = reinterpret_cast<const float4 *>(z);
        const int n4 = V / 4;
        constexpr float NINF = -INFINITY;
        for (int i0 = threadIdx.x; i0 < n4; i0 += 8 * NT) {
            float4 x[8];
#pragma unroll
            for (int k = 0; k < 8; ++k) {
                const int i = i0 + k * NT;
                x[k] = i < n4 ? __ldcs(z4 + i) : make_float4(NINF, NINF, NINF, NINF);
            }
            float mx = NINF;
#pragma unroll
            for (int k = 0; k < 8; ++k) mx = fmaxf(mx, fmaxf(fmaxf(x[k].x, x[k].y), fmaxf(x[k].z, x[k].w)));
            mx *= kLog2e;
            if (mx > m) {
                s *= fast_exp2(m - mx);  // m = -inf: s is 0 and stays 0
                m = mx;
            }
            if (m != NINF) {
#pragma unroll
                for (int k = 0; k < 8; ++k)
                    s += (fast_exp2(fmaf(x[k].x, kLog2e, -m)) + fast_exp2(fmaf(x[k].y, kLog2e, -m))) +
                         (fast_exp2(fmaf(x[k].z, kLog2e, -m)) + fast_exp2(fmaf(x[k].w, kLog2e, -m)));
            }
        }
    } else {
        for (int i = threadIdx.x; i < V; i += NT) {
            const float y = z[i] * kLog2e;
            if (y > m) {
                s *= fast_exp2(m - y);
                m = y;
            }
            s += fast_exp2(y - m);
        }
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const float m2 = __shfl_xor_sync(0xffffffffu, m, o);
        const float s2 = __shfl_xor_sync(0xffffffffu, s, o);
        lse_merge(m, s, m2, s2);
    }
    const int lane = threadIdx.x & 31, wid = threadIdx.x >> 5;
    if (lane == 0) {
        sm_m[wid] = m;
        sm_s[wid] = s;
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        float M = sm_m[0], S = sm_s[0];
        for (int w2 = 1; w2 < NT / 32; ++w2) lse_merge(M, S, sm_m[w2], sm_s[w2]);
        const int x = tokens[(size_t)b * n + t];
        float res;
        if (x < 0 || x >= V) {
            raise_error(err, ERR_TOKEN);
            res = __int_as_float(0x7fc00000);
        } else {
            res = z[x] - (M + log2f(S)) * kLn2;
        }
        lp[(size_t)b * n + t] = res;
    }
}

__global__ void ppl_finish(const float *__restrict__ lp, const int32_t *__restrict__ n_valid, int B, int n,
                           float tau_p, float *__restrict__ ppl, uint8_t *__restrict__ stop)
{
    wait_prior_grid();  // the row terms come from ppl_rows
    const int b = blockIdx.x * blockDim.x + threadIdx.x;
    if (b >= B) return;
    const int nb = n_valid ? min(n_valid[b], n) : n;
    if (nb <= 0) {
        ppl[b] = __int_as_float(0x7fc00000);
        stop[b] = 0;
        return;
    }
    float sum = 0.f;
    for (int t = 0; t < nb; ++t) sum += lp[(size_t)b * n + t];
    const float p = expf(-sum / (float)nb);
    ppl[b] = p;
    stop[b] = p <= tau_p ? 1 : 0;
}

cudaError_t launch_ppl(const float *logits, const int32_t *tokens, const int32_t *n_valid, int B, int n,
                       int V, float tau_p, float *ppl, uint8_t *stop, float *lp_ws, unsigned *err,
                       cudaStream_t s)
{
    cudaError_t e;
    if (n > 0) {
        e = launch_pdl(ppl_rows<512>, dim3(n, B), dim3(512), 0, s, logits, tokens, n_valid, n, V, lp_ws, err);
        if (e != cudaSuccess || (e = cudaGetLastError()) != cudaSuccess) return e;
    }
    e = launch_pdl(ppl_finish, dim3((B + 127) / 128), dim3(128), 0, s, lp_ws, n_valid, B, n, tau_p, ppl, stop);
    return e != cudaSuccess ? e : cudaGetLastError();
}

}  // namespace reco
