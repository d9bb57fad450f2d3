// decode.cu -- decode attention over the ragged compacted cache, the per-token
// attention whose cost the compression lowers (Sec. 1; Sec. 2.2; Sec. 4.2).
//
// bf16 path (decode_mma): a persistent split-K flash-decode.  Every CTA first builds
// the same work plan from lens: a key-chunk length C chosen so the total number of
// (unit, chunk) items is a few per warp, and the prefix sum of chunks per unit.  Each
// warp then takes items from an atomic counter.  An item's keys stream from HBM in
// 16-key blocks through a private 3-stage shared-memory ring filled with cp.async
// (zero-fill past the end); each thread copies exactly the 16-byte pieces it later
// reads, so no barrier is needed and the piece-major layout has no bank conflicts.
// QK^T and PV run on mma.sync m16n8k16 (bf16 in, fp32 accumulate) with the G <= 8
// query heads of the KV head packed into one MMA tile.  The head dimension is
// permuted consistently on the Q and K sides (and on the V and output sides) so
// that each thread's fragments are contiguous 16-byte pieces of a row.  A unit split over several items writes partial
// (max, sum, output) triples; the last item to finish (atomic ticket, no waiting)
// merges them.  The appended token (k_new, v_new) is read from the inputs and written
// into the cache by the warp that covers its index; the last warp of the grid to
// finish advances lens.
//
// float32 path (decode_simt): one CTA per unit, four warps over the keys, G <= 16.
#include "common.cuh"
#include "internal.h"

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
    ws.max_items = kDecodeMaxTarget + (int)units;
    ws.counters = (int32_t *)take((2 + units) * 4);
    ws.part_ml = (float *)take((size_t)ws.max_items * G * 2 * 4);
    ws.part_o = (float *)take((size_t)ws.max_items * G * kv.d * 4);
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
    int units, Hq, Hkv, G, L_cap, max_items, append, out_bf16;
    float c2;  // scale * log2(e)
    unsigned *err;
};

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
        if (dd == 0 && a.lse) a.lse[row] = Ls > 0.f ? (M + log2f(Ls)) * kLn2 : -INFINITY;
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

// cp.async of one 16-byte piece into shared memory; src_bytes 0 writes zeros.
__device__ __forceinline__ void cp_async16(uint32_t dst, const void *src, int src_bytes)
{
    asm volatile("cp.async.cg.shared.global [%0], [%1], 16, %2;" ::"r"(dst), "l"(src), "r"(src_bytes));
}
__device__ __forceinline__ void cp_async_commit() { asm volatile("cp.async.commit_group;"); }
template <int N> __device__ __forceinline__ void cp_async_wait() { asm volatile("cp.async.wait_group %0;" ::"n"(N)); }

// Issue the 16-byte pieces one thread needs for the 16-key block at kb into its slots
// of a ring stage.  Piece p of lane l sits at ((p * 32) + l) * 16 bytes, so each warp-
// wide shared load of piece p reads 512 contiguous bytes.  Pieces 0 .. 2*NKI-1 hold K
// rows kb+g and kb+8+g (head-dim elements 8c + 32i ..), pieces 2*NKI .. hold V rows
// kb+2c, kb+2c+1, kb+2c+8, kb+2c+9 (elements 8g + 64i ..).  Rows at or past k1 are
// zero-filled; the appended row (index Lapp) comes from k_new / v_new.
template <int D>
__device__ __forceinline__ void issue_block(uint32_t stage_base, const __nv_bfloat16 *Kp, const __nv_bfloat16 *Vp,
                                            const __nv_bfloat16 *kn, const __nv_bfloat16 *vn, int kb, int k1,
                                            int Lapp, int g, int c, int lane)
{
    constexpr int NKI = D / 32, NVI = D / 64;
#pragma unroll
    for (int nt = 0; nt < 2; ++nt) {
        const int j = kb + 8 * nt + g;
        const __nv_bfloat16 *row = (j == Lapp) ? kn : Kp + (long)(j < k1 ? j : 0) * D;
        const int nbytes = j < k1 ? 16 : 0;
#pragma unroll
        for (int i = 0; i < NKI; ++i)
            cp_async16(stage_base + ((nt * NKI + i) * 32 + lane) * 16, row + 8 * c + 32 * i, nbytes);
    }
#pragma unroll
    for (int x = 0; x < 4; ++x) {
        const int j = kb + 2 * c + (x & 1) + 8 * (x >> 1);
        const __nv_bfloat16 *row = (j == Lapp) ? vn : Vp + (long)(j < k1 ? j : 0) * D;
        const int nbytes = j < k1 ? 16 : 0;
#pragma unroll
        for (int i = 0; i < NVI; ++i)
            cp_async16(stage_base + ((2 * NKI + x * NVI + i) * 32 + lane) * 16, row + 8 * g + 64 * i, nbytes);
    }
}

__device__ __forceinline__ uint4 lds_u4(uint32_t addr)
{
    uint4 r;
    asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];" : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w) : "r"(addr));
    return r;
}

constexpr int kDecodeStages = 3;
constexpr int kDecodeWarps = 4;

template <int D>
__global__ void __launch_bounds__(128, 2) decode_mma(DecodeArgs a)
{
    constexpr int NW = kDecodeWarps;
    constexpr int NKI = D / 32;  // 16-byte K pieces per row per thread
    constexpr int NVI = D / 64;  // 16-byte V pieces per row per thread
    constexpr int KS = D / 16;   // k-steps of QK^T
    constexpr int MT = D / 16;   // m-tiles of PV (d on M)
    // dynamic shared memory: the per-warp cp.async rings, then the work plan
    extern __shared__ __align__(16) unsigned char smem_raw[];
    constexpr int RING_BYTES = kDecodeStages * (2 * NKI + 4 * NVI) * 32 * 16;
    const uint32_t ring_base = (uint32_t)__cvta_generic_to_shared(smem_raw);
    int *sm_pre = reinterpret_cast<int *>(smem_raw + NW * RING_BYTES);  // [units + 1] first item of each unit
    int *sm_len = sm_pre + a.units + 1;  // [units] effective length (-1: invalid unit)
    __shared__ long long sm_red[NW];
    __shared__ int sm_scan[NW * 32 + 1];
    const int tid = threadIdx.x, lane = tid & 31, wid = tid >> 5;
    const int units = a.units;

    // ---- plan: identical in every CTA
    const int seg = (units + blockDim.x - 1) / blockDim.x;
    const int u_lo = min(units, tid * seg), u_hi = min(units, u_lo + seg);
    long long tot = 0;
    for (int u = u_lo; u < u_hi; ++u) {
        const int L = a.lens[u];
        const bool ok = unit_ok(L, a.L_cap, a.append);
        if (!ok && blockIdx.x == 0) raise_error(a.err, (a.append && L == a.L_cap) ? ERR_ROOM : ERR_LEN);
        sm_len[u] = ok ? L + a.append : -1;
        tot += ok ? L + a.append : 0;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) tot += __shfl_xor_sync(0xffffffffu, tot, o);
    if (lane == 0) sm_red[wid] = tot;
    __syncthreads();
    tot = 0;
    for (int w = 0; w < NW; ++w) tot += sm_red[w];
    const int total_warps = gridDim.x * NW;
    const long long target = min((long long)kDecodeMaxTarget, 4LL * total_warps);
    long long C = (tot + target - 1) / target;
    C = ((C + 63) / 64) * 64;
    if (C < 256) C = 256;
    int my_items = 0;
    for (int u = u_lo; u < u_hi; ++u) {
        const int le = max(sm_len[u], 0);
        my_items += max(1, (int)((le + C - 1) / C));
    }
    // exclusive scan of my_items over the block
    {
        int incl = my_items;
#pragma unroll
        for (int o = 1; o < 32; o <<= 1) {
            int n = __shfl_up_sync(0xffffffffu, incl, o);
            if (lane >= o) incl += n;
        }
        if (lane == 31) sm_scan[wid] = incl;
        __syncthreads();
        int wbase = 0;
        for (int w = 0; w < wid; ++w) wbase += sm_scan[w];
        int run = wbase + incl - my_items;
        for (int u = u_lo; u < u_hi; ++u) {
            sm_pre[u] = run;
            const int le = max(sm_len[u], 0);
            run += max(1, (int)((le + C - 1) / C));
        }
        if (tid == blockDim.x - 1) sm_pre[units] = run;
    }
    __syncthreads();
    const int total_items = sm_pre[units];
    const int g = lane >> 2, c = lane & 3;
    const bool out_bf16 = a.out_bf16 != 0;

    for (;;) {
        int item = 0;
        if (lane == 0) item = atomicAdd(&a.counters[0], 1);
        item = __shfl_sync(0xffffffffu, item, 0);
        if (item >= total_items) break;
        int lo = 0, hi = units - 1;  // last unit whose first item <= item
        while (lo < hi) {
            const int mid = (lo + hi + 1) >> 1;
            if (sm_pre[mid] <= item) lo = mid; else hi = mid - 1;
        }
        const int u = lo;
        const int first = sm_pre[u], nsplit = sm_pre[u + 1] - first;
        const int split = item - first;
        const int le_raw = sm_len[u];
        const bool valid = le_raw >= 0;
        const int le = valid ? le_raw : 0;
        const int Lapp = (valid && a.append) ? le - 1 : -1;  // index of the appended row
        const int k0 = (int)min((long long)split * C, (long long)le);
        const int k1 = (int)min((long long)k0 + C, (long long)le);
        const long lb = u / a.Hkv;
        const int h = u % a.Hkv;
        const int G = a.G;
        const __nv_bfloat16 *Kp = reinterpret_cast<const __nv_bfloat16 *>(a.K) + (long)u * a.L_cap * D;
        const __nv_bfloat16 *Vp = reinterpret_cast<const __nv_bfloat16 *>(a.V) + (long)u * a.L_cap * D;
        const __nv_bfloat16 *kn = a.append ? reinterpret_cast<const __nv_bfloat16 *>(a.k_new) + (long)u * D : Kp;
        const __nv_bfloat16 *vn = a.append ? reinterpret_cast<const __nv_bfloat16 *>(a.v_new) + (long)u * D : Vp;
        const long qrow0 = lb * a.Hq + (long)h * G;

        // Q fragments (rows g < G), head dim permuted: k-step j takes elements
        // 8c + 32(j/2) + 4(j%2) + {0,1} (a0) and + {2,3} (a2).
        uint32_t qa[KS][2];
        {
            const __nv_bfloat16 *qp = reinterpret_cast<const __nv_bfloat16 *>(a.q) + (qrow0 + g) * D;
#pragma unroll
            for (int i = 0; i < NKI; ++i) {
                uint4 wv = make_uint4(0, 0, 0, 0);
                if (g < G) wv = *reinterpret_cast<const uint4 *>(qp + 8 * c + 32 * i);
                qa[2 * i][0] = wv.x;
                qa[2 * i][1] = wv.y;
                qa[2 * i + 1][0] = wv.z;
                qa[2 * i + 1][1] = wv.w;
            }
        }
        float o[MT][4];
#pragma unroll
        for (int t = 0; t < MT; ++t) o[t][0] = o[t][1] = o[t][2] = o[t][3] = 0.f;
        float m = -INFINITY, l = 0.f;

        constexpr int NP = 2 * NKI + 4 * NVI;  // pieces per thread per block
        const uint32_t ring = ring_base + (uint32_t)wid * (kDecodeStages * NP * 32 * 16);
        const int nblk = (k1 - k0 + 15) / 16;
#pragma unroll
        for (int p = 0; p < kDecodeStages - 1; ++p) {
            if (p < nblk)
                issue_block<D>(ring + p * NP * 512, Kp, Vp, kn, vn, k0 + 16 * p, k1, Lapp, g, c, lane);
            cp_async_commit();
        }
        for (int bi = 0; bi < nblk; ++bi) {
            {
                const int nb = bi + kDecodeStages - 1;
                if (nb < nblk)
                    issue_block<D>(ring + (nb % kDecodeStages) * NP * 512, Kp, Vp, kn, vn, k0 + 16 * nb, k1, Lapp,
                                   g, c, lane);
                cp_async_commit();
            }
            cp_async_wait<kDecodeStages - 1>();
            const int kb = k0 + 16 * bi;
            const uint32_t st = ring + (bi % kDecodeStages) * NP * 512 + lane * 16;
            float s0[4] = {0.f, 0.f, 0.f, 0.f}, s1[4] = {0.f, 0.f, 0.f, 0.f};
#pragma unroll
            for (int i = 0; i < NKI; ++i) {
                const uint4 k0v = lds_u4(st + (0 * NKI + i) * 512);
                const uint4 k1v = lds_u4(st + (1 * NKI + i) * 512);
                mma_bf16(s0, qa[2 * i][0], 0u, qa[2 * i][1], 0u, k0v.x, k0v.y);
                mma_bf16(s1, qa[2 * i][0], 0u, qa[2 * i][1], 0u, k1v.x, k1v.y);
                mma_bf16(s0, qa[2 * i + 1][0], 0u, qa[2 * i + 1][1], 0u, k0v.z, k0v.w);
                mma_bf16(s1, qa[2 * i + 1][0], 0u, qa[2 * i + 1][1], 0u, k1v.z, k1v.w);
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
            const float mn = fmaxf(m, mb);
            const float base = (mn == -INFINITY) ? 0.f : mn;
            const float alpha = fast_exp2(m - base);
            const float p0 = fast_exp2(x0 - base), p1 = fast_exp2(x1 - base);
            const float p2 = fast_exp2(x2 - base), p3 = fast_exp2(x3 - base);
            l = l * alpha + ((p0 + p1) + (p2 + p3));
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
            // P enters the PV product as bf16 hi + lo parts (two MMAs), which keeps about
            // 16 significant bits of each probability instead of 8.
            uint32_t ph0, ph1, pl0, pl1;
            split_bf16(p0, p1, ph0, pl0);
            split_bf16(p2, p3, ph1, pl1);
#pragma unroll
            for (int i = 0; i < NVI; ++i) {
                const uint4 v0 = lds_u4(st + (2 * NKI + 0 * NVI + i) * 512);
                const uint4 v1 = lds_u4(st + (2 * NKI + 1 * NVI + i) * 512);
                const uint4 v2 = lds_u4(st + (2 * NKI + 2 * NVI + i) * 512);
                const uint4 v3 = lds_u4(st + (2 * NKI + 3 * NVI + i) * 512);
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    const uint32_t W0 = word(v0, x), W1 = word(v1, x), W2 = word(v2, x), W3 = word(v3, x);
                    const uint32_t A0 = __byte_perm(W0, W1, 0x5410), A1 = __byte_perm(W0, W1, 0x7632);
                    const uint32_t A2 = __byte_perm(W2, W3, 0x5410), A3 = __byte_perm(W2, W3, 0x7632);
                    mma_bf16(o[4 * i + x], A0, A1, A2, A3, ph0, ph1);
                    mma_bf16(o[4 * i + x], A0, A1, A2, A3, pl0, pl1);
                }
            }
        }
        l += __shfl_xor_sync(0xffffffffu, l, 1);
        l += __shfl_xor_sync(0xffffffffu, l, 2);

        // the warp that covers the appended index writes the new row into the cache
        if (Lapp >= k0 && Lapp < k1) {
            constexpr int PCS = D / 8;  // 16-byte pieces per row
            if (lane < 2 * PCS) {
                const bool isv = lane >= PCS;
                const int pc = isv ? lane - PCS : lane;
                const __nv_bfloat16 *src = (isv ? vn : kn) + pc * 8;
                __nv_bfloat16 *dst = reinterpret_cast<__nv_bfloat16 *>(isv ? a.V : a.K) +
                                     ((long)u * a.L_cap + Lapp) * D + pc * 8;
                *reinterpret_cast<uint4 *>(dst) = *reinterpret_cast<const uint4 *>(src);
            }
        }

        const int q0 = 2 * c, q1 = 2 * c + 1;
        const float l0 = __shfl_sync(0xffffffffu, l, q0 * 4), l1 = __shfl_sync(0xffffffffu, l, q1 * 4);
        if (nsplit == 1) {
            const float inv0 = l0 > 0.f ? 1.f / l0 : 0.f, inv1 = l1 > 0.f ? 1.f / l1 : 0.f;
#pragma unroll
            for (int i = 0; i < NVI; ++i) {
                const long d0 = 64 * i + 8 * g;
#pragma unroll
                for (int x = 0; x < 4; ++x) {
                    if (q0 < G) {
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + q0) * D + d0 + 2 * x, o[4 * i + x][0] * inv0);
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + q0) * D + d0 + 2 * x + 1, o[4 * i + x][2] * inv0);
                    }
                    if (q1 < G) {
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + q1) * D + d0 + 2 * x, o[4 * i + x][1] * inv1);
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + q1) * D + d0 + 2 * x + 1, o[4 * i + x][3] * inv1);
                    }
                }
            }
            if (c == 0 && g < G && a.lse) a.lse[qrow0 + g] = l > 0.f ? (m + log2f(l)) * kLn2 : -INFINITY;
        } else {
            float *po = a.part_o + (size_t)item * G * D;
#pragma unroll
            for (int i = 0; i < NVI; ++i) {
                const int d0 = 64 * i + 8 * g;
                if (q0 < G) {
                    float4 *dst = reinterpret_cast<float4 *>(po + (size_t)q0 * D + d0);
                    dst[0] = make_float4(o[4 * i + 0][0], o[4 * i + 0][2], o[4 * i + 1][0], o[4 * i + 1][2]);
                    dst[1] = make_float4(o[4 * i + 2][0], o[4 * i + 2][2], o[4 * i + 3][0], o[4 * i + 3][2]);
                }
                if (q1 < G) {
                    float4 *dst = reinterpret_cast<float4 *>(po + (size_t)q1 * D + d0);
                    dst[0] = make_float4(o[4 * i + 0][1], o[4 * i + 0][3], o[4 * i + 1][1], o[4 * i + 1][3]);
                    dst[1] = make_float4(o[4 * i + 2][1], o[4 * i + 2][3], o[4 * i + 3][1], o[4 * i + 3][3]);
                }
            }
            if (c == 0 && g < G) {
                a.part_ml[((size_t)item * G + g) * 2 + 0] = m;
                a.part_ml[((size_t)item * G + g) * 2 + 1] = l;
            }
            __threadfence();
            __syncwarp();
            int old = 0;
            if (lane == 0) old = atomicAdd(&a.counters[2 + u], 1);
            old = __shfl_sync(0xffffffffu, old, 0);
            if (old == nsplit - 1) {  // last item of this unit: merge the partials
                __threadfence();
                constexpr int PER = D / 32;
                for (int qq = 0; qq < G; ++qq) {
                    float M = -INFINITY;
                    for (int s = 0; s < nsplit; ++s)
                        M = fmaxf(M, __ldcg(a.part_ml + ((size_t)(first + s) * G + qq) * 2));
                    float Ls = 0.f, acc[PER];
#pragma unroll
                    for (int e = 0; e < PER; ++e) acc[e] = 0.f;
                    if (M != -INFINITY) {
                        for (int s = 0; s < nsplit; ++s) {
                            const size_t it = (size_t)(first + s) * G + qq;
                            const float ms = __ldcg(a.part_ml + it * 2);
                            const float wt = fast_exp2(ms - M);
                            Ls += __ldcg(a.part_ml + it * 2 + 1) * wt;
                            const float *src = a.part_o + it * D + lane * PER;
#pragma unroll
                            for (int e = 0; e < PER; ++e) acc[e] += __ldcg(src + e) * wt;
                        }
                    }
                    const float inv = Ls > 0.f ? 1.f / Ls : 0.f;
#pragma unroll
                    for (int e = 0; e < PER; ++e)
                        store_out<__nv_bfloat16>(a.out, out_bf16, (qrow0 + qq) * D + lane * PER + e, acc[e] * inv);
                    if (lane == 0 && a.lse) a.lse[qrow0 + qq] = Ls > 0.f ? (M + log2f(Ls)) * kLn2 : -INFINITY;
                }
            }
        }
    }
    // the last warp of the grid advances the lengths (every plan has been read by then)
    int done = 0;
    if (lane == 0) done = atomicAdd(&a.counters[1], 1);
    done = __shfl_sync(0xffffffffu, done, 0);
    if (done == total_warps - 1 && a.append) {
        __threadfence();
        for (int u = lane; u < units; u += 32)
            if (sm_len[u] >= 0) a.lens[u] = sm_len[u];
    }
}

constexpr int kMaxMmaUnits = 8192;  // plan (8 B per unit) + rings stay within one CTA's shared memory

static int mma_blocks_per_sm(const void *fn, size_t smem)
{
    int n = 0;
    if (cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, fn, 128, smem) != cudaSuccess || n < 1) n = 1;
    return n;
}

cudaError_t launch_decode(const reco_kv &kv, const void *q, const void *k_new, const void *v_new,
                          int32_t *lens, float scale, void *out, reco_dtype out_dtype, float *lse,
                          const DecodeWs &ws, unsigned *err, cudaStream_t s)
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
    a.max_items = ws.max_items;
    a.append = (k_new && v_new) ? 1 : 0;
    a.out_bf16 = out_dtype == RECO_BF16 ? 1 : 0;
    a.c2 = scale * kLog2e;
    a.err = err;
    if (kv.dtype == RECO_BF16 && a.G <= 8 && a.units <= kMaxMmaUnits) {
        cudaError_t e = cudaMemsetAsync(ws.counters, 0, (size_t)(2 + a.units) * 4, s);
        if (e != cudaSuccess) return e;
        const size_t ring = (size_t)kDecodeWarps * kDecodeStages * (kv.d == 64 ? 8 : 16) * 32 * 16;
        const size_t smem = ring + (size_t)(2 * a.units + 1) * sizeof(int);
        const void *fn = kv.d == 64 ? (const void *)decode_mma<64> : (const void *)decode_mma<128>;
        e = cudaFuncSetAttribute(fn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        const int grid = device_sm_count() * mma_blocks_per_sm(fn, smem);
        if (kv.d == 64)
            decode_mma<64><<<grid, 128, smem, s>>>(a);
        else
            decode_mma<128><<<grid, 128, smem, s>>>(a);
        return cudaGetLastError();
    }
    const unsigned grid = (unsigned)a.units;
    if (kv.dtype == RECO_F32) {
        if (kv.d == 64) decode_simt<float, 64><<<grid, 128, 0, s>>>(a);
        else decode_simt<float, 128><<<grid, 128, 0, s>>>(a);
    } else {
        if (kv.d == 64) decode_simt<__nv_bfloat16, 64><<<grid, 128, 0, s>>>(a);
        else decode_simt<__nv_bfloat16, 128><<<grid, 128, 0, s>>>(a);
    }
    return cudaGetLastError();
}

}  // namespace reco
