// vocab.cu -- the two vocabulary-side steps of ReCo's generation control (Sec. 3.3).
//
// reflect_penalty: Eq. 3 picks beta_i in {0, beta/2, beta} from the band of the
// step reward (float32 compares); Eq. 4 subtracts it from the logit of every
// reflection token, in place.  R is a set: an id listed twice is penalised once.
//
// ppl_rows + ppl_finish: Eq. 5 log p(x_t) = z[x_t] - logsumexp(z) per answer row
// (one CTA per row, one streaming pass with an online max/sum), then per sequence
// PPL = exp(-mean log p) and the Eq. 6 stop flag PPL <= tau_p.
#include "common.cuh"
#include "internal.h"

namespace reco {

__global__ void reflect_penalty_kernel(float *logits, int V, const int32_t *__restrict__ ids, int n_ids,
                                       const float *__restrict__ rewards, float tau_l, float tau_h,
                                       float beta, float *beta_out, unsigned *err)
{
    const int b = blockIdx.x;
    const float v = rewards[b];
    const float bi = (v <= tau_l) ? 0.f : ((v >= tau_h) ? beta : beta * 0.5f);
    if (threadIdx.x == 0 && beta_out) beta_out[b] = bi;
    for (int i = threadIdx.x; i < n_ids; i += blockDim.x) {
        const int id = ids[i];
        if (id < 0 || id >= V) {
            if (b == 0) raise_error(err, ERR_ID);
            continue;
        }
        bool dup = false;
        for (int k = 0; k < i && !dup; ++k) dup = ids[k] == id;
        if (dup || bi == 0.f) continue;
        float *p = logits + (size_t)b * V + id;
        *p = __fsub_rn(*p, bi);
    }
}

cudaError_t launch_penalty(float *logits, int B, int V, const int32_t *ids, int n_ids,
                           const float *rewards, float tau_l, float tau_h, float beta, float *beta_out,
                           unsigned *err, cudaStream_t s)
{
    int nt = n_ids < 32 ? 32 : (n_ids > 256 ? 256 : ((n_ids + 31) / 32) * 32);
    reflect_penalty_kernel<<<B, nt, 0, s>>>(logits, V, ids, n_ids, rewards, tau_l, tau_h, beta, beta_out,
                                            err);
    return cudaGetLastError();
}

// Online (max, sum) in the log2 domain over four values.
__device__ __forceinline__ void ms_add4(float &m, float &s, float a, float b, float c, float d)
{
    const float mx = fmaxf(fmaxf(a, b), fmaxf(c, d));
    if (mx > m) {
        s *= fast_exp2(m - mx);
        m = mx;
    }
    s += fast_exp2(a - m) + fast_exp2(b - m) + fast_exp2(c - m) + fast_exp2(d - m);
}

template <int NT>
__global__ void __launch_bounds__(NT) ppl_rows(const float *__restrict__ logits,
                                               const int32_t *__restrict__ tokens,
                                               const int32_t *__restrict__ n_valid, int n, int V,
                                               float *__restrict__ lp, unsigned *err)
{
    __shared__ float sm_m[NT / 32], sm_s[NT / 32];
    const int t = blockIdx.x, b = blockIdx.y;
    const int nb = n_valid ? min(n_valid[b], n) : n;
    if (t >= nb) return;
    const float *z = logits + ((size_t)b * n + t) * V;
    float m = -INFINITY, s = 0.f;
    if ((V & 3) == 0) {
        const float4 *z4 = reinterpret_cast<const float4 *>(z);
        for (int i = threadIdx.x; i < V / 4; i += NT) {
            const float4 x = __ldcs(z4 + i);
            ms_add4(m, s, x.x * kLog2e, x.y * kLog2e, x.z * kLog2e, x.w * kLog2e);
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
        float r;
        if (x < 0 || x >= V) {
            raise_error(err, ERR_TOKEN);
            r = __int_as_float(0x7fc00000);
        } else {
            r = z[x] - (M + log2f(S)) * kLn2;
        }
        lp[(size_t)b * n + t] = r;
    }
}

__global__ void ppl_finish(const float *__restrict__ lp, const int32_t *__restrict__ n_valid, int B, int n,
                           float tau_p, float *__restrict__ ppl, uint8_t *__restrict__ stop)
{
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
    if (n > 0) {
        ppl_rows<512><<<dim3(n, B), 512, 0, s>>>(logits, tokens, n_valid, n, V, lp_ws, err);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    ppl_finish<<<(B + 127) / 128, 128, 0, s>>>(lp_ws, n_valid, B, n, tau_p, ppl, stop);
    return cudaGetLastError();
}

}  // namespace reco
