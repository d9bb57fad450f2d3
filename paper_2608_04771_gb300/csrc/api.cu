// api.cu -- the extern "C" entry points of libreco (declared in include/reco.h):
// host-side argument checks, workspace carving, the sticky device error word, and
// the host helpers for Eq. 1, the keep count, the Eq. 3 band and the probe trigger.
#include <math.h>
#include <stdarg.h>
#include <stdio.h>

#include <mutex>
#include <string>

#include <cuda.h>

#include "common.cuh"
#include "internal.h"

namespace {

thread_local std::string g_last_error;

reco_status fail(reco_status st, const char *fmt, ...)
{
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_last_error = buf;
    return st;
}

reco_status cuda_fail(cudaError_t e, const char *where)
{
    return fail(RECO_ECUDA, "%s: %s", where, cudaGetErrorString(e));
}

// One sticky error word per device; kernels receive its device address.
__device__ unsigned int g_reco_error_word;

std::mutex g_mu;
unsigned *g_err_addr[128];
int g_sm_count[128];

reco_status error_word(unsigned **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= 128) return fail(RECO_EUNSUPPORTED, "device index %d out of range", dev);
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_err_addr[dev]) {
        void *p = nullptr;
        e = cudaGetSymbolAddress(&p, g_reco_error_word);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(error word)");
        g_err_addr[dev] = (unsigned *)p;
    }
    *out = g_err_addr[dev];
    return RECO_OK;
}

bool al16(const void *p) { return ((uintptr_t)p & 15u) == 0; }

reco_status check_kv(const reco_kv *kv, bool need_kv_ptrs = true)
{
    if (!kv) return fail(RECO_EINVAL, "kv descriptor is NULL");
    if (kv->n_layers < 1 || kv->B < 1 || kv->H_kv < 1 || kv->H_q < 1 || kv->L_cap < 1)
        return fail(RECO_EINVAL, "kv dimensions must be >= 1 (layers %d, B %d, H_q %d, H_kv %d, L_cap %d)",
                    kv->n_layers, kv->B, kv->H_q, kv->H_kv, kv->L_cap);
    if (kv->H_q % kv->H_kv != 0) return fail(RECO_EINVAL, "H_q (%d) is not a multiple of H_kv (%d)", kv->H_q, kv->H_kv);
    if (kv->dtype != RECO_F32 && kv->dtype != RECO_BF16) return fail(RECO_EINVAL, "unknown dtype %d", (int)kv->dtype);
    if (kv->d != 64 && kv->d != 128) return fail(RECO_EUNSUPPORTED, "head dim %d (supported: 64, 128)", kv->d);
    long long units = (long long)kv->n_layers * kv->B * kv->H_kv;
    if (units > 65535) return fail(RECO_EUNSUPPORTED, "%lld units exceed 65535", units);
    if (need_kv_ptrs) {
        if (!kv->k || !kv->v) return fail(RECO_EINVAL, "K or V pointer is NULL");
        if (!al16(kv->k) || !al16(kv->v)) return fail(RECO_EINVAL, "K and V must be 16-byte aligned");
    }
    return RECO_OK;
}

reco_status check_ws(void *ws, size_t have, size_t need)
{
    if (need == 0) return RECO_OK;
    if (!ws) return fail(RECO_EINVAL, "workspace is NULL (%zu bytes needed)", need);
    if (((uintptr_t)ws & 255u) != 0) return fail(RECO_EINVAL, "workspace must be 256-byte aligned");
    if (have < need) return fail(RECO_EINVAL, "workspace has %zu bytes, %zu needed", have, need);
    return RECO_OK;
}

}  // namespace

namespace reco {
bool score_shape_supported(const reco_kv &kv, int w);

int device_sm_count()
{
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0 || dev >= 128) return 148;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_sm_count[dev]) {
        int n = 0;
        if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n < 1) n = 148;
        g_sm_count[dev] = n;
    }
    return g_sm_count[dev];
}
typedef CUresult (*EncodeTiledFn)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                  const cuuint64_t *, const cuuint32_t *, const cuuint32_t *, CUtensorMapInterleave,
                                  CUtensorMapSwizzle, CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn()
{
    static EncodeTiledFn fn = nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!fn) {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = (EncodeTiledFn)p;
    }
    return fn;
}

bool encode_bf16_2d(void *map, const void *base, unsigned long long rows, int cols, int box_cols, int box_rows)
{
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {(cuuint64_t)cols, (cuuint64_t)rows};
    const cuuint64_t strides[1] = {(cuuint64_t)cols * 2};
    const cuuint32_t box[2] = {(cuuint32_t)box_cols, (cuuint32_t)box_rows};
    const cuuint32_t estr[2] = {1, 1};
    return fn(reinterpret_cast<CUtensorMap *>(map), CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base),
              dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

}  // namespace reco

extern "C" {

const char *reco_last_error(void) { return g_last_error.c_str(); }

reco_status reco_retention_ratio(const float *rewards, int n, double base, double delta, double *ratio_out)
{
    if (!rewards || !ratio_out) return fail(RECO_EINVAL, "NULL pointer");
    if (n < 1) return fail(RECO_EINVAL, "reward history is empty");
    double sum = 0.0, vmin = rewards[0], vmax = rewards[0];
    for (int i = 0; i < n; ++i) {
        const double v = rewards[i];
        sum += v;
        vmin = v < vmin ? v : vmin;
        vmax = v > vmax ? v : vmax;
    }
    const double mean = sum / (double)n, range = vmax - vmin;
    *ratio_out = range == 0.0 ? base : base - delta * (((double)rewards[n - 1] - mean) / range);
    return RECO_OK;
}

reco_status reco_keep_count(double ratio, int L, int w, int32_t *m_out)
{
    if (!m_out) return fail(RECO_EINVAL, "NULL pointer");
    if (w < 1 || L < w) return fail(RECO_EINVAL, "need 1 <= w <= L (w %d, L %d)", w, L);
    if (!(ratio == ratio)) return fail(RECO_EINVAL, "ratio is NaN");
    const double f = floor(ratio * (double)L);
    *m_out = f < (double)w ? w : (f > (double)L ? L : (int32_t)f);
    return RECO_OK;
}

int reco_penalty_band(float v, float tau_l, float tau_h)
{
    if (v <= tau_l) return 0;
    if (v >= tau_h) return 2;
    return 1;
}

int reco_probe_trigger(float v_prev, float v_cur, float tau_h) { return v_prev >= tau_h && v_cur >= tau_h; }

reco_status reco_workspace_bytes(reco_op op, const reco_kv *kv, int w, size_t *bytes_out)
{
    if (!bytes_out) return fail(RECO_EINVAL, "NULL pointer");
    reco_status st;
    switch (op) {
    case RECO_OP_SCORE:
        if ((st = check_kv(kv, false)) != RECO_OK) return st;
        if (w < 1) return fail(RECO_EINVAL, "window w must be >= 1");
        *bytes_out = reco::score_ws_layout(*kv, w, nullptr).bytes;
        return RECO_OK;
    case RECO_OP_SELECT:
        if ((st = check_kv(kv, false)) != RECO_OK) return st;
        *bytes_out = reco::select_ws_layout(*kv, nullptr).bytes;
        return RECO_OK;
    case RECO_OP_DECODE:
        if ((st = check_kv(kv, false)) != RECO_OK) return st;
        *bytes_out = reco::decode_ws_layout(*kv, nullptr).bytes;
        return RECO_OK;
    case RECO_OP_SAMPLE:
        if (w < 1 || w > reco::kSampleSeg * reco::kSampleMaxSeg)
            return fail(RECO_EINVAL, "vocabulary size %d outside [1, %d]", w, reco::kSampleSeg * reco::kSampleMaxSeg);
        *bytes_out = (size_t)((w + reco::kSampleSeg - 1) / reco::kSampleSeg) * 8;
        return RECO_OK;
    case RECO_OP_PPL:
        if (w < 0) return fail(RECO_EINVAL, "answer rows B*n must be >= 0");
        *bytes_out = reco::align256((size_t)w * 4);
        return RECO_OK;
    }
    return fail(RECO_EINVAL, "unknown op %d", (int)op);
}

reco_status reco_check(cudaStream_t stream)
{
    cudaError_t e = cudaStreamSynchronize(stream);
    if (e != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    unsigned *p;
    reco_status st = error_word(&p);
    if (st != RECO_OK) return st;
    unsigned h = 0;
    if ((e = cudaMemcpyAsync(&h, p, sizeof h, cudaMemcpyDeviceToHost, stream)) != cudaSuccess)
        return cuda_fail(e, "read error word");
    if ((e = cudaStreamSynchronize(stream)) != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
    if (h) {
        if ((e = cudaMemsetAsync(p, 0, sizeof h, stream)) != cudaSuccess) return cuda_fail(e, "clear error word");
        if ((e = cudaStreamSynchronize(stream)) != cudaSuccess) return cuda_fail(e, "cudaStreamSynchronize");
        return fail(RECO_EDEVICE, "device error word 0x%x:%s%s%s%s%s%s%s", h, (h & reco::ERR_LEN) ? " length-out-of-range" : "",
                    (h & reco::ERR_KEEP) ? " keep-out-of-range" : "", (h & reco::ERR_ID) ? " id-out-of-range" : "",
                    (h & reco::ERR_TOKEN) ? " token-out-of-range" : "", (h & reco::ERR_ROOM) ? " no-room-to-append" : "",
                    (h & reco::ERR_INTERNAL) ? " internal-check" : "", (h & reco::ERR_NORM) ? " normaliser-not-finite" : "");
    }
    return RECO_OK;
}

reco_status reco_score_cache(const reco_kv *kv, const void *q_win, const int32_t *lens, const int32_t *keep, int w,
                             int pool_kernel, float scale, float *scores, void *ws, size_t ws_bytes,
                             cudaStream_t stream)
{
    reco_status st = check_kv(kv);
    if (st != RECO_OK) return st;
    if (!q_win || !lens || !scores) return fail(RECO_EINVAL, "NULL q_win, lens or scores");
    if (!al16(q_win) || ((uintptr_t)scores & 3u) || ((uintptr_t)lens & 3u) || ((uintptr_t)keep & 3u))
        return fail(RECO_EINVAL, "q_win must be 16-byte aligned, lens, keep and scores 4-byte aligned");
    if (w < 1 || w > kv->L_cap) return fail(RECO_EINVAL, "window w=%d outside [1, L_cap=%d]", w, kv->L_cap);
    if (pool_kernel < 1 || (pool_kernel & 1) == 0) return fail(RECO_EINVAL, "pool_kernel %d must be odd and >= 1", pool_kernel);
    if (!(scale == scale)) return fail(RECO_EINVAL, "scale is NaN");
    const int G = kv->H_q / kv->H_kv;
    if ((long long)G * w > 4096) return fail(RECO_EUNSUPPORTED, "G*w = %lld window rows exceed 4096", (long long)G * w);
    if (!reco::score_shape_supported(*kv, w))
        return fail(RECO_EUNSUPPORTED, "G*w*d too large for the scoring kernels (G %d, w %d, d %d)", G, w, kv->d);
    reco::ScoreWs lay = reco::score_ws_layout(*kv, w, ws);
    if ((st = check_ws(ws, ws_bytes, lay.bytes)) != RECO_OK) return st;
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_score(*kv, q_win, lens, keep, w, pool_kernel, scale, scores, lay, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_score_cache launch");
}

reco_status reco_score_cache_lse(const reco_kv *kv, const void *q_win, const int32_t *lens, const int32_t *keep,
                                 const float *row_lse, int w, int pool_kernel, float scale, float *scores, void *ws,
                                 size_t ws_bytes, cudaStream_t stream)
{
    reco_status st = check_kv(kv);
    if (st != RECO_OK) return st;
    if (!q_win || !lens || !row_lse || !scores) return fail(RECO_EINVAL, "NULL q_win, lens, row_lse or scores");
    if (!al16(q_win) || ((uintptr_t)scores & 3u) || ((uintptr_t)lens & 3u) || ((uintptr_t)keep & 3u) ||
        ((uintptr_t)row_lse & 3u))
        return fail(RECO_EINVAL, "q_win must be 16-byte aligned, lens, keep, row_lse and scores 4-byte aligned");
    if (w < 1 || w > kv->L_cap) return fail(RECO_EINVAL, "window w=%d outside [1, L_cap=%d]", w, kv->L_cap);
    if (pool_kernel < 1 || (pool_kernel & 1) == 0) return fail(RECO_EINVAL, "pool_kernel %d must be odd and >= 1", pool_kernel);
    if (!(scale == scale)) return fail(RECO_EINVAL, "scale is NaN");
    const int G = kv->H_q / kv->H_kv;
    if ((long long)G * w > 4096) return fail(RECO_EUNSUPPORTED, "G*w = %lld window rows exceed 4096", (long long)G * w);
    if (!reco::score_shape_supported(*kv, w))
        return fail(RECO_EUNSUPPORTED, "G*w*d too large for the scoring kernels (G %d, w %d, d %d)", G, w, kv->d);
    reco::ScoreWs lay = reco::score_ws_layout(*kv, w, ws);
    if ((st = check_ws(ws, ws_bytes, lay.bytes)) != RECO_OK) return st;
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_score_lse(*kv, q_win, lens, keep, row_lse, w, pool_kernel, scale, scores, lay, err,
                                           stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_score_cache_lse launch");
}

reco_status reco_lse_push(const float *lse, int64_t n, float *ring, int slots, int64_t *slot, cudaStream_t stream)
{
    if (n < 1 || slots < 1) return fail(RECO_EINVAL, "need n >= 1 and slots >= 1");
    if (!lse || !ring || !slot) return fail(RECO_EINVAL, "NULL lse, ring or slot");
    if (((uintptr_t)lse & 3u) || ((uintptr_t)ring & 3u) || ((uintptr_t)slot & 7u))
        return fail(RECO_EINVAL, "lse and ring must be 4-byte aligned, slot 8-byte aligned");
    unsigned *err;
    reco_status st = error_word(&err);
    if (st != RECO_OK) return st;
    cudaError_t e = reco::launch_lse_push(lse, (long)n, ring, slots, reinterpret_cast<long long *>(slot), err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_lse_push launch");
}

reco_status reco_copy_row(const void *src, int64_t rows, int64_t row_bytes, const int64_t *index, void *dst,
                          cudaStream_t stream)
{
    if (rows < 1 || row_bytes < 16 || row_bytes % 16) return fail(RECO_EINVAL, "need rows >= 1 and row_bytes a positive multiple of 16");
    if (!src || !index || !dst) return fail(RECO_EINVAL, "NULL src, index or dst");
    if (!al16(src) || !al16(dst) || ((uintptr_t)index & 7u))
        return fail(RECO_EINVAL, "src and dst must be 16-byte aligned, index 8-byte aligned");
    unsigned *err;
    reco_status st = error_word(&err);
    if (st != RECO_OK) return st;
    cudaError_t e = reco::launch_copy_row(src, (long long)rows, (long long)row_bytes,
                                          reinterpret_cast<const long long *>(index), dst, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_copy_row launch");
}

reco_status reco_select_compact(const reco_kv *kv, const float *scores, int32_t *lens, const int32_t *keep, int w,
                                int32_t *kept_idx, void *ws, size_t ws_bytes, cudaStream_t stream)
{
    reco_status st = check_kv(kv);
    if (st != RECO_OK) return st;
    if (!scores || !lens || !keep) return fail(RECO_EINVAL, "NULL scores, lens or keep");
    if (((uintptr_t)scores & 3u) || ((uintptr_t)lens & 3u) || ((uintptr_t)keep & 3u) || ((uintptr_t)kept_idx & 3u))
        return fail(RECO_EINVAL, "scores, lens, keep and kept_idx must be 4-byte aligned");
    if (w < 1 || w > kv->L_cap) return fail(RECO_EINVAL, "window w=%d outside [1, L_cap=%d]", w, kv->L_cap);
    reco::SelectWs lay = reco::select_ws_layout(*kv, ws);
    if ((st = check_ws(ws, ws_bytes, lay.bytes)) != RECO_OK) return st;
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_select_compact(*kv, scores, lens, keep, w, kept_idx, lay, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_select_compact launch");
}

reco_status reco_select_topm(const reco_kv *kv, const float *scores, const int32_t *lens, const int32_t *keep, int w,
                             int32_t *kept_idx, void *ws, size_t ws_bytes, cudaStream_t stream)
{
    reco_status st = check_kv(kv, false);
    if (st != RECO_OK) return st;
    if (!scores || !lens || !keep || !kept_idx) return fail(RECO_EINVAL, "NULL scores, lens, keep or kept_idx");
    if (((uintptr_t)scores & 3u) || ((uintptr_t)lens & 3u) || ((uintptr_t)keep & 3u) || ((uintptr_t)kept_idx & 3u))
        return fail(RECO_EINVAL, "scores, lens, keep and kept_idx must be 4-byte aligned");
    if (w < 1 || w > kv->L_cap) return fail(RECO_EINVAL, "window w=%d outside [1, L_cap=%d]", w, kv->L_cap);
    reco::SelectWs lay = reco::select_ws_layout(*kv, ws);
    if ((st = check_ws(ws, ws_bytes, lay.bytes)) != RECO_OK) return st;
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_select_only(*kv, scores, lens, keep, w, kept_idx, lay, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_select_topm launch");
}

reco_status reco_compact(const reco_kv *kv, const int32_t *kept_idx, int32_t *lens, const int32_t *keep, int w,
                         cudaStream_t stream)
{
    reco_status st = check_kv(kv);
    if (st != RECO_OK) return st;
    if (!kept_idx || !lens || !keep) return fail(RECO_EINVAL, "NULL kept_idx, lens or keep");
    if (((uintptr_t)lens & 3u) || ((uintptr_t)keep & 3u) || ((uintptr_t)kept_idx & 3u))
        return fail(RECO_EINVAL, "lens, keep and kept_idx must be 4-byte aligned");
    if (w < 1 || w > kv->L_cap) return fail(RECO_EINVAL, "window w=%d outside [1, L_cap=%d]", w, kv->L_cap);
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_compact(*kv, kept_idx, lens, keep, w, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_compact launch");
}

}  // extern "C"

namespace {
reco_status decode_checked(const reco_kv *kv, const void *q, const void *k_new, const void *v_new, int32_t *lens,
                           float scale, void *out, reco_dtype out_dtype, float *lse, float *ring, int slots,
                           int64_t *slot, void *q_ring, void *ws, size_t ws_bytes, cudaStream_t stream,
                           const char *name)
{
    reco_status st = check_kv(kv);
    if (st != RECO_OK) return st;
    if (!q || !lens || !out) return fail(RECO_EINVAL, "NULL q, lens or out");
    if ((k_new == nullptr) != (v_new == nullptr)) return fail(RECO_EINVAL, "k_new and v_new must both be given or both NULL");
    if (!al16(q) || !al16(out) || (k_new && (!al16(k_new) || !al16(v_new))))
        return fail(RECO_EINVAL, "q, out, k_new and v_new must be 16-byte aligned");
    if (((uintptr_t)lens & 3u) || ((uintptr_t)lse & 3u)) return fail(RECO_EINVAL, "lens and lse must be 4-byte aligned");
    if (out_dtype != RECO_F32 && out_dtype != RECO_BF16) return fail(RECO_EINVAL, "unknown out_dtype %d", (int)out_dtype);
    const int G = kv->H_q / kv->H_kv;
    if (G > 16) return fail(RECO_EUNSUPPORTED, "G = %d query heads per KV head (at most 16)", G);
    if (!(scale == scale)) return fail(RECO_EINVAL, "scale is NaN");
    reco::DecodeWs lay = reco::decode_ws_layout(*kv, ws);
    if ((st = check_ws(ws, ws_bytes, lay.bytes)) != RECO_OK) return st;
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_decode(*kv, q, k_new, v_new, lens, scale, out, out_dtype, lse, lay, err, stream, ring,
                                        slots, reinterpret_cast<long long *>(slot), q_ring);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, name);
}
}  // namespace

extern "C" {

reco_status reco_decode_attn(const reco_kv *kv, const void *q, const void *k_new, const void *v_new, int32_t *lens,
                             float scale, void *out, reco_dtype out_dtype, float *lse, void *ws, size_t ws_bytes,
                             cudaStream_t stream)
{
    return decode_checked(kv, q, k_new, v_new, lens, scale, out, out_dtype, lse, nullptr, 0, nullptr, nullptr, ws,
                          ws_bytes, stream, "reco_decode_attn launch");
}

reco_status reco_decode_attn_ring(const reco_kv *kv, const void *q, const void *k_new, const void *v_new,
                                  int32_t *lens, float scale, void *out, reco_dtype out_dtype, float *ring, int slots,
                                  int64_t *slot, void *q_ring, void *ws, size_t ws_bytes, cudaStream_t stream)
{
    if (slots < 1 || !ring || !slot) return fail(RECO_EINVAL, "need slots >= 1 and non-NULL ring and slot");
    if (((uintptr_t)ring & 3u) || ((uintptr_t)slot & 7u))
        return fail(RECO_EINVAL, "ring must be 4-byte aligned, slot 8-byte aligned");
    if (q_ring && !al16(q_ring)) return fail(RECO_EINVAL, "q_ring must be 16-byte aligned");
    return decode_checked(kv, q, k_new, v_new, lens, scale, out, out_dtype, nullptr, ring, slots, slot, q_ring, ws,
                          ws_bytes, stream, "reco_decode_attn_ring launch");
}

reco_status reco_reflect_penalty(float *logits, int B, int V, const int32_t *ids, int n_ids, const float *rewards,
                                 float tau_l, float tau_h, float beta, float *beta_out, cudaStream_t stream)
{
    if (B < 1 || V < 1 || n_ids < 0) return fail(RECO_EINVAL, "need B >= 1, V >= 1, n_ids >= 0");
    if (!logits || !rewards || (n_ids > 0 && !ids)) return fail(RECO_EINVAL, "NULL logits, rewards or ids");
    if (B > 65535) return fail(RECO_EUNSUPPORTED, "B = %d exceeds 65535", B);
    if (!(beta >= 0.f)) return fail(RECO_EINVAL, "beta must be >= 0");
    unsigned *err;
    reco_status st = error_word(&err);
    if (st != RECO_OK) return st;
    cudaError_t e = reco::launch_penalty(logits, B, V, ids, n_ids, rewards, tau_l, tau_h, beta, beta_out, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_reflect_penalty launch");
}

reco_status reco_penalty_sample(float *logits, int B, int V, const int32_t *ids, int n_ids, const float *rewards,
                                float tau_l, float tau_h, float beta, const float *uniforms, int32_t *tokens,
                                float *beta_out, void *ws, size_t ws_bytes, cudaStream_t stream)
{
    if (B < 1 || V < 1 || n_ids < 0) return fail(RECO_EINVAL, "need B >= 1, V >= 1, n_ids >= 0");
    if (!logits || !rewards || !uniforms || !tokens || (n_ids > 0 && !ids))
        return fail(RECO_EINVAL, "NULL logits, rewards, uniforms, tokens or ids");
    if (((uintptr_t)logits | (uintptr_t)rewards | (uintptr_t)uniforms | (uintptr_t)tokens) & 3u)
        return fail(RECO_EINVAL, "logits, rewards, uniforms and tokens must be 4-byte aligned");
    if (B > 65535) return fail(RECO_EUNSUPPORTED, "B = %d exceeds 65535", B);
    if (V > reco::kSampleSeg * reco::kSampleMaxSeg)
        return fail(RECO_EUNSUPPORTED, "V = %d exceeds %d", V, reco::kSampleSeg * reco::kSampleMaxSeg);
    if (!(beta >= 0.f)) return fail(RECO_EINVAL, "beta must be >= 0");
    const size_t nseg = (size_t)(V + reco::kSampleSeg - 1) / reco::kSampleSeg;
    reco_status st = check_ws(ws, ws_bytes, (size_t)B * nseg * 8);
    if (st != RECO_OK) return st;
    if ((uintptr_t)ws & 7u) return fail(RECO_EINVAL, "workspace must be 8-byte aligned");
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_penalty_sample(logits, B, V, ids, n_ids, rewards, tau_l, tau_h, beta, uniforms, tokens,
                                                beta_out, (float2 *)ws, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_penalty_sample launch");
}

reco_status reco_answer_ppl(const float *logits, const int32_t *tokens, const int32_t *n_valid, int B, int n, int V,
                            float tau_p, float *ppl, uint8_t *stop, void *ws, size_t ws_bytes, cudaStream_t stream)
{
    if (B < 1 || n < 0 || V < 1) return fail(RECO_EINVAL, "need B >= 1, n >= 0, V >= 1");
    if (B > 65535 || n > 65535) return fail(RECO_EUNSUPPORTED, "B or n exceeds 65535");
    if (!ppl || !stop || (n > 0 && (!logits || !tokens))) return fail(RECO_EINVAL, "NULL logits, tokens, ppl or stop");
    if (((uintptr_t)logits & 3u)) return fail(RECO_EINVAL, "logits must be 4-byte aligned");
    reco_status st = check_ws(ws, ws_bytes, reco::align256((size_t)B * n * 4));
    if (st != RECO_OK) return st;
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_ppl(logits, tokens, n_valid, B, n, V, tau_p, ppl, stop, (float *)ws, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_answer_ppl launch");
}

}  // extern "C"

// ---------------------------------------------------------------- allocation-free answer PPL
// Some callers cannot hand the library any device memory of their own: a plug-in
// running inside a host engine that has already reserved every byte of the GPU for
// its own pool, or plain C code that has no device allocator to call.  For them the
// answer-PPL step can run on a fixed scratch array that lives in the library itself
// (one float per answer row), so the caller passes only its inputs and outputs.
// The array is part of the loaded module: every GPU that loads the library holds its
// 256 KB until the process exits.
static __device__ __align__(256) float g_ppl_static_rows[RECO_PPL_STATIC_MAX_ROWS];

namespace {
float *g_ppl_static_addr[128];

// Device address of g_ppl_static_rows on the current device, looked up once per device
// (the host-side name of the array is not a device address).
reco_status ppl_static_scratch(float **out)
{
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetDevice");
    if (dev < 0 || dev >= 128) return fail(RECO_EUNSUPPORTED, "device index %d out of range", dev);
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_ppl_static_addr[dev]) {
        float *p = nullptr;
        e = cudaGetSymbolAddress((void **)&p, g_ppl_static_rows);
        if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(static PPL scratch)");
        g_ppl_static_addr[dev] = p;
    }
    *out = g_ppl_static_addr[dev];
    return RECO_OK;
}
}  // namespace

extern "C" reco_status reco_answer_ppl_static(const float *logits, const int32_t *tokens, const int32_t *n_valid,
                                              int B, int n, int V, float tau_p, float *ppl, uint8_t *stop,
                                              cudaStream_t stream)
{
    if (B < 1 || n < 0 || V < 1) return fail(RECO_EINVAL, "need B >= 1, n >= 0, V >= 1");
    if (B > 65535 || n > 65535) return fail(RECO_EUNSUPPORTED, "B or n exceeds 65535");
    if ((long long)B * n > RECO_PPL_STATIC_MAX_ROWS)
        return fail(RECO_EINVAL, "B*n = %lld answer rows exceed the static scratch of %d rows", (long long)B * n,
                    RECO_PPL_STATIC_MAX_ROWS);
    if (!ppl || !stop || (n > 0 && (!logits || !tokens))) return fail(RECO_EINVAL, "NULL logits, tokens, ppl or stop");
    if (((uintptr_t)logits & 3u)) return fail(RECO_EINVAL, "logits must be 4-byte aligned");
    float *scratch;
    reco_status st = ppl_static_scratch(&scratch);
    if (st != RECO_OK) return st;
    unsigned *err;
    if ((st = error_word(&err)) != RECO_OK) return st;
    cudaError_t e = reco::launch_ppl(logits, tokens, n_valid, B, n, V, tau_p, ppl, stop, scratch, err, stream);
    return e == cudaSuccess ? RECO_OK : cuda_fail(e, "reco_answer_ppl_static launch");
}
