// internal.h -- launcher interface between the C ABI layer (api.cu) and the kernels.
#pragma once
#include <cuda_runtime.h>
#include <stddef.h>
#include <stdint.h>

#include "../../include/reco.h"

namespace reco {

// Keys per scoring work item (one CTA per (unit, chunk) in both scoring passes).
constexpr int kScoreChunk = 2048;
// Decode (m, l, O) partial slots in the workspace: two per warp of a grid of up to
// 256 SMs x 8 warps (the workspace size may not depend on the device; a larger grid
// takes the SIMT path).
constexpr int kDecodePartSlots = 4096;
// Sampling: logits per pass-1 segment, and the most segments a row may have.
constexpr int kSampleSeg = 4096;
constexpr int kSampleMaxSeg = 1024;

inline size_t align256(size_t x) { return (x + 255) & ~size_t(255); }

struct ScoreWs {  // regions carved from the caller's workspace
    float *part_m, *part_z;  // [units][n_chunks][R]  per-chunk row max (log2) / row sum
    float *rowb;             // [units][R]            log2 of the row normaliser
    float *raw;              // [units][L_cap]        unpooled scores
    int32_t *ulist;          // [units]               units to score, ascending (with a keep mask)
    int32_t *ucount;         // [1]                   entries of ulist
    size_t bytes;
};

// Which units a scoring call covers.  With keep == nullptr every unit; otherwise a
// unit whose sequence keeps its whole cache this time (keep[b] >= lens[unit], the
// selection's no-op) is skipped: none of its keys are read and its scores are not
// written.  A unit with an out-of-range length is never skipped, so it still raises
// the length error.
struct ScoreMask {
    const int32_t *keep;  // [B] or nullptr
    int B, Hkv;
#ifdef __CUDACC__
    __device__ __forceinline__ bool skip(long u, int L, int w, int L_cap) const
    {
        return keep != nullptr && L >= w && L <= L_cap && keep[(u / Hkv) % B] >= L;
    }
#endif
};

struct SelectWs {
    int32_t *idx;    // [units][L_cap] kept indices (when the caller passes none)
    int32_t *count;  // [units] rows to compact (0 = skip unit)
    size_t bytes;
};

struct DecodeWs {
    int32_t *counters;  // [2 + units]: [0] a warp stopped early, [1] finished warps, [2 + u] merge tickets
    float *part_ml;     // [part_slots][G][2]  (m log2, l)
    float *part_o;      // [part_slots][G][d]  unnormalised output
    int part_slots;
    size_t bytes;
};

ScoreWs score_ws_layout(const reco_kv &kv, int w, void *base);
SelectWs select_ws_layout(const reco_kv &kv, void *base);
DecodeWs decode_ws_layout(const reco_kv &kv, void *base);

// Launchers return cudaSuccess or the launch error.  All arguments validated by the caller.
cudaError_t launch_score(const reco_kv &kv, const void *q_win, const int32_t *lens, const int32_t *keep, int w,
                         int pool, float scale, float *scores, const ScoreWs &ws, unsigned *err, cudaStream_t s);
cudaError_t launch_score_lse(const reco_kv &kv, const void *q_win, const int32_t *lens, const int32_t *keep,
                             const float *row_lse, int w, int pool, float scale, float *scores, const ScoreWs &ws,
                             unsigned *err, cudaStream_t s);
cudaError_t launch_copy_row(const void *src, long long rows, long long row_bytes, const long long *index, void *dst,
                            unsigned *err, cudaStream_t s);
cudaError_t launch_lse_push(const float *lse, long n, float *ring, int slots, long long *slot, unsigned *err,
                            cudaStream_t s);
cudaError_t launch_select_compact(const reco_kv &kv, const float *scores, int32_t *lens,
                                  const int32_t *keep, int w, int32_t *kept_idx, const SelectWs &ws,
                                  unsigned *err, cudaStream_t s);
cudaError_t launch_select_only(const reco_kv &kv, const float *scores, const int32_t *lens, const int32_t *keep,
                               int w, int32_t *kept_idx, const SelectWs &ws, unsigned *err, cudaStream_t s);
cudaError_t launch_compact(const reco_kv &kv, const int32_t *kept_idx, int32_t *lens, const int32_t *keep, int w,
                           unsigned *err, cudaStream_t s);
// ring: optional [2 * slots][layers * B * H_q] lse ring; the launch writes rows *slot and
// *slot + slots and advances *slot.
cudaError_t launch_decode(const reco_kv &kv, const void *q, const void *k_new, const void *v_new,
                          int32_t *lens, float scale, void *out, reco_dtype out_dtype, float *lse,
                          const DecodeWs &ws, unsigned *err, cudaStream_t s, float *ring = nullptr,
                          int slots = 0, long long *slot = nullptr, void *qring = nullptr);
cudaError_t launch_penalty(float *logits, int B, int V, const int32_t *ids, int n_ids,
                           const float *rewards, float tau_l, float tau_h, float beta, float *beta_out,
                           unsigned *err, cudaStream_t s);
cudaError_t launch_penalty_sample(float *logits, int B, int V, const int32_t *ids, int n_ids, const float *rewards,
                                  float tau_l, float tau_h, float beta, const float *uniforms, int32_t *tokens,
                                  float *beta_out, float2 *part, unsigned *err, cudaStream_t s);
cudaError_t launch_ppl(const float *logits, const int32_t *tokens, const int32_t *n_valid, int B, int n,
                       int V, float tau_p, float *ppl, uint8_t *stop, float *lp_ws, unsigned *err,
                       cudaStream_t s);

// Device properties cached per device.
int device_sm_count();

// Encode a 2-D tensor map over a row-major bf16 matrix [rows, cols] with boxes of
// box_rows x box_cols elements and 128-byte swizzle (box_cols * 2 <= 128).
// Returns false if the driver entry point is unavailable or the encode fails.
bool encode_bf16_2d(void *map /* CUtensorMap */, const void *base, unsigned long long rows, int cols,
                    int box_cols, int box_rows);

}  // namespace reco
