/*
 * reco.h -- C ABI of libreco, the GB300 (sm_103a) library for the data-parallel
 * hot path of ReCo, "Fewer Tokens, Smaller Cache: Reward-Coordinated Efficient
 * Reasoning": reward-set retention (Eq. 1), attention-guided cache scoring
 * (Eq. 2), per-head top-m selection with in-place compaction (Sec. 3.2), decode
 * attention over the ragged compacted cache, the reward-banded reflection
 * penalty (Eq. 3-4) with the draw of the next token from the penalised logits
 * (Sec. 3.3), and the answer-perplexity stop test (Eq. 5-6).
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Pointers are DEVICE pointers owned by the caller unless marked "host".
 *    The library never allocates device memory: calls that need scratch take a
 *    caller-owned workspace sized by reco_workspace_bytes() (the decode's must
 *    be zero-filled before its first use; each call leaves it reusable), except
 *    reco_answer_ppl_static, which uses a fixed array inside the library.
 *  - Device calls are asynchronous on the given stream and return after the
 *    launches are queued.  They return RECO_OK, or an error status before
 *    launching anything when a host-side check fails (nothing is modified then).
 *  - Problems only visible on the device (a length outside its range, an id or
 *    token outside [0, V)) never make a kernel read or write out of bounds: the
 *    affected unit is skipped and a sticky device error word is set.
 *    reco_check() synchronises the stream, returns RECO_EDEVICE if the word is
 *    set, and clears it.
 *  - reco_last_error() returns the calling thread's last error message.
 *  - Nothing throws across this ABI.
 *
 * Cache layout (struct reco_kv): K and V are separate contiguous arrays of shape
 * [n_layers][B][H_kv][L_cap][d], one row of d elements per cached token, rows of
 * one (layer, sequence, KV head) "unit" contiguous.  lens[n_layers][B][H_kv]
 * (int32, device) holds each unit's current length; rows >= lens are unused and
 * never read.  Query head hq belongs to KV head hq / G with G = H_q / H_kv.
 */
#ifndef RECO_H
#define RECO_H

#include <stddef.h>
#include <stdint.h>
#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    RECO_OK = 0,
    RECO_EINVAL = 1,       /* bad argument (checked on the host, before any launch) */
    RECO_EUNSUPPORTED = 2, /* valid but not implemented (e.g. head_dim not 64 or 128) */
    RECO_ECUDA = 3,        /* a CUDA runtime call failed */
    RECO_EDEVICE = 4       /* the device error word was set by an earlier kernel */
} reco_status;

typedef enum { RECO_F32 = 0, RECO_BF16 = 1 } reco_dtype;

typedef struct {
    void *k;          /* device, [n_layers][B][H_kv][L_cap][d], dtype */
    void *v;          /* device, same shape and dtype as k */
    int n_layers;     /* >= 1 */
    int B;            /* sequences, >= 1 */
    int H_q;          /* query heads, a multiple of H_kv */
    int H_kv;         /* KV heads, >= 1 */
    int L_cap;        /* rows allocated per unit, >= 1 */
    int d;            /* head dimension: 64 or 128 */
    reco_dtype dtype; /* RECO_F32 or RECO_BF16 */
} reco_kv;

typedef enum {
    RECO_OP_SCORE = 0,
    RECO_OP_SELECT = 1,
    RECO_OP_DECODE = 2,
    RECO_OP_PPL = 3,
    RECO_OP_SAMPLE = 4
} reco_op;

/* ---------------------------------------------------------------- host helpers */

/* Eq. 1 (Sec. 3.2): lambda_i = base - delta * (v_i - mean) / (v_max - v_min),
 * the statistics taken over rewards[0..n-1] (host, float32, step order, the
 * last entry being the current step's v_i).  When v_max == v_min the adjustment
 * is 0.  Computed in double.  RECO_EINVAL if n < 1 or a pointer is NULL.       */
reco_status reco_retention_ratio(const float *rewards, int n, double base, double delta,
                                 double *ratio_out);

/* m_i = lambda_i * L (Sec. 3.2): floor(ratio * L) clamped to [w, L].  m counts the
 * w window tokens that are always kept.  RECO_EINVAL unless 1 <= w <= L.       */
reco_status reco_keep_count(double ratio, int L, int w, int32_t *m_out);

/* Eq. 3 band of reward v: 0 (v <= tau_l), 1 (tau_l < v < tau_h), 2 (v >= tau_h);
 * the penalty is 0, beta/2, beta.  float32 comparisons.                       */
int reco_penalty_band(float v, float tau_l, float tau_h);

/* Sec. 3.3 early-stop probe: 1 when v_prev >= tau_h and v_cur >= tau_h.       */
int reco_probe_trigger(float v_prev, float v_cur, float tau_h);

/* Workspace bytes the device call `op` needs for this cache shape (and window w
 * for RECO_OP_SCORE, answer batch B*n passed in `w` for RECO_OP_PPL).  For
 * RECO_OP_SAMPLE, kv is NULL, `w` is the vocabulary size V and the result is the
 * size per sequence (reco_penalty_sample needs B times it).  The size does not
 * depend on the device or on lens.  Alignment: 256 bytes.                      */
reco_status reco_workspace_bytes(reco_op op, const reco_kv *kv, int w, size_t *bytes_out);

/* Thread-local message describing the last non-OK status ("" if none).        */
const char *reco_last_error(void);

/* Synchronise `stream`; RECO_EDEVICE (and clear) if a kernel set the device
 * error word, RECO_ECUDA if the stream reported a CUDA error.                  */
reco_status reco_check(cudaStream_t stream);

/* ---------------------------------------------------------------- device calls */

/* Eq. 2 (Sec. 3.2, attention-guided selection) for the units of the cache.
 * For unit (layer, b, h) of length L = lens[unit] and window w:
 *   logit[g,t,j] = scale * q_win[layer,b,h*G+g,t,:] . K[unit, j, :]
 *   window query t sits at position L-w+t and sees keys j <= L-w+t (causal);
 *   raw[j]  = (1/G) * sum_g sum_t softmax_j(logit[g,t,:])
 *   scores[unit, j] = max(raw[i] : |i-j| <= pool_kernel/2, 0 <= i < L-w)
 * for the candidates j in [0, L-w); entries j >= L-w are left unchanged.
 *   q_win  : [n_layers][B][H_q][w][d], same dtype as the cache (device)
 *   lens   : [n_layers][B][H_kv] int32 (device), w <= lens <= L_cap
 *   keep   : [B] int32 (device) or NULL.  NULL scores every unit.  Given (the keep
 *            counts the following reco_select_compact call receives), a unit with
 *            keep[b] >= L is skipped: a sequence that is not compressed this time
 *            (keep == L, the selection's no-op) costs no key reads, and its rows of
 *            scores are left unchanged.  Sequences reach step boundaries at
 *            different tokens (Sec. 3.1), so most calls compress few of them.
 *   scores : [n_layers][B][H_kv][L_cap] float32 (device, written)
 *   pool_kernel: odd, >= 1 (1 = Eq. 2 as printed); scale: e.g. 1/sqrt(d)
 *   ws     : workspace of reco_workspace_bytes(RECO_OP_SCORE, kv, w) bytes
 * A unit with lens outside [w, L_cap] is skipped (device error word set).     */
reco_status reco_score_cache(const reco_kv *kv, const void *q_win, const int32_t *lens, const int32_t *keep,
                             int w, int pool_kernel, float scale, float *scores, void *ws, size_t ws_bytes,
                             cudaStream_t stream);

/* Eq. 2 as reco_score_cache computes it, with the row normalisers of the window
 * queries taken from the decode instead of from a first pass over the keys.  In
 * Eq. 2 each window row is softmax_j over the keys its query may see; when the
 * window queries are the queries of the last w decoded tokens (Sec. 3.2, the
 * observation window), window query t of unit (layer, b, h) is the query of the
 * token at position L-w+t, and when that token was decoded the cache held exactly
 * its keys j <= L-w+t.  The log-sum-exp reco_decode_attn returned for that query
 * is then the row's log normaliser, so only one pass over K remains.
 *   row_lse: [w][n_layers][B][H_q] float32 (device): row_lse[t][layer][b][hq] =
 *            log sum_{j <= L-w+t} exp(scale * q_win[layer,b,hq,t,:] . K[unit,j,:])
 *            (natural log; the lse output of the reco_decode_attn call that
 *            appended the token at position L-w+t, same scale).  The caller
 *            vouches for that correspondence: no compression of the unit between
 *            those decodes and this call.  A non-finite entry sets the device
 *            error word; that row then adds nothing to the scores.
 * Every candidate key (j < L-w) precedes the whole window, so each row's term of
 * Eq. 2 needs only its query and its normaliser: the window rows may come in any
 * order, as long as q_win row t and row_lse row t belong to the same token.
 * Every other argument, the result and the workspace are those of
 * reco_score_cache.                                                             */
reco_status reco_score_cache_lse(const reco_kv *kv, const void *q_win, const int32_t *lens, const int32_t *keep,
                                 const float *row_lse, int w, int pool_kernel, float scale, float *scores, void *ws,
                                 size_t ws_bytes, cudaStream_t stream);

/* Keeps the decode's log-sum-exps of the last tokens on the device for
 * reco_score_cache_lse (Sec. 3.2's observation window): copies lse[0:n] into rows
 * *slot and *slot + slots of ring and advances *slot to (*slot + 1) % slots, all on
 * the device, so a captured graph can push every token.  The second half of the ring
 * mirrors the first, so the rows of the last w <= slots pushes are one contiguous
 * [w][n] array: ring[s0 .. s0 + w - 1] with s0 = (*slot - w) mod slots, which is
 * reco_score_cache_lse's row_lse when lse is the decode's output for each token.
 *   lse  : [n] float32 (device), e.g. the lse output of reco_decode_attn (n =
 *          n_layers * B * H_q)
 *   ring : [2 * slots][n] float32 (device, two rows written)
 *   slot : int64 (device, read and advanced); a value outside [0, slots) writes
 *          nothing and sets the device error word.                              */
reco_status reco_lse_push(const float *lse, int64_t n, float *ring, int slots, int64_t *slot, cudaStream_t stream);

/* Step-loop utility, not a step of the method: copies row *index of src, a
 * [rows][row_bytes] device array, into dst, with the row chosen on the device, so a
 * captured graph copies a different row on every replay (e.g. the next token's inputs
 * from a pool, selected by the same counter the decode advances).
 *   src   : [rows][row_bytes] (device, 16-byte aligned), row_bytes a multiple of 16
 *   index : int64 (device, read only); a value outside [0, rows) copies nothing and
 *           sets the device error word
 *   dst   : [row_bytes] (device, 16-byte aligned, written)                        */
reco_status reco_copy_row(const void *src, int64_t rows, int64_t row_bytes, const int64_t *index, void *dst,
                          cudaStream_t stream);

/* Top-m selection and in-place compaction (Sec. 3.2: keep the m_i best tokens,
 * the latest w always retained; compress the L cached tokens down to m_i).
 * For unit (layer, b, h) with L = lens[unit] and m = keep[b]:
 *   kept = the m-w candidates j < L-w with the largest scores[unit, j] (float32
 *          order; equal scores keep the lower index) followed by L-w .. L-1,
 *          in ascending order;
 *   K[unit, r] = K[unit, kept[r]] and V[unit, r] = V[unit, kept[r]] for r < m
 *          (in place, row order preserved); lens[unit] = m.
 *   keep     : [B] int32 (device), w <= keep[b] <= lens (m == L is a no-op)
 *   kept_idx : [n_layers][B][H_kv][L_cap] int32 (device) or NULL; if given, the
 *              first m entries of each unit receive `kept`
 *   ws       : workspace of reco_workspace_bytes(RECO_OP_SELECT, kv, w) bytes
 * A unit with an out-of-range length or keep count is left untouched (device
 * error word set).                                                             */
reco_status reco_select_compact(const reco_kv *kv, const float *scores, int32_t *lens,
                                const int32_t *keep, int w, int32_t *kept_idx, void *ws,
                                size_t ws_bytes, cudaStream_t stream);

/* The two halves of reco_select_compact as separate calls, for callers that want the
 * kept indices before the cache moves (for example to compact per-token state of their
 * own with the same indices) or that time the two steps apart.
 * reco_select_topm writes exactly the `kept` that reco_select_compact computes (Sec. 3.2:
 * the m-w best candidates, ties to the lower index, then the window, ascending) into the
 * first keep[b] entries of each unit of kept_idx, and changes nothing else: K, V and lens
 * are left as they are.
 *   scores, lens, keep, w : as reco_select_compact (lens is only read)
 *   kept_idx : [n_layers][B][H_kv][L_cap] int32 (device, written; required)
 *   ws       : workspace of reco_workspace_bytes(RECO_OP_SELECT, kv, w) bytes
 * A unit with an out-of-range length or keep count gets no indices (device error word
 * set).  The kv pointers may be NULL: the cache is not touched.                     */
reco_status reco_select_topm(const reco_kv *kv, const float *scores, const int32_t *lens, const int32_t *keep,
                             int w, int32_t *kept_idx, void *ws, size_t ws_bytes, cudaStream_t stream);

/* In-place compaction of every unit to the rows kept_idx names (Sec. 3.2, the cache
 * compressed from L to m_i tokens): with L = lens[unit] and m = keep[b],
 *   K[unit, r] = K[unit, kept_idx[unit, r]] and V likewise for r < m, lens[unit] = m,
 * for each unit with w <= m < L; m == L leaves the unit as it is.  No workspace.
 *   kept_idx : [n_layers][B][H_kv][L_cap] int32 (device), e.g. from reco_select_topm.
 *              Entry r must lie in [r, L): any strictly increasing list of rows below L
 *              qualifies.  Row r's source is then never a row an earlier destination
 *              overwrote, so the copy in place is exact.  An entry outside [r, L) is not
 *              copied and sets the device error word.
 *   lens     : [n_layers][B][H_kv] int32 (device, in: L, out: m)
 *   keep     : [B] int32 (device)
 * A unit with lens outside [w, L_cap] or keep outside [w, lens] is left untouched (device
 * error word set).                                                                   */
reco_status reco_compact(const reco_kv *kv, const int32_t *kept_idx, int32_t *lens, const int32_t *keep, int w,
                         cudaStream_t stream);

/* Decode attention over the ragged compacted cache: the per-token attention whose
 * cost the compression lowers (Sec. 1; Sec. 2.2; Sec. 4.2, main results).
 * If k_new and v_new are both non-NULL, each unit first appends its new row at
 * index lens[unit] (which must be < L_cap) and the length grows by one; lens is
 * updated when the kernel finishes.  Then for every query head hq of unit u:
 *   out[layer,b,hq,:] = softmax_j(scale * q[layer,b,hq,:] . K[u,j,:]) V[u,j,:],
 *   j over the unit's rows, lse[layer,b,hq] = natural log of the softmax sum.
 *   q            : [n_layers][B][H_q][d], cache dtype (device)
 *   k_new, v_new : [n_layers][B][H_kv][d], cache dtype (device) or both NULL
 *   out          : [n_layers][B][H_q][d] of out_dtype (RECO_F32 or RECO_BF16)
 *   lse          : [n_layers][B][H_q] float32 or NULL
 *   ws           : workspace of reco_workspace_bytes(RECO_OP_DECODE, kv, 0) bytes,
 *                  zero-filled before its first use (e.g. cudaMemset); every call
 *                  leaves its counters zero again, so it can be reused as it is;
 *                  calls sharing one workspace must not overlap on the GPU
 * A unit with a length outside [0, L_cap] (or no room to append) writes zeros
 * and lse = -inf, and sets the device error word.                              */
reco_status reco_decode_attn(const reco_kv *kv, const void *q, const void *k_new, const void *v_new,
                             int32_t *lens, float scale, void *out, reco_dtype out_dtype, float *lse,
                             void *ws, size_t ws_bytes, cudaStream_t stream);

/* reco_decode_attn whose log-sum-exps go into the device ring that
 * reco_score_cache_lse reads (Sec. 3.2's observation window: the lse of the last
 * decoded tokens are the row normalisers of Eq. 2), instead of an lse array: the launch
 * writes lse[layer,b,hq] into rows *slot and *slot + slots of ring and then advances
 * *slot to (*slot + 1) % slots, all on the device, so a captured graph decodes every
 * token with no separate push.  It is reco_decode_attn followed by reco_lse_push in one
 * launch, with the same results.
 *   ring   : [2 * slots][n_layers * B * H_q] float32 (device, two rows written)
 *   slot   : int64 (device, read and advanced); a value outside [0, slots) writes no
 *            ring row, leaves *slot as it is and sets the device error word
 *   q_ring : [n_layers][B][H_q][slots][d], the cache dtype, 16-byte aligned (device),
 *            or NULL: row *slot of every query head's `slots` rows receives that
 *            head's query.  With slots = w it then holds the queries of the last w
 *            tokens in slot order (token t in slot t mod w), the same order as ring
 *            rows 0..w-1: together the q_win and row_lse of reco_score_cache_lse, with
 *            no gather (its result does not depend on the order of the window rows).
 * Every other argument, the result and the workspace are those of reco_decode_attn.    */
reco_status reco_decode_attn_ring(const reco_kv *kv, const void *q, const void *k_new, const void *v_new,
                                  int32_t *lens, float scale, void *out, reco_dtype out_dtype, float *ring,
                                  int slots, int64_t *slot, void *q_ring, void *ws, size_t ws_bytes,
                                  cudaStream_t stream);

/* Eq. 3 + Eq. 4 (Sec. 3.3, reward-banded reflection penalty), in place:
 *   beta_b = 0, beta/2 or beta by the band of rewards[b] (float32 compares);
 *   logits[b, u] -= beta_b once for each distinct id u in ids[0..n_ids-1];
 *   all other logits are left bit-for-bit unchanged.
 *   logits  : [B][V] float32 (device, in/out)
 *   ids     : [n_ids] int32 (device); ids outside [0, V) are skipped and set the
 *             device error word
 *   rewards : [B] float32 (device), the just-completed step's v_i per sequence
 *   beta_out: [B] float32 (device) or NULL, receives beta_b                     */
reco_status reco_reflect_penalty(float *logits, int B, int V, const int32_t *ids, int n_ids,
                                 const float *rewards, float tau_l, float tau_h, float beta,
                                 float *beta_out, cudaStream_t stream);

/* Eq. 3 + Eq. 4 in place, then one draw per sequence from softmax of the penalised
 * logits (Sec. 3.3: while the next step is generated its tokens are sampled from
 * softmax of the penalised logits, temperature 1), by inversion of the distribution
 * in token order at a draw the caller supplies:
 *   p         = softmax(logits[b, :]) after the penalty,
 *   tokens[b] = the smallest j with p_j > 0 and sum_{i<=j} p_i > uniforms[b];
 * if rounding leaves no such j (a draw at the top of [0, 1), or NaN), the last j with
 * p_j > 0; a row whose logits are all -inf gets -1.  Logits must be finite or -inf.
 *   logits, ids, n_ids, rewards, tau_l, tau_h, beta, beta_out : as reco_reflect_penalty
 *            (the logits are penalised in place exactly as reco_reflect_penalty does)
 *   uniforms : [B] float32 (device), one draw in [0, 1) per sequence
 *   tokens   : [B] int32 (device, written)
 *   ws       : at least B * reco_workspace_bytes(RECO_OP_SAMPLE, NULL, V) bytes (not
 *              touched when logits are 16-byte aligned, V is a multiple of 4 and
 *              V <= 393216: then one launch with a cluster of CTAs per row does all)
 * V may be at most 4194304.  The probabilities are float32 (2^x on the special-
 * function unit), so a draw within about 1e-5 of a boundary of the cumulative
 * distribution may select the neighbouring token.                              */
reco_status reco_penalty_sample(float *logits, int B, int V, const int32_t *ids, int n_ids, const float *rewards,
                                float tau_l, float tau_h, float beta, const float *uniforms, int32_t *tokens,
                                float *beta_out, void *ws, size_t ws_bytes, cudaStream_t stream);

/* Eq. 5 + Eq. 6 (Sec. 3.3, early stopping via answer confidence):
 *   lp[b,t] = logits[b,t,tokens[b,t]] - logsumexp(logits[b,t,:])   (natural log)
 *   ppl[b]  = exp(-(1/n_b) sum_{t < n_b} lp[b,t]),  stop[b] = ppl[b] <= tau_p
 * with n_b = n_valid[b] (clamped to n) or n when n_valid is NULL; n_b == 0 gives
 * ppl = NaN and stop = 0.  Raw logits, no penalty, temperature 1.
 *   logits : [B][n][V] float32 (device); tokens : [B][n] int32 (device)
 *   ppl    : [B] float32 (device, written); stop : [B] uint8 (device, written)
 *   ws     : workspace of reco_workspace_bytes(RECO_OP_PPL, NULL, B*n) bytes
 * A token outside [0, V) makes that sequence's ppl NaN and stop 0 and sets the
 * device error word.                                                           */
reco_status reco_answer_ppl(const float *logits, const int32_t *tokens, const int32_t *n_valid, int B,
                            int n, int V, float tau_p, float *ppl, uint8_t *stop, void *ws,
                            size_t ws_bytes, cudaStream_t stream);

/* Allocation-free variant of reco_answer_ppl (the paper has no counterpart: this is
 * a library convenience).  Same arguments and results as reco_answer_ppl, but the
 * per-row scratch is a fixed array inside the library instead of a caller workspace,
 * for callers that cannot allocate device memory (for example a plug-in whose host
 * engine has reserved the whole GPU, or C code with no device allocator).
 *   - B*n must not exceed RECO_PPL_STATIC_MAX_ROWS, else RECO_EINVAL (nothing runs).
 *   - Allocates nothing: no cudaMalloc / cudaFree, no allocating library routine.
 *   - The first call on each device looks up the array's device address (once, with
 *     that device current); make that first call before any stream capture.
 *   - All calls on a device share the one array and it keeps the last call's
 *     contents; every entry a call reads is written by that call first, so nothing
 *     needs clearing, but calls whose executions overlap on the GPU race on it.
 *   - Every GPU that loads the library holds the array (256 KB) until process exit. */
#define RECO_PPL_STATIC_MAX_ROWS 65536
reco_status reco_answer_ppl_static(const float *logits, const int32_t *tokens, const int32_t *n_valid, int B,
                                   int n, int V, float tau_p, float *ppl, uint8_t *stop, cudaStream_t stream);

#ifdef __cplusplus
}
#endif

#endif /* RECO_H */
