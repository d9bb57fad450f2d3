/*
 * reco_oracle.c -- plain, slow, fp64 CPU oracle for the ReCo hot path
 * ("Fewer Tokens, Smaller Cache: Reward-Coordinated Efficient Reasoning").
 *
 * TEST INFRASTRUCTURE ONLY.  This file is the independent definition that the
 * CUDA library is checked against.  Only the test suite, the smoke check and the
 * benchmark's CPU-baseline / reference arm may load it.  It shares no code,
 * header, table or constant with the CUDA library, and the library never calls it.
 *
 * Every function is the paper's definition written out with explicit loops in
 * double precision.  Inputs arrive as float32 arrays (bf16 inputs are widened to
 * float32 exactly by the caller, then to double here).  Nothing is blocked, fused
 * or reordered beyond what the definition states.  The only parallelism is an
 * OpenMP loop over independent (layer, sequence, KV-head) units in the batched
 * wrappers; each unit is computed by the same serial code.
 *
 * Readings of points the paper leaves open:
 *   - Eq. 1 with v_max == v_min (one reward, or all equal): the adjustment is 0.
 *   - Eq. 1 statistics run over all step rewards v_1..v_i, the current one included.
 *   - keep count m = clamp(floor(lambda_i * L), w, L); m counts the window.
 *   - Eq. 2 logits carry the attention scale (default 1/sqrt(d)); window query t
 *     (t = 0..w-1) sits at cache position L-w+t and sees keys j <= L-w+t.
 *   - GQA: KV head h serves query heads h*G .. h*G+G-1; the score is the mean
 *     over those G heads of the per-head window sums.
 *   - Max-pool (kernel k, odd, stride 1) over the candidate range [0, L-w), the
 *     window [j-k/2, j+k/2] clipped to that range; k = 1 is Eq. 2 unchanged.
 *   - Top-m: m-w candidates with the largest pooled score, ties to the lower
 *     index, plus the w window tokens; indices ascending.  The ranking compares
 *     float32 scores (the precision the kernel decides in).
 *   - Eq. 3 bands compare float32 rewards with float32 thresholds.
 *   - Eq. 4 subtracts the band penalty once per distinct id of R.
 *   - Sampling after Eq. 4: temperature 1, one draw per row by inversion of the
 *     CDF in token-index order at a uniform draw the caller supplies.
 *   - Eq. 5 uses raw logits, natural log; an empty answer has PPL = NaN, no stop.
 *   - Early-stop probe: v_{i-1} >= tau_h and v_i >= tau_h.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Timing plumbing, no arithmetic: the number of threads the OpenMP loops of the
 * batched wrappers use (the benchmark times the oracle on one core and on all). */
void oracle_set_threads(int n)
{
#ifdef _OPENMP
    omp_set_num_threads(n > 0 ? n : 1);
#else
    (void)n;
#endif
}

int oracle_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

/* ------------------------------------------------------------------------- */
/* Eq. 1 (Sec. 3.2, "Reward-driven retention"): lambda_i = lambda - delta *   */
/* (v_i - mean) / (v_max - v_min), statistics over the trajectory's rewards.  */
/* rewards[0..n-1] are v_1..v_i in step order; rewards[n-1] is v_i.          */
/* ------------------------------------------------------------------------- */
double oracle_retention_ratio(const float *rewards, int n, double base, double delta)
{
    if (n < 1) return NAN;
    double sum = 0.0;
    double vmin = (double)rewards[0];
    double vmax = (double)rewards[0];
    for (int s = 0; s < n; ++s) {
        double v = (double)rewards[s];
        sum += v;
        if (v < vmin) vmin = v;
        if (v > vmax) vmax = v;
    }
    double mean = sum / (double)n;
    double range = vmax - vmin;
    if (range == 0.0) return base; /* 0/0: no adjustment (reading) */
    double vi = (double)rewards[n - 1];
    return base - delta * ((vi - mean) / range);
}

/* m_i = lambda_i * L (Sec. 3.2), floored and clamped to [w, L]. */
int oracle_keep_count(double ratio, int L, int w)
{
    double x = floor(ratio * (double)L);
    long m = (long)x;
    if (x < (double)w) m = w;
    if (x > (double)L) m = L;
    return (int)m;
}

/* ------------------------------------------------------------------------- */
/* Eq. 2 (Sec. 3.2, "Attention-guided selection") for one KV head.            */
/*   q   : [G][w][d]  window queries of the G query heads of this KV head     */
/*   k   : [L][d]     cached keys (row pitch d)                               */
/*   raw : [L]        (1/G) sum_g sum_t softmax_j(scale * q_{g,t} . k_j)      */
/*   pooled : [L-w]   max-pool of raw over the candidate range (may be NULL)  */
/* ------------------------------------------------------------------------- */
void oracle_score_unit(const float *q, const float *k, int G, int w, int L, int d,
                       double scale, int pool, double *raw, double *pooled)
{
    double *logit = (double *)malloc(sizeof(double) * (size_t)(L > 0 ? L : 1));
    double *acc = (double *)calloc((size_t)(L > 0 ? L : 1), sizeof(double));
    for (int g = 0; g < G; ++g) {
        for (int t = 0; t < w; ++t) {
            const float *qr = q + ((size_t)g * w + t) * d;
            int visible = L - w + t + 1; /* keys 0 .. L-w+t */
            double mx = -INFINITY;
            for (int j = 0; j < visible; ++j) {
                double dot = 0.0;
                for (int c = 0; c < d; ++c) dot += (double)qr[c] * (double)k[(size_t)j * d + c];
                logit[j] = scale * dot;
                if (logit[j] > mx) mx = logit[j];
            }
            double Z = 0.0;
            for (int j = 0; j < visible; ++j) Z += exp(logit[j] - mx);
            for (int j = 0; j < visible; ++j) acc[j] += exp(logit[j] - mx) / Z;
        }
    }
    for (int j = 0; j < L; ++j) raw[j] = acc[j] / (double)G;
    if (pooled) {
        int nc = L - w;
        int half = pool / 2;
        for (int j = 0; j < nc; ++j) {
            int lo = j - half < 0 ? 0 : j - half;
            int hi = j + half > nc - 1 ? nc - 1 : j + half;
            double mx = -INFINITY;
            for (int i = lo; i <= hi; ++i)
                if (raw[i] > mx) mx = raw[i];
            pooled[j] = mx;
        }
    }
    free(logit);
    free(acc);
}

/* Batched Eq. 2 over every (layer, sequence, KV head).
 *   q_win  : [Ly][B][Hq][w][d]      K : [Ly][B][Hkv][Lcap][d]
 *   lens   : [Ly][B][Hkv]           scores_out : [Ly][B][Hkv][Lcap], pooled
 *   candidates in [0, len-w), the rest left untouched.                       */
void oracle_score_cache(const float *q_win, const float *K, const int32_t *lens,
                        int Ly, int B, int Hq, int Hkv, int Lcap, int d, int w,
                        int pool, double scale, double *scores_out)
{
    int G = Hq / Hkv;
    long units = (long)Ly * B * Hkv;
#pragma omp parallel for schedule(dynamic, 1)
    for (long u = 0; u < units; ++u) {
        int h = (int)(u % Hkv);
        long lb = u / Hkv; /* layer*B + b */
        int L = lens[u];
        const float *q = q_win + ((size_t)lb * Hq + (size_t)h * G) * w * d;
        const float *k = K + (size_t)u * Lcap * d;
        double *raw = (double *)malloc(sizeof(double) * (size_t)L);
        oracle_score_unit(q, k, G, w, L, d, scale, pool, raw, scores_out + (size_t)u * Lcap);
        free(raw);
    }
}

/* ------------------------------------------------------------------------- */
/* Top-m selection (Sec. 3.2): keep the m-w best candidates in [0, L-w) by     */
/* float32 score, ties to the lower index, then the w window tokens.          */
/* Writes m ascending indices to idx.  Returns m, or -1 on bad sizes.         */
/* ------------------------------------------------------------------------- */
static const float *g_sort_scores;
static int cmp_desc_then_index(const void *a, const void *b)
{
    int i = *(const int *)a, j = *(const int *)b;
    float si = g_sort_scores[i], sj = g_sort_scores[j];
    if (si > sj) return -1;
    if (si < sj) return 1;
    return (i < j) ? -1 : (i > j);
}

int oracle_select_unit(const float *scores, int L, int w, int m, int32_t *idx)
{
    if (w < 1 || L < w || m < w || m > L) return -1;
    int nc = L - w, kc = m - w;
    int *order = (int *)malloc(sizeof(int) * (size_t)(nc > 0 ? nc : 1));
    char *kept = (char *)calloc((size_t)(nc > 0 ? nc : 1), 1);
    for (int j = 0; j < nc; ++j) order[j] = j;
    g_sort_scores = scores; /* single-threaded use only (see batched wrapper) */
    qsort(order, (size_t)nc, sizeof(int), cmp_desc_then_index);
    for (int r = 0; r < kc; ++r) kept[order[r]] = 1;
    int c = 0;
    for (int j = 0; j < nc; ++j)
        if (kept[j]) idx[c++] = j;
    for (int t = 0; t < w; ++t) idx[c++] = nc + t;
    free(order);
    free(kept);
    return c;
}

/* Batched selection: scores [units][Lcap] (pooled, float32), keep[b] per
 * sequence, idx_out [units][Lcap] (first m entries written).  Serial, because
 * qsort's comparator reads one shared score pointer.                          */
void oracle_select_batch(const float *scores, const int32_t *lens, const int32_t *keep,
                         int Ly, int B, int Hkv, int Lcap, int w, int32_t *idx_out)
{
    long units = (long)Ly * B * Hkv;
    for (long u = 0; u < units; ++u) {
        int b = (int)((u / Hkv) % B);
        oracle_select_unit(scores + (size_t)u * Lcap, lens[u], w, keep[b], idx_out + (size_t)u * Lcap);
    }
}

/* Compaction (Sec. 3.2, "compress the L cached tokens down to m_i"):
 * out[r] = in[idx[r]] for r < m, row length d.  Out of place.                */
void oracle_gather_unit(const float *in, const int32_t *idx, int m, int d, float *out)
{
    for (int r = 0; r < m; ++r)
        for (int c = 0; c < d; ++c) out[(size_t)r * d + c] = in[(size_t)idx[r] * d + c];
}

/* ------------------------------------------------------------------------- */
/* Decode attention over the (compacted) cache: the per-token attention whose  */
/* cost compression lowers (Sec. 1, Sec. 2.2, Sec. 4.2).  Textbook softmax     */
/* attention of one query over rows 0..len-1.  Natural-log lse.               */
/* ------------------------------------------------------------------------- */
void oracle_decode_unit(const float *q, const float *k, const float *v, int len, int d,
                        double scale, double *out, double *lse)
{
    if (len <= 0) {
        for (int c = 0; c < d; ++c) out[c] = 0.0;
        if (lse) *lse = -INFINITY;
        return;
    }
    double *logit = (double *)malloc(sizeof(double) * (size_t)len);
    double mx = -INFINITY;
    for (int j = 0; j < len; ++j) {
        double dot = 0.0;
        for (int c = 0; c < d; ++c) dot += (double)q[c] * (double)k[(size_t)j * d + c];
        logit[j] = scale * dot;
        if (logit[j] > mx) mx = logit[j];
    }
    double Z = 0.0;
    for (int j = 0; j < len; ++j) Z += exp(logit[j] - mx);
    for (int c = 0; c < d; ++c) out[c] = 0.0;
    for (int j = 0; j < len; ++j) {
        double p = exp(logit[j] - mx) / Z;
        for (int c = 0; c < d; ++c) out[c] += p * (double)v[(size_t)j * d + c];
    }
    if (lse) *lse = mx + log(Z);
    free(logit);
}

/* Batched decode: q [Ly][B][Hq][d], K/V [Ly][B][Hkv][Lcap][d], lens [units].
 * out [Ly][B][Hq][d] (double), lse [Ly][B][Hq] (double, may be NULL).        */
void oracle_decode_batch(const float *q, const float *K, const float *V, const int32_t *lens,
                         int Ly, int B, int Hq, int Hkv, int Lcap, int d, double scale,
                         double *out, double *lse)
{
    int G = Hq / Hkv;
    long rows = (long)Ly * B * Hq;
#pragma omp parallel for schedule(dynamic, 4)
    for (long r = 0; r < rows; ++r) {
        int hq = (int)(r % Hq);
        long lb = r / Hq;
        long u = lb * Hkv + hq / G;
        oracle_decode_unit(q + (size_t)r * d, K + (size_t)u * Lcap * d, V + (size_t)u * Lcap * d,
                           lens[u], d, scale, out + (size_t)r * d, lse ? lse + r : NULL);
    }
}

/* ------------------------------------------------------------------------- */
/* Eq. 3 (Sec. 3.3): band 0 (v <= tau_l), 1 (tau_l < v < tau_h), 2 (v >= tau_h) */
/* compared in float32.                                                       */
/* ------------------------------------------------------------------------- */
int oracle_penalty_band(float v, float tau_l, float tau_h)
{
    if (v <= tau_l) return 0;
    if (v >= tau_h) return 2;
    return 1;
}

/* Eq. 3 + Eq. 4 in place on logits [B][V]: z(u) -= beta_i once for each
 * distinct u in R.  beta_out[b] receives beta_i (may be NULL).  Ids outside
 * [0, V) are ignored and counted in the return value.                        */
int oracle_reflect_penalty(float *logits, int B, int V, const int32_t *ids, int n_ids,
                           const float *rewards, float tau_l, float tau_h, float beta,
                           float *beta_out)
{
    char *in_R = (char *)calloc((size_t)V, 1);
    int bad = 0;
    for (int i = 0; i < n_ids; ++i) {
        if (ids[i] < 0 || ids[i] >= V) { ++bad; continue; }
        in_R[ids[i]] = 1;
    }
    for (int b = 0; b < B; ++b) {
        int band = oracle_penalty_band(rewards[b], tau_l, tau_h);
        double beta_i = band == 0 ? 0.0 : (band == 1 ? (double)beta / 2.0 : (double)beta);
        if (beta_out) beta_out[b] = (float)beta_i;
        if (beta_i == 0.0) continue;
        for (int u = 0; u < V; ++u)
            if (in_R[u]) {
                size_t o = (size_t)b * V + u;
                logits[o] = (float)((double)logits[o] - beta_i);
            }
    }
    free(in_R);
    return bad;
}

/* ------------------------------------------------------------------------- */
/* Sampling from the penalised logits (Sec. 3.3, after Eq. 4: the next token  */
/* is drawn from softmax(z~), temperature 1).  Eq. 3 + Eq. 4 are applied in    */
/* place first (oracle_reflect_penalty), then each row draws one token by      */
/* inversion: with p = softmax(z~ row) and the given uniform u[b], the token   */
/* is the smallest j with p_j > 0 and sum_{i<=j} p_i > u.  If rounding leaves  */
/* no such j (u at the top of [0, 1)), the last j with p_j > 0 is taken; a row */
/* of -inf logits gets -1.  cdf_lo / cdf_hi (may be NULL) receive             */
/* sum_{i<j} p_i and sum_{i<=j} p_i of the chosen token.  Returns the number  */
/* of ids outside [0, V).                                                      */
/* ------------------------------------------------------------------------- */
int oracle_penalty_sample(float *logits, int B, int V, const int32_t *ids, int n_ids,
                          const float *rewards, float tau_l, float tau_h, float beta,
                          const float *uniforms, int32_t *tokens, double *cdf_lo, double *cdf_hi)
{
    int bad = oracle_reflect_penalty(logits, B, V, ids, n_ids, rewards, tau_l, tau_h, beta, NULL);
    for (int b = 0; b < B; ++b) {
        const float *z = logits + (size_t)b * V;
        double M = -INFINITY;
        for (int j = 0; j < V; ++j)
            if ((double)z[j] > M) M = (double)z[j];
        int tok = -1;
        double lo = 0.0, hi = 0.0;
        if (M != -INFINITY) {
            double Z = 0.0;
            for (int j = 0; j < V; ++j) Z += exp((double)z[j] - M);
            double u = (double)uniforms[b];
            double c = 0.0;
            int last = -1;
            double last_lo = 0.0;
            for (int j = 0; j < V; ++j) {
                double p = exp((double)z[j] - M) / Z;
                double prev = c;
                c += p;
                if (p > 0.0) {
                    last = j;
                    last_lo = prev;
                }
                if (c > u && p > 0.0) {
                    tok = j;
                    lo = prev;
                    hi = c;
                    break;
                }
            }
            if (tok < 0) {
                tok = last;
                lo = last_lo;
                hi = c;
            }
        }
        tokens[b] = tok;
        if (cdf_lo) cdf_lo[b] = lo;
        if (cdf_hi) cdf_hi[b] = hi;
    }
    return bad;
}

/* Early-stop probe trigger (Sec. 3.3): reward in the top band for two
 * consecutive steps.                                                          */
int oracle_probe_trigger(float v_prev, float v_cur, float tau_h)
{
    return (v_prev >= tau_h) && (v_cur >= tau_h);
}

/* ------------------------------------------------------------------------- */
/* Eq. 5 + Eq. 6 (Sec. 3.3): PPL(a) = exp(-(1/n) sum_t log p(x_t | x_<t)),     */
/* stop iff PPL <= tau_p.  logits [B][n][V], tokens [B][n], n_valid [B] or     */
/* NULL (all n).  log p = z[x] - (M + log sum exp(z - M)).                    */
/* ------------------------------------------------------------------------- */
void oracle_answer_ppl(const float *logits, const int32_t *tokens, const int32_t *n_valid,
                       int B, int n, int V, float tau_p, double *ppl, uint8_t *stop)
{
#pragma omp parallel for schedule(static)
    for (int b = 0; b < B; ++b) {
        int nv = n_valid ? n_valid[b] : n;
        if (nv > n) nv = n;
        if (nv <= 0) { ppl[b] = NAN; stop[b] = 0; continue; }
        double sum_lp = 0.0;
        for (int t = 0; t < nv; ++t) {
            const float *z = logits + ((size_t)b * n + t) * V;
            double M = -INFINITY;
            for (int u = 0; u < V; ++u)
                if ((double)z[u] > M) M = (double)z[u];
            double Z = 0.0;
            for (int u = 0; u < V; ++u) Z += exp((double)z[u] - M);
            int x = tokens[(size_t)b * n + t];
            sum_lp += (double)z[x] - (M + log(Z));
        }
        ppl[b] = exp(-sum_lp / (double)nv);
        stop[b] = ppl[b] <= (double)tau_p;
    }
}
