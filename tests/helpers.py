"""Shared helpers for the GPU parity tests: run the CUDA path through the C ABI and
compare with the oracle under the stated tolerances.

Tolerances (fixed by the task's stated bars, restated here):
  scores, PPL        |gpu - oracle| <= 1e-3 * |oracle| + 1e-7 * max_j oracle  (the
                     floor covers tails that underflow in float32)
  kept-index sets    bit-exact, except candidates whose oracle score lies within
                     1e-5 relative of the oracle's (m-w)-th largest candidate score
  compacted rows     bit-exact (pure data movement)
  decode output      1e-4 abs (float32 cache), 2e-2 abs (bf16 cache)
  penalised logits   bit-exact
  stop flags         exact unless |PPL - tau_p| <= 1e-3 * tau_p
"""
from __future__ import annotations

import numpy as np
import torch

import oracle
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

SCORE_RTOL = 1e-3
SCORE_FLOOR = 1e-7
TIE_RTOL = 1e-5
DECODE_ATOL = {"f32": 1e-4, "bf16": 2e-2}
PPL_RTOL = 1e-3


def np32(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy()


def keep_counts(wl: W.Workload, L: int | None = None, ratio: float | None = None):
    """Per-sequence keep counts from the library's host helpers (Eq. 1) and, separately,
    from the oracle; asserts they agree exactly and returns them."""
    hist = W.make_reward_history(wl)
    L = wl.L if L is None else L
    lib_m, ora_m = [], []
    for b in range(wl.batch):
        r_lib = reco.reco_retention_ratio(hist[b], wl.base, wl.delta) if ratio is None else ratio
        r_ora = oracle.retention_ratio(hist[b], wl.base, wl.delta) if ratio is None else ratio
        lib_m.append(reco.reco_keep_count(r_lib, L, wl.w))
        ora_m.append(oracle.keep_count(r_ora, L, wl.w))
    assert lib_m == ora_m
    return np.array(lib_m, np.int32)


def gpu_score(wl, K, V, q_win, lens, pool=None):
    kv = reco.make_kv(K, V, wl.h_q)
    scores = torch.zeros(K.shape[:4], dtype=torch.float32, device=K.device)
    ws = reco.workspace(reco.RECO_OP_SCORE, kv, wl.w, K.device)
    reco.reco_score_cache(kv, q_win, lens, wl.w, wl.pool if pool is None else pool, wl.scale(), scores, ws)
    return scores


def gpu_select(wl, K, V, scores, lens, keep):
    kv = reco.make_kv(K, V, wl.h_q)
    kept = torch.full(K.shape[:4], -1, dtype=torch.int32, device=K.device)
    ws = reco.workspace(reco.RECO_OP_SELECT, kv, wl.w, K.device)
    keep_t = torch.as_tensor(keep, dtype=torch.int32, device=K.device)
    reco.reco_select_compact(kv, scores, lens, keep_t, wl.w, kept, ws)
    return kept


def gpu_select_split(wl, K, V, scores, lens, keep):
    """reco_select_topm, then reco_compact on the indices it wrote (the two halves of
    reco_select_compact as separate calls)."""
    kv = reco.make_kv(K, V, wl.h_q)
    kept = torch.full(K.shape[:4], -1, dtype=torch.int32, device=K.device)
    ws = reco.workspace(reco.RECO_OP_SELECT, kv, wl.w, K.device)
    keep_t = torch.as_tensor(keep, dtype=torch.int32, device=K.device)
    reco.reco_select_topm(kv, scores, lens, keep_t, wl.w, kept, ws)
    reco.reco_compact(kv, kept, lens, keep_t, wl.w)
    return kept


def gpu_decode(wl, K, V, lens, q, k_new=None, v_new=None, out_dtype=torch.float32):
    kv = reco.make_kv(K, V, wl.h_q)
    out = torch.empty(q.shape, dtype=out_dtype, device=q.device)
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device=q.device)
    ws = reco.workspace(reco.RECO_OP_DECODE, kv, 0, q.device)
    reco.reco_decode_attn(kv, q, k_new, v_new, lens, wl.scale(), out, lse, ws)
    return out, lse


def assert_scores_close(gpu: np.ndarray, ora: np.ndarray, what=""):
    floor = SCORE_FLOOR * float(np.max(ora)) if ora.size else 0.0
    err = np.abs(gpu.astype(np.float64) - ora)
    bad = ~(err <= SCORE_RTOL * np.abs(ora) + floor)  # NaN counts as a mismatch
    assert not bad.any(), f"{what}: {bad.sum()} scores off, worst {np.nanmax(err) if err.size else 0:.3e}"


def assert_kept_match(gpu_idx: np.ndarray, ora_idx: np.ndarray, ora_scores: np.ndarray, L: int, w: int,
                      m: int, what=""):
    g = gpu_idx[:m]
    assert np.all(np.diff(g) > 0) and g[0] >= 0 and g[-1] < L, f"{what}: not sorted/unique/in range"
    assert np.array_equal(g[m - w:], np.arange(L - w, L)), f"{what}: window not kept"
    gs, os_ = set(g.tolist()), set(ora_idx[:m].tolist())
    if gs == os_:
        return 0
    cand = ora_scores[:L - w]
    kc = m - w
    sk = np.sort(cand)[::-1][kc - 1]
    diff = gs ^ os_
    for j in diff:
        assert j < L - w and abs(cand[j] - sk) <= TIE_RTOL * abs(sk), \
            f"{what}: index {j} differs with score {cand[j]!r} vs boundary {sk!r}"
    return len(diff)


SAMPLE_EPS = 1e-5  # draws this close to a CDF boundary may take the neighbouring token


def assert_tokens_valid(got, zp, u, ref, max_inexact):
    """Sampled tokens vs the oracle's draw: equal, or (a draw within SAMPLE_EPS of a boundary of
    the cumulative distribution) between the oracle's tokens at u -/+ SAMPLE_EPS and with mass.
    zp: the penalised logits [B, V]; at most max_inexact rows may differ."""
    got = np.asarray(got)
    B = got.shape[0]
    none = np.zeros(0, np.int32)
    zero = np.zeros(B, np.float32)
    _, t_lo, _, _, _ = oracle.penalty_sample(zp, none, zero, (np.asarray(u) - SAMPLE_EPS).astype(np.float32))
    _, t_hi, _, _, _ = oracle.penalty_sample(zp, none, zero, (np.asarray(u) + SAMPLE_EPS).astype(np.float32))
    exact = got == ref
    has_mass = np.array([g >= 0 and zp[b, g] != -np.inf for b, g in enumerate(got)])
    near = (got >= t_lo) & (got <= t_hi) & has_mass
    bad = np.nonzero(~(exact | near))[0]
    assert bad.size == 0, [(b, got[b], ref[b], t_lo[b], t_hi[b]) for b in bad[:5]]
    assert (~exact).sum() <= max_inexact, int((~exact).sum())
