"""Full-size workloads in the launch configuration bench.py times (driver.HotPath),
checked on sampled units that the oracle computes one by one."""
import numpy as np
import pytest
import torch

import oracle
from helpers import (DECODE_ATOL, PPL_RTOL, assert_kept_match, assert_scores_close, np32)
from paper_2608_04771_gb300 import driver, reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


@pytest.mark.parametrize("name,out_dtype", [("32b", torch.bfloat16), ("7b", torch.bfloat16), ("1.5b", torch.bfloat16),
                                            ("7b", torch.float32)])
def test_full_size_sampled_units(name, out_dtype):
    """bf16 output is what bench.py runs (driver.HotPath's default); fp32 output checks the
    same launch at the tighter bar."""
    wl = W.WORKLOADS[name]
    hp = driver.HotPath(wl, DEV, out_dtype=out_dtype, keep_pristine=False)
    units = [(0, 0, 0), (wl.layers // 2, wl.batch // 2, wl.h_kv - 1), (wl.layers - 1, wl.batch - 1, wl.h_kv // 2),
             (1, wl.batch - 1, 0), (wl.layers - 2, 0, wl.h_kv - 1)]
    G = wl.G
    saved = {}
    for (l, b, h) in units:
        saved[(l, b, h)] = (np32(hp.K[l, b, h, :wl.L]), np32(hp.V[l, b, h, :wl.L]),
                            np32(hp.q_win[l, b, h * G:(h + 1) * G]))
    z0 = hp.logits.cpu().numpy().copy() if hp.has_vocab else None
    hp.step()
    reco.reco_check()
    torch.cuda.synchronize()
    check_steps = sorted({0, 1, wl.decode_steps // 2, wl.decode_steps - 1})
    atol = DECODE_ATOL[wl.dtype]
    for (l, b, h) in units:
        K0, V0, q = saved[(l, b, h)]
        m = int(hp.keep_host[b])
        _, pooled = oracle.score_unit(q, K0, wl.w, wl.scale(), wl.pool)
        got_s = hp.scores[l, b, h, :wl.L - wl.w].cpu().numpy()
        assert_scores_close(got_s, pooled, f"{name} unit {(l, b, h)}")
        ora_idx = oracle.select_unit(pooled.astype(np.float32), wl.L, wl.w, m)
        gk = hp.kept[l, b, h].cpu().numpy()
        assert_kept_match(gk, ora_idx, pooled, wl.L, wl.w, m, f"{name} unit {(l, b, h)}")
        # Compaction and decode follow the GPU's own kept set: equal to the oracle's, or a
        # selection that differs only inside the tie band and is just as valid.
        idx = gk[:m]
        Kc = np.zeros((wl.L_cap, wl.d), np.float32)
        Vc = np.zeros((wl.L_cap, wl.d), np.float32)
        Kc[:m], Vc[:m] = oracle.gather_unit(K0, idx), oracle.gather_unit(V0, idx)
        dk = np32(hp.dk[:, l, b, h])
        dv = np32(hp.dv[:, l, b, h])
        Kc[m:m + wl.decode_steps], Vc[m:m + wl.decode_steps] = dk, dv
        np.testing.assert_array_equal(np32(hp.K[l, b, h, :m + wl.decode_steps]), Kc[:m + wl.decode_steps])
        np.testing.assert_array_equal(np32(hp.V[l, b, h, :m + wl.decode_steps]), Vc[:m + wl.decode_steps])
        assert int(hp.lens[l, b, h]) == m + wl.decode_steps
        for s in check_steps:
            qs = np32(hp.dq[s, l, b, h * G:(h + 1) * G])
            got = hp.out[s, l, b, h * G:(h + 1) * G].float().cpu().numpy()
            for g in range(G):
                o, lse = oracle.decode_unit(qs[g], Kc, Vc, m + s + 1, wl.scale())
                # a bf16 output adds its own rounding: half an ulp, at most 2^-8 of |o|
                tol = atol + (np.abs(o) * 2.0 ** -8 if out_dtype == torch.bfloat16 else 0.0)
                assert (np.abs(got[g] - o) <= tol).all(), (name, s, l, b, h, g, float(np.abs(got[g] - o).max()))
                assert abs(float(hp.lse[s, l, b, h * G + g]) - lse) < 1e-3
    if hp.has_vocab:
        # the penalty ran once per decode step on the same logits buffer
        ids = W.make_reflection_ids(wl)
        ref = z0
        for _ in range(wl.decode_steps):
            ref, beta_ref, _ = oracle.reflect_penalty(ref, ids, hp.hist[:, -1], wl.tau_l, wl.tau_h, wl.beta)
        np.testing.assert_array_equal(hp.logits.cpu().numpy().view(np.uint32), ref.view(np.uint32))
        np.testing.assert_array_equal(hp.beta.cpu().numpy(), beta_ref)
        ppl_ref, stop_ref = oracle.answer_ppl(np32(hp.ans_logits), hp.ans_tokens.cpu().numpy(), None, wl.tau_p)
        got = hp.ppl.cpu().numpy().astype(np.float64)
        assert np.all(np.abs(got - ppl_ref) <= PPL_RTOL * ppl_ref)
        assert np.array_equal(hp.stop.cpu().numpy().astype(bool), stop_ref)


@pytest.mark.parametrize("name", ["7b", "1.5b", "32b"])
def test_full_size_one_pass_scores_sampled(name):
    """reco_score_cache_lse on the full workload cache, as bench.py times it: each window
    query's normaliser is the lse of the library's decode of that query over the keys Eq. 2
    lets it see (lens L-w+t+1, no append); sampled units against the oracle's Eq. 2 scores
    (its own normalisers) and its selection."""
    wl = W.WORKLOADS[name]
    hp = driver.HotPath(wl, DEV, out_dtype=torch.float32, keep_pristine=False)
    ws_dec = reco.workspace(reco.RECO_OP_DECODE, hp.kv, 0, DEV)
    row_lse = torch.empty((wl.w, wl.layers, wl.batch, wl.h_q), dtype=torch.float32, device=DEV)
    out = torch.empty((wl.layers, wl.batch, wl.h_q, wl.d), dtype=torch.float32, device=DEV)
    for t in range(wl.w):
        lens_t = hp.lens0 - (wl.w - 1 - t)
        reco.reco_decode_attn(hp.kv, hp.q_win[:, :, :, t, :].contiguous(), None, None, lens_t, wl.scale(), out,
                              row_lse[t], ws_dec)
    scores = torch.zeros_like(hp.scores)
    reco.reco_score_cache_lse(hp.kv, hp.q_win, hp.lens, row_lse, wl.w, wl.pool, wl.scale(), scores, hp.ws_score)
    reco.reco_check()
    kept = torch.full(hp.K.shape[:4], -1, dtype=torch.int32, device=DEV)
    G = wl.G
    units = [(0, 0, 0), (wl.layers // 2, wl.batch // 2, wl.h_kv - 1), (wl.layers - 1, wl.batch - 1, wl.h_kv // 2)]
    saved = {u: (np32(hp.K[u[0], u[1], u[2], :wl.L]), np32(hp.q_win[u[0], u[1], u[2] * G:(u[2] + 1) * G]))
             for u in units}
    reco.reco_select_compact(hp.kv, scores, hp.lens, hp.keep, wl.w, kept, hp.ws_select)
    reco.reco_check()
    for (l, b, h) in units:
        K0, q = saved[(l, b, h)]
        m = int(hp.keep_host[b])
        _, pooled = oracle.score_unit(q, K0, wl.w, wl.scale(), wl.pool)
        assert_scores_close(scores[l, b, h, :wl.L - wl.w].cpu().numpy(), pooled, f"{name} unit {(l, b, h)}")
        ora_idx = oracle.select_unit(pooled.astype(np.float32), wl.L, wl.w, m)
        assert_kept_match(kept[l, b, h].cpu().numpy(), ora_idx, pooled, wl.L, wl.w, m, f"{name} unit {(l, b, h)}")
