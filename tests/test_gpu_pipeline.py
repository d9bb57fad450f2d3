"""Score -> select/compact -> decode end to end vs the oracle run on the same inputs.

The oracle ranks its own float64 scores (rounded to float32, the precision the
kernel decides in); kept sets must agree except near-boundary candidates (see
helpers).  Decode outputs are compared on every unit against the oracle's attention
over the rows the GPU kept: the oracle's own set, or one that differs from it only
inside the tie band and is just as valid a selection."""
import numpy as np
import pytest
import torch

import oracle
from helpers import (DECODE_ATOL, assert_kept_match, assert_scores_close, gpu_decode, gpu_score, gpu_select,
                     keep_counts, np32)
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


def run_pipeline(wl, ratio=None, steps=None):
    steps = wl.decode_steps if steps is None else steps
    K, V = W.make_cache(wl, DEV, canary=True)
    K0, V0 = np.nan_to_num(np32(K)), np.nan_to_num(np32(V))
    lens = W.make_lens(wl, DEV)
    lens_np = lens.cpu().numpy()
    q = W.make_qwin(wl, DEV)
    keep = keep_counts(wl, ratio=ratio)
    scores = gpu_score(wl, K, V, q, lens)
    kept = gpu_select(wl, K, V, scores, lens, keep)
    reco.reco_check()
    ora_scores = oracle.score_cache(np32(q), K0, lens_np, wl.w, wl.pool, wl.scale())
    ora_idx = oracle.select_batch(ora_scores.astype(np.float32), lens_np, keep, wl.w)
    got_scores, got_kept = scores.cpu().numpy(), kept.cpu().numpy()
    Kg, Vg = np32(K), np32(V)
    same = np.zeros((wl.layers, wl.batch, wl.h_kv), bool)
    Kc, Vc = np.zeros_like(K0), np.zeros_like(V0)
    for l in range(wl.layers):
        for b in range(wl.batch):
            for h in range(wl.h_kv):
                L, m = int(lens_np[l, b, h]), int(keep[b])
                assert_scores_close(got_scores[l, b, h, :L - wl.w], ora_scores[l, b, h, :L - wl.w])
                nd = assert_kept_match(got_kept[l, b, h], ora_idx[l, b, h], ora_scores[l, b, h], L, wl.w, m)
                gi = got_kept[l, b, h, :m]
                np.testing.assert_array_equal(Kg[l, b, h, :m], K0[l, b, h, gi])  # compaction is exact
                np.testing.assert_array_equal(Vg[l, b, h, :m], V0[l, b, h, gi])
                same[l, b, h] = nd == 0
                Kc[l, b, h, :m] = oracle.gather_unit(K0[l, b, h], gi)
                Vc[l, b, h, :m] = oracle.gather_unit(V0[l, b, h], gi)
    assert same.mean() >= 0.9, f"kept sets differ (within the tie band) on {(~same).sum()} units"
    L_np = np.broadcast_to(keep.reshape(1, -1, 1), lens_np.shape).copy()
    np.testing.assert_array_equal(lens.cpu().numpy(), L_np)
    G = wl.G
    for s in range(steps):
        qd, kn, vn = W.make_decode_step(wl, s, DEV)
        out, lse = gpu_decode(wl, K, V, lens, qd, kn, vn)
        reco.reco_check()
        kn_np, vn_np, q_np = np32(kn), np32(vn), np32(qd)
        got = out.cpu().numpy()
        for l in range(wl.layers):
            for b in range(wl.batch):
                for h in range(wl.h_kv):
                    Lc = L_np[l, b, h]
                    Kc[l, b, h, Lc], Vc[l, b, h, Lc] = kn_np[l, b, h], vn_np[l, b, h]
                    L_np[l, b, h] = Lc + 1
                    for g in range(G):
                        o, _ = oracle.decode_unit(q_np[l, b, h * G + g], Kc[l, b, h], Vc[l, b, h], Lc + 1,
                                                  wl.scale())
                        err = np.abs(got[l, b, h * G + g] - o)
                        assert (err <= DECODE_ATOL[wl.dtype]).all(), (s, l, b, h, g, np.nanmax(err))
        np.testing.assert_array_equal(lens.cpu().numpy(), L_np)


def test_tiny_config_reward_ratio():
    """Tiny workload, reward 0.8 alone: lambda = 0.25, m = 128 of 512 (one decode step)."""
    wl = W.WORKLOADS["tiny"]
    assert keep_counts(wl).tolist() == [128]
    run_pipeline(wl)


def test_tiny_config_explicit_ratio_half():
    """The Tiny workload's fallback ratio 0.5: m = 256."""
    wl = W.WORKLOADS["tiny"]
    assert keep_counts(wl, ratio=0.5).tolist() == [256]
    run_pipeline(wl, ratio=0.5)


@pytest.mark.parametrize("name", ["1.5b", "7b", "32b"])
def test_reduced_bf16_stacks(name):
    """The bf16 workloads with fewer layers, a shorter cache and two decode steps."""
    wl = W.WORKLOADS[name].reduced(layers=2, batch=2, L=2300, decode_steps=2)
    run_pipeline(wl)
