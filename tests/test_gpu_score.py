"""reco_score_cache vs the oracle's Eq. 2 scores (float64), element by element.

Shapes span several 128-key tiles, two 2048-key chunks and a ragged tail; lengths
are ragged per unit; rows past each length are NaN canaries (never read)."""
import numpy as np
import pytest
import torch

import oracle
from helpers import assert_scores_close, gpu_score, np32
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


def _check(wl, lens_np, pool):
    K, V = W.make_cache(wl, DEV, canary=False)  # the test poisons rows >= its own lengths
    q = W.make_qwin(wl, DEV)
    lens = torch.from_numpy(lens_np).to(DEV)
    # rows in [lens, L) are valid data the kernel must not read: poison them too
    for l in range(wl.layers):
        for b in range(wl.batch):
            for h in range(wl.h_kv):
                K[l, b, h, int(lens_np[l, b, h]):] = float("nan")
    scores = gpu_score(wl, K, V, q, lens, pool)
    reco.reco_check()
    ora = oracle.score_cache(np32(q), np.nan_to_num(np32(K)), lens_np, wl.w, pool, wl.scale())
    got = scores.cpu().numpy()
    for l in range(wl.layers):
        for b in range(wl.batch):
            for h in range(wl.h_kv):
                nc = int(lens_np[l, b, h]) - wl.w
                assert_scores_close(got[l, b, h, :nc], ora[l, b, h, :nc], f"unit {(l, b, h)}")


def test_tiny_fp32_scores():
    wl = W.WORKLOADS["tiny"]
    _check(wl, W.make_lens(wl).numpy(), 7)


@pytest.mark.parametrize("name,pool", [("1.5b", 7), ("7b", 7), ("7b", 1), ("32b", 7)])
def test_bf16_scores_ragged(name, pool):
    base = W.WORKLOADS[name]
    wl = base.reduced(layers=1, batch=2, L=2600, decode_steps=40)
    rng = np.random.default_rng(5)
    lens = rng.integers(wl.w, wl.L_cap + 1, (1, 2, wl.h_kv)).astype(np.int32)
    lens[0, 0, 0] = wl.L_cap  # full capacity
    lens[0, 1, 0] = wl.w  # no candidates at all
    if wl.h_kv > 1:
        lens[0, 1, 1] = wl.w + 1  # a single candidate
    _check(wl, lens, pool)


def test_fp32_d128_and_bf16_d64_scores():
    for dtype, d in [("f32", 128), ("bf16", 64)]:
        wl = W.WORKLOADS["7b"].reduced(layers=2, batch=1, h_q=8, h_kv=2, d=d, dtype=dtype, L=700,
                                       decode_steps=5, w=24)
        _check(wl, np.full((2, 1, 2), 700, np.int32), 5)


def test_bad_length_sets_device_error():
    wl = W.WORKLOADS["tiny"]
    K, V = W.make_cache(wl, DEV)
    q = W.make_qwin(wl, DEV)
    lens = torch.tensor([[[wl.w - 1, 600]]], dtype=torch.int32, device=DEV)  # below w; above L_cap
    gpu_score(wl, K, V, q, lens)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    reco.reco_check()
