"""reco_score_cache with a keep mask (Sec. 3.1-3.2: sequences reach step boundaries at
different tokens, so a compression call usually compresses only a few of them).

A unit whose sequence keeps its whole cache (keep[b] >= lens[unit]) is skipped: its
rows of scores must come back bit-for-bit as they went in.  Every other unit must get
exactly the unmasked call's scores (same kernels, same per-unit arithmetic) and stay
within tolerance of the oracle.  Covers the tensor-core passes (one buffer and split
query columns), the float32 SIMT passes, units of one sequence split by the mask, a
call that skips everything, and a bad length that the mask must not hide."""
import numpy as np
import pytest
import torch

import oracle
from helpers import assert_scores_close, np32
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"
SENTINEL = -12345.0


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


def _score(wl, K, V, q, lens, keep):
    kv = reco.make_kv(K, V, wl.h_q)
    scores = torch.full(K.shape[:4], SENTINEL, dtype=torch.float32, device=DEV)
    ws = reco.workspace(reco.RECO_OP_SCORE, kv, wl.w, DEV)
    keep_t = None if keep is None else torch.as_tensor(keep, dtype=torch.int32, device=DEV)
    reco.reco_score_cache(kv, q, lens, wl.w, wl.pool, wl.scale(), scores, ws, keep=keep_t)
    reco.reco_check()
    return scores.cpu().numpy()


def _check(wl, lens_np, keep, oracle_too=True):
    K, V = W.make_cache(wl, DEV, canary=False)
    q = W.make_qwin(wl, DEV)
    lens = torch.from_numpy(lens_np).to(DEV)
    full = _score(wl, K, V, q, lens, None)
    got = _score(wl, K, V, q, lens, keep)
    ora = oracle.score_cache(np32(q), np32(K), lens_np, wl.w, wl.pool, wl.scale()) if oracle_too else None
    n_skip = 0
    for l in range(wl.layers):
        for b in range(wl.batch):
            for h in range(wl.h_kv):
                L = int(lens_np[l, b, h])
                if keep[b] >= L:  # skipped: untouched
                    n_skip += 1
                    assert (got[l, b, h] == SENTINEL).all(), (l, b, h)
                    continue
                nc = L - wl.w
                np.testing.assert_array_equal(got[l, b, h, :nc].view(np.uint32), full[l, b, h, :nc].view(np.uint32))
                assert (got[l, b, h, nc:] == SENTINEL).all()
                if ora is not None:
                    assert_scores_close(got[l, b, h, :nc], ora[l, b, h, :nc], f"unit {(l, b, h)}")
    return n_skip


def _ragged(wl, seed):
    rng = np.random.default_rng(seed)
    return rng.integers(wl.w + 1, wl.L_cap + 1, (wl.layers, wl.batch, wl.h_kv)).astype(np.int32)


@pytest.mark.parametrize("name", ["7b", "32b"])  # 7B: G*w = 224 (one buffer); 32B: 320 (split columns)
def test_bf16_mask_skips_some_sequences(name):
    wl = W.WORKLOADS[name].reduced(layers=2, batch=5, L=2300, decode_steps=40)
    lens = _ragged(wl, 11)
    keep = np.full(wl.batch, 1 << 30, np.int32)  # every unit of these sequences is skipped
    keep[1] = wl.w  # compress sequence 1 ...
    keep[3] = int(np.median(lens[:, 3]))  # ... and the units of sequence 3 that are longer than keep
    n_skip = _check(wl, lens, keep)
    assert 0 < n_skip < wl.layers * wl.batch * wl.h_kv


def test_fp32_mask_simt_path():
    wl = W.WORKLOADS["tiny"].reduced(layers=2, batch=3, L=500, decode_steps=13)
    lens = _ragged(wl, 12)
    keep = np.array([1 << 30, wl.w, 1 << 30], np.int32)
    assert _check(wl, lens, keep) == 2 * 2 * wl.h_kv


def test_mask_that_skips_everything_and_nothing():
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=3, L=900, decode_steps=10)
    lens = _ragged(wl, 13)
    assert _check(wl, lens, np.full(3, 1 << 30, np.int32), oracle_too=False) == wl.batch * wl.h_kv
    assert _check(wl, lens, np.full(3, wl.w, np.int32), oracle_too=False) == 0


def test_mask_does_not_hide_a_bad_length():
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=2, L=300, decode_steps=4)
    K, V = W.make_cache(wl, DEV, canary=False)
    q = W.make_qwin(wl, DEV)
    lens_np = np.full((1, 2, wl.h_kv), 200, np.int32)
    lens_np[0, 0, 0] = wl.L_cap + 1  # out of range, in a sequence the mask would skip
    kv = reco.make_kv(K, V, wl.h_q)
    scores = torch.zeros(K.shape[:4], dtype=torch.float32, device=DEV)
    ws = reco.workspace(reco.RECO_OP_SCORE, kv, wl.w, DEV)
    keep = torch.tensor([1 << 30, wl.w], dtype=torch.int32, device=DEV)
    reco.reco_score_cache(kv, q, torch.from_numpy(lens_np).to(DEV), wl.w, wl.pool, wl.scale(), scores, ws, keep=keep)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    reco.reco_check()
