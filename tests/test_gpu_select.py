"""reco_select_compact (and its two halves as separate calls, reco_select_topm then
reco_compact) vs the oracle: kept indices and compacted rows bit-exact.

The scores are generator inputs given to both sides, so the selection decision is
taken on identical float32 values and must agree exactly, ties included."""
import numpy as np
import pytest
import torch

import oracle
from helpers import gpu_select, gpu_select_split, np32
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


def _bits(t: torch.Tensor) -> np.ndarray:
    return t.cpu().view(torch.int16 if t.dtype == torch.bfloat16 else torch.int32).numpy()


def _run_case(wl, lens_np, keep_np, scores_np, split=False):
    K, V = W.make_cache(wl, DEV, canary=False)
    K0, V0 = K.clone(), V.clone()
    lens = torch.from_numpy(lens_np).to(DEV)
    scores = torch.from_numpy(scores_np).to(DEV)
    kept = (gpu_select_split if split else gpu_select)(wl, K, V, scores, lens, keep_np)
    reco.reco_check()
    ora_idx = oracle.select_batch(scores_np, lens_np, keep_np, wl.w)
    Kb, Vb, K0b, V0b = _bits(K), _bits(V), _bits(K0), _bits(V0)
    kept_np = kept.cpu().numpy()
    lens_after = lens.cpu().numpy()
    for l in range(wl.layers):
        for b in range(wl.batch):
            for h in range(wl.h_kv):
                L, m = int(lens_np[l, b, h]), int(keep_np[b])
                idx = ora_idx[l, b, h, :m]
                np.testing.assert_array_equal(kept_np[l, b, h, :m], idx)
                assert lens_after[l, b, h] == m
                np.testing.assert_array_equal(Kb[l, b, h, :m], K0b[l, b, h, idx])
                np.testing.assert_array_equal(Vb[l, b, h, :m], V0b[l, b, h, idx])
                np.testing.assert_array_equal(Kb[l, b, h, m:], K0b[l, b, h, m:])  # tail untouched
                np.testing.assert_array_equal(Vb[l, b, h, m:], V0b[l, b, h, m:])


def _tie_scores(rng, shape, levels):
    return (rng.integers(0, levels, shape) / levels).astype(np.float32)


@pytest.mark.parametrize("split", [False, True])
@pytest.mark.parametrize("dtype,d", [("bf16", 128), ("bf16", 64), ("f32", 64), ("f32", 128)])
def test_select_compact_ragged_with_ties(dtype, d, split):
    wl = W.WORKLOADS["1.5b"].reduced(layers=2, batch=3, h_q=4, h_kv=2, d=d, dtype=dtype, L=1200,
                                     decode_steps=37, w=32, outliers=0)
    rng = np.random.default_rng(1)
    lens = rng.integers(600, wl.L_cap + 1, (wl.layers, wl.batch, wl.h_kv)).astype(np.int32)
    keep = np.array([wl.w + int(rng.integers(0, lens[:, b].min() - wl.w + 1)) for b in range(wl.batch)],
                    np.int32)
    scores = rng.random((wl.layers, wl.batch, wl.h_kv, wl.L_cap)).astype(np.float32)
    scores[0, 1] = _tie_scores(rng, wl.L_cap, 7)  # heavy ties
    scores[1, 2, 0] = 0.5  # all equal: lowest indices win
    _run_case(wl, lens, keep, scores, split)


@pytest.mark.parametrize("split", [False, True])
def test_select_edge_cases(split):
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=5, h_q=4, h_kv=1, L=300, decode_steps=0, w=16)
    rng = np.random.default_rng(2)
    lens = np.array([[[300]], [[300]], [[16]], [[300]], [[257]]], np.int32).reshape(1, 5, 1)
    keep = np.array([16, 300, 16, 299, 100], np.int32)  # window only, identity, L == w, chain, ragged
    scores = rng.random((1, 5, 1, 300)).astype(np.float32)
    scores[0, 3, 0, :] = 1.0
    scores[0, 3, 0, 0] = 0.0  # drop only candidate 0: every kept row moves up by one (in-place chain)
    _run_case(wl, lens, keep, scores, split)


def test_select_plateaus_from_maxpool_shape():
    """Plateaus like a max-pool produces (runs of equal values) at the selection boundary."""
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=2, h_q=4, h_kv=2, L=4096, decode_steps=0, w=32)
    rng = np.random.default_rng(3)
    raw = rng.random((1, 2, 2, 4096)).astype(np.float32)
    pooled = np.maximum.reduce([np.roll(raw, s, axis=-1) for s in range(-3, 4)])
    lens = np.full((1, 2, 2), 4096, np.int32)
    keep = np.array([1024, 2000], np.int32)
    _run_case(wl, lens, keep, pooled.astype(np.float32))


def test_select_bad_keep_sets_device_error_and_skips_unit():
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=2, h_q=4, h_kv=1, L=200, decode_steps=0, w=16)
    K, V = W.make_cache(wl, DEV, canary=False)
    K0 = K.clone()
    lens = torch.full((1, 2, 1), 200, dtype=torch.int32, device=DEV)
    scores = torch.rand((1, 2, 1, 200), device=DEV)
    gpu_select(wl, K, V, scores, lens, np.array([201, 50], np.int32))  # keep > L for sequence 0
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    assert torch.equal(K[0, 0].view(torch.int16), K0[0, 0].view(torch.int16))
    assert int(lens[0, 0, 0]) == 200 and int(lens[0, 1, 0]) == 50
    reco.reco_check()  # the word was cleared and the context is still usable


def test_select_compact_beyond_shared_memory_keys():
    """Units with more candidates than the shared-memory selection holds (48 Ki keys) take
    the selection that reads its keys from global memory: same results, ties included."""
    wl = W.WORKLOADS["1.5b"].reduced(layers=1, batch=2, h_q=2, h_kv=1, L=50_000, decode_steps=8, w=32,
                                     outliers=0)
    assert wl.L_cap - wl.w > 48 * 1024
    rng = np.random.default_rng(21)
    lens = np.array([[[50_000], [49_500]]], np.int32)
    keep = np.array([12_345, 30_001], np.int32)
    _run_case(wl, lens, keep, _tie_scores(rng, (1, 2, 1, wl.L_cap), 4096))


def test_select_topm_touches_only_the_indices():
    wl = W.WORKLOADS["7b"].reduced(layers=2, batch=3, h_q=8, h_kv=2, L=700, decode_steps=5, w=32)
    K, V = W.make_cache(wl, DEV, canary=False)
    K0, V0 = K.clone(), V.clone()
    rng = np.random.default_rng(8)
    lens_np = rng.integers(400, 701, (2, 3, 2)).astype(np.int32)
    keep_np = np.array([100, 32, 399], np.int32)
    scores_np = rng.random((2, 3, 2, wl.L_cap)).astype(np.float32)
    lens = torch.from_numpy(lens_np).to(DEV)
    kv = reco.make_kv(K, V, wl.h_q)
    kept = torch.full(K.shape[:4], -1, dtype=torch.int32, device=DEV)
    ws = reco.workspace(reco.RECO_OP_SELECT, kv, wl.w, DEV)
    reco.reco_select_topm(kv, torch.from_numpy(scores_np).to(DEV), lens, torch.from_numpy(keep_np).to(DEV), wl.w,
                          kept, ws)
    reco.reco_check()
    assert torch.equal(K.view(torch.int16), K0.view(torch.int16)) and torch.equal(V.view(torch.int16),
                                                                                   V0.view(torch.int16))
    np.testing.assert_array_equal(lens.cpu().numpy(), lens_np)
    ora = oracle.select_batch(scores_np, lens_np, keep_np, wl.w)
    got = kept.cpu().numpy()
    for l in range(2):
        for b in range(3):
            for h in range(2):
                m = int(keep_np[b])
                np.testing.assert_array_equal(got[l, b, h, :m], ora[l, b, h, :m])
                assert (got[l, b, h, m:] == -1).all()


def test_compact_refuses_indices_outside_r_to_L():
    """reco_compact copies only sources in [r, L): a source below its destination (which an
    earlier destination may have overwritten) or at/after the unit's length is refused."""
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=2, h_q=4, h_kv=1, L=64, decode_steps=4, w=4)
    K, V = W.make_cache(wl, DEV, canary=False)
    K0 = K.clone()
    kv = reco.make_kv(K, V, wl.h_q)
    lens = torch.tensor([[[64], [40]]], dtype=torch.int32, device=DEV)
    keep = torch.tensor([8, 8], dtype=torch.int32, device=DEV)
    kept = torch.zeros(K.shape[:4], dtype=torch.int32, device=DEV)
    kept[0, 0, 0, :8] = torch.tensor([2, 0, 9, 20, 60, 61, 62, 63])  # row 1 <- row 0: refused
    kept[0, 1, 0, :8] = torch.tensor([1, 2, 3, 4, 5, 6, 7, 40])  # row 40 == L: refused
    reco.reco_compact(kv, kept, lens, keep, wl.w)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    Kb, K0b = _bits(K), _bits(K0)
    for r, src in enumerate([2, None, 9, 20, 60, 61, 62, 63]):
        np.testing.assert_array_equal(Kb[0, 0, 0, r], K0b[0, 0, 0, r if src is None else src])
    for r, src in enumerate([1, 2, 3, 4, 5, 6, 7, None]):
        np.testing.assert_array_equal(Kb[0, 1, 0, r], K0b[0, 1, 0, r if src is None else src])
    assert lens.flatten().tolist() == [8, 8]
    reco.reco_check()


@pytest.mark.parametrize("split", [False, True])
def test_select_compact_walks_many_units_with_untouched_sequences(split):
    """8192 units (64 layers x 16 sequences x 8 KV heads): every CTA walks a few dozen units.
    Half the sequences keep their whole cache (keep = L: identity indices, nothing moves, the
    compaction skips them) and the others compress, with ties."""
    wl = W.WORKLOADS["7b"].reduced(layers=64, batch=16, h_q=8, h_kv=8, L=96, w=8, decode_steps=0)
    rng = np.random.default_rng(77)
    L_seq = rng.integers(40, 97, wl.batch)
    lens_np = np.broadcast_to(L_seq[None, :, None], (wl.layers, wl.batch, wl.h_kv)).astype(np.int32).copy()
    keep_np = np.where(np.arange(wl.batch) % 2 == 0, L_seq, rng.integers(wl.w, L_seq)).astype(np.int32)
    scores_np = _tie_scores(rng, (wl.layers, wl.batch, wl.h_kv, wl.L_cap), 16)
    _run_case(wl, lens_np, keep_np, scores_np, split=split)
