"""reco_score_cache_lse: Eq. 2 with the window rows' normalisers taken from the decode.

The window queries are decoded one token at a time (each call appends the token's key and
value and returns the log-sum-exp of its query over the keys it sees), then the scores of
the final cache come from one pass over K with those log-sum-exps.  They are compared with
the oracle's Eq. 2 scores of the same cache and window (float64, its own normalisers),
element by element, and the kept sets with the oracle's selection."""
import numpy as np
import pytest
import torch

import oracle
from helpers import assert_kept_match, assert_scores_close, gpu_select, np32
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


def _window_case(wl, L_final):
    """Full cache, window queries, and the per-unit initial lengths L_final - w."""
    Kf, Vf = W.make_cache(wl, DEV, canary=False)
    q_win = W.make_qwin(wl, DEV)
    lens_f = np.asarray(L_final, np.int32)
    return Kf, Vf, q_win, lens_f, lens_f - wl.w


def _rows_at(X, pos):
    """X[l, b, h, pos[l, b, h], :] for every unit."""
    idx = torch.from_numpy(pos.astype(np.int64)).to(DEV)[..., None, None].expand(*pos.shape, 1, X.shape[-1])
    return torch.gather(X, 3, idx).squeeze(3).contiguous()


def _decode_window(wl, Kf, Vf, q_win, lens0):
    """Decode the w window tokens into a cache that starts at lens0 rows: returns the cache,
    the final lengths (device) and row_lse [w, Ly, B, Hq] from the decode calls."""
    K = Kf.clone()
    V = Vf.clone()
    kv = reco.make_kv(K, V, wl.h_q)
    ws = reco.workspace(reco.RECO_OP_DECODE, kv, 0, DEV)
    lens = torch.from_numpy(lens0.copy()).to(DEV)
    row_lse = torch.empty((wl.w, wl.layers, wl.batch, wl.h_q), dtype=torch.float32, device=DEV)
    out = torch.empty((wl.layers, wl.batch, wl.h_q, wl.d), dtype=torch.float32, device=DEV)
    for t in range(wl.w):
        kn, vn = _rows_at(Kf, lens0 + t), _rows_at(Vf, lens0 + t)
        q = q_win[:, :, :, t, :].contiguous()
        reco.reco_decode_attn(kv, q, kn, vn, lens, wl.scale(), out, row_lse[t], ws)
    reco.reco_check()
    return K, V, lens, row_lse


def _score_lse(wl, K, V, q_win, lens, row_lse, keep=None, fill=0.0):
    kv = reco.make_kv(K, V, wl.h_q)
    scores = torch.full(K.shape[:4], fill, dtype=torch.float32, device=DEV)
    ws = reco.workspace(reco.RECO_OP_SCORE, kv, wl.w, DEV)
    reco.reco_score_cache_lse(kv, q_win, lens, row_lse, wl.w, wl.pool, wl.scale(), scores, ws, keep=keep)
    return scores


def _compare(wl, got, ora, lens_f, skip=()):
    for l in range(wl.layers):
        for b in range(wl.batch):
            if b in skip:
                continue
            for h in range(wl.h_kv):
                nc = int(lens_f[l, b, h]) - wl.w
                assert_scores_close(got[l, b, h, :nc], ora[l, b, h, :nc], f"unit {(l, b, h)}")


CASES = [
    # (workload, reduction): bf16 on the tensor-core pass, fp32 and d 64 on the SIMT pass
    ("7b", dict(layers=2, batch=2, L=900, decode_steps=40)),
    ("32b", dict(layers=1, batch=2, L=700, decode_steps=70)),
    ("7b", dict(layers=1, batch=2, h_q=8, h_kv=2, d=64, L=600, decode_steps=40, w=24)),
    ("tiny", dict(L=512, decode_steps=20)),
]


@pytest.mark.parametrize("name,red", CASES)
def test_lse_scores_from_decoded_window(name, red):
    """The normalisers come from the library's own decode of the window tokens."""
    wl = W.WORKLOADS[name].reduced(**red)
    rng = np.random.default_rng(11)
    L_final = rng.integers(wl.w + 1, wl.L_cap - 2, (wl.layers, wl.batch, wl.h_kv)).astype(np.int32)
    L_final[0, 0, 0] = wl.w  # no candidates at all
    Kf, Vf, q_win, lens_f, lens0 = _window_case(wl, L_final)
    K, V, lens, row_lse = _decode_window(wl, Kf, Vf, q_win, lens0)
    assert np.array_equal(lens.cpu().numpy(), lens_f)
    got = _score_lse(wl, K, V, q_win, lens, row_lse).cpu().numpy()
    reco.reco_check()
    ora = oracle.score_cache(np32(q_win), np32(Kf), lens_f, wl.w, wl.pool, wl.scale())
    _compare(wl, got, ora, lens_f)


def test_lse_scores_from_oracle_normalisers():
    """The normalisers come from the oracle's decode of each window row (fp64 rounded to
    fp32), so this isolates the one-pass scoring from the decode."""
    wl = W.WORKLOADS["7b"].reduced(layers=2, batch=2, L=1300, decode_steps=40)
    L_final = np.random.default_rng(3).integers(wl.w + 1, wl.L_cap, (2, 2, wl.h_kv)).astype(np.int32)
    Kf, Vf, q_win, lens_f, lens0 = _window_case(wl, L_final)
    qn, Kn, Vn = np32(q_win), np32(Kf), np32(Vf)
    row_lse = np.stack([oracle.decode_batch(qn[:, :, :, t, :], Kn, Vn, lens0 + t + 1, wl.scale())[1]
                        for t in range(wl.w)]).astype(np.float32)
    lens = torch.from_numpy(lens_f).to(DEV)
    got = _score_lse(wl, Kf, Vf, q_win, lens, torch.from_numpy(row_lse).to(DEV)).cpu().numpy()
    reco.reco_check()
    ora = oracle.score_cache(qn, Kn, lens_f, wl.w, wl.pool, wl.scale())
    _compare(wl, got, ora, lens_f)


def test_lse_keep_mask_and_selection():
    """With keep counts, only the sequences compressed now are scored (the others' rows of
    scores stay as they were), and the kept sets match the oracle's selection up to the
    tie band."""
    wl = W.WORKLOADS["7b"].reduced(layers=2, batch=3, L=1500, decode_steps=40)
    L_final = np.random.default_rng(8).integers(800, wl.L_cap, (2, 3, wl.h_kv)).astype(np.int32)
    L_final[:, 1, :] = 1200  # one length for the whole sequence: its keep count below is a no-op
    Kf, Vf, q_win, lens_f, lens0 = _window_case(wl, L_final)
    K, V, lens, row_lse = _decode_window(wl, Kf, Vf, q_win, lens0)
    keep = np.array([400, 1200, 700], np.int32)  # sequence 1 keeps its whole cache: skipped
    keep_t = torch.from_numpy(keep).to(DEV)
    scores = _score_lse(wl, K, V, q_win, lens, row_lse, keep=keep_t, fill=-7.0)
    got = scores.cpu().numpy()
    reco.reco_check()
    assert np.all(got[:, 1] == -7.0)
    ora = oracle.score_cache(np32(q_win), np32(Kf), lens_f, wl.w, wl.pool, wl.scale())
    _compare(wl, got, ora, lens_f, skip=(1,))
    kept = gpu_select(wl, K, V, scores, lens, keep).cpu().numpy()
    reco.reco_check()
    for l in range(wl.layers):
        for b in (0, 2):
            for h in range(wl.h_kv):
                L = int(lens_f[l, b, h])
                m = min(int(keep[b]), L)
                ora_idx = oracle.select_unit(ora[l, b, h].astype(np.float32), L, wl.w, m)
                assert_kept_match(kept[l, b, h], ora_idx, ora[l, b, h], L, wl.w, m, f"unit {(l, b, h)}")


def test_non_finite_normaliser_sets_device_error():
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=1, L=300, decode_steps=4)
    Kf, Vf, q_win, lens_f, _ = _window_case(wl, np.full((1, 1, wl.h_kv), 300, np.int32))
    row_lse = torch.full((wl.w, 1, 1, wl.h_q), 5.0, dtype=torch.float32, device=DEV)
    row_lse[3, 0, 0, 2] = float("nan")
    scores = _score_lse(wl, Kf, Vf, q_win, torch.from_numpy(lens_f).to(DEV), row_lse)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE and "normaliser" in str(e.value)
    assert torch.isfinite(scores).all()
    reco.reco_check()


def test_lse_push_ring_and_slot():
    """Each push writes its ring row and the mirror row `slots` further on at the device slot
    and advances the slot modulo `slots` (bit-exact copies), so the last w pushes are the
    contiguous rows s0 .. s0+w-1 with s0 = (slot - w) mod slots.  An out-of-range slot
    writes nothing and sets the error word."""
    n, slots, w = 1000, 5, 3
    ring = torch.full((2 * slots, n), -1.0, device=DEV)
    slot = torch.tensor([3], dtype=torch.int64, device=DEV)
    vals = [torch.randn(n, device=DEV) for _ in range(7)]
    for v in vals:
        reco.reco_lse_push(v, ring, slot)
    reco.reco_check()
    nxt = int(slot.item())
    assert nxt == (3 + 7) % slots
    assert torch.equal(ring[:slots], ring[slots:])
    last = {(3 + i) % slots: v for i, v in enumerate(vals)}
    for k, v in last.items():
        assert torch.equal(ring[k], v)
    s0 = (nxt - w) % slots
    assert torch.equal(ring[s0:s0 + w], torch.stack(vals[-w:]))
    slot.fill_(9)
    before = ring.clone()
    reco.reco_lse_push(vals[0], ring, slot)
    with pytest.raises(reco.RecoError):
        reco.reco_check()
    assert torch.equal(ring, before) and int(slot.item()) == 9


@pytest.mark.parametrize("dtype,h_q,h_kv,L", [("bf16", 28, 4, 700), ("bf16", 16, 1, 300), ("f32", 8, 2, 200)])
def test_decode_attn_ring_matches_decode_then_push(dtype, h_q, h_kv, L):
    """reco_decode_attn_ring is reco_decode_attn followed by reco_lse_push: the same outputs,
    cache and lengths, the lse in ring rows slot and slot + S (bit-exact), the slot advanced
    (with a wrap-around), each head's query in its row slot of q_ring (the other rows
    untouched), on the TMA path (bf16, G 7), the SIMT path (G 16, and float32)."""
    wl = W.WORKLOADS["7b"].reduced(layers=2, batch=3, h_q=h_q, h_kv=h_kv, L=L, decode_steps=4, dtype=dtype)
    Ka, Va = W.make_cache(wl, DEV, canary=False)
    Kb, Vb = Ka.clone(), Va.clone()
    rng = np.random.default_rng(5)
    lens_np = rng.integers(1, L + 1, (wl.layers, wl.batch, wl.h_kv)).astype(np.int32)
    la, lb = torch.from_numpy(lens_np).to(DEV), torch.from_numpy(lens_np).to(DEV)
    kva, kvb = reco.make_kv(Ka, Va, wl.h_q), reco.make_kv(Kb, Vb, wl.h_q)
    wsa, wsb = reco.workspace(reco.RECO_OP_DECODE, kva, 0, DEV), reco.workspace(reco.RECO_OP_DECODE, kvb, 0, DEV)
    S, n = 3, wl.layers * wl.batch * wl.h_q
    ring_a, ring_b = torch.zeros((2 * S, n), device=DEV), torch.zeros((2 * S, n), device=DEV)
    slot_a, slot_b = torch.tensor([1], dtype=torch.int64, device=DEV), torch.tensor([1], dtype=torch.int64, device=DEV)
    q_ring = torch.full((wl.layers, wl.batch, wl.h_q, S, wl.d), -3.0, dtype=wl.torch_dtype, device=DEV)
    q_ref = q_ring.clone()
    for s in range(4):
        q, kn, vn = W.make_decode_step(wl, s, DEV)
        oa, ob = torch.empty(q.shape, device=DEV), torch.empty(q.shape, device=DEV)
        lse = torch.empty(q.shape[:3], device=DEV)
        reco.reco_decode_attn(kva, q, kn, vn, la, wl.scale(), oa, lse, wsa)
        reco.reco_lse_push(lse, ring_a, slot_a)
        q_ref[:, :, :, (1 + s) % S] = q
        reco.reco_decode_attn_ring(kvb, q, kn, vn, lb, wl.scale(), ob, ring_b, slot_b, wsb, q_ring=q_ring)
        reco.reco_check()
        assert torch.equal(oa, ob) and torch.equal(la, lb)
        assert torch.equal(ring_a, ring_b) and int(slot_b.item()) == (2 + s) % S
        assert torch.equal(q_ring.view(torch.uint8), q_ref.view(torch.uint8))
    assert torch.equal(Ka.view(torch.uint8), Kb.view(torch.uint8))
    # an out-of-range slot: no ring row written, slot kept, the error word set
    before = ring_b.clone()
    slot_b.fill_(S)
    q, kn, vn = W.make_decode_step(wl, 9, DEV)
    reco.reco_decode_attn_ring(kvb, q, None, None, lb, wl.scale(), torch.empty(q.shape, device=DEV), ring_b, slot_b, wsb,
                               q_ring=q_ring)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    assert torch.equal(ring_b, before) and int(slot_b.item()) == S
    assert torch.equal(q_ring.view(torch.uint8), q_ref.view(torch.uint8))
    reco.reco_check()


def test_copy_row_selects_the_row_on_the_device():
    """reco_copy_row copies row *index, read on the device: plain calls, a captured graph whose
    index moves between replays, a row of several grid passes, and out-of-range indices (nothing
    copied, the device error word set)."""
    rng = np.random.default_rng(11)
    src = torch.from_numpy(rng.integers(0, 256, (5, 4096 * 3 + 16 * 7), dtype=np.uint8)).to(DEV)
    dst = torch.zeros(src.shape[1], dtype=torch.uint8, device=DEV)
    idx = torch.zeros(1, dtype=torch.int64, device=DEV)
    for r in (0, 4, 2):
        idx.fill_(r)
        reco.reco_copy_row(src, idx, dst)
        reco.reco_check()
        assert torch.equal(dst, src[r])
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        reco.reco_copy_row(src, idx, dst, s)
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=s):
            reco.reco_copy_row(src, idx, dst, s)
    torch.cuda.synchronize()
    for r in (3, 1):
        idx.fill_(r)
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(dst, src[r])
    big = torch.from_numpy(rng.integers(0, 256, (2, 24 << 20), dtype=np.uint8)).to(DEV)  # several passes
    dbig = torch.zeros(big.shape[1], dtype=torch.uint8, device=DEV)
    idx.fill_(1)
    reco.reco_copy_row(big, idx, dbig)
    reco.reco_check()
    assert torch.equal(dbig, big[1])
    before = dst.clone()
    for bad in (5, -1):
        idx.fill_(bad)
        reco.reco_copy_row(src, idx, dst)
        with pytest.raises(reco.RecoError) as e:
            reco.reco_check()
        assert e.value.status == reco.RECO_EDEVICE
        assert torch.equal(dst, before)
    reco.reco_check()


def test_decode_attn_ring_split_over_unit_ranges():
    """8200 units run as two launches: the lse of every query head in ring rows slot and
    slot + S, its query in q_ring row slot, the outputs and lengths those of reco_decode_attn,
    and the slot advanced once."""
    wl = W.WORKLOADS["7b"].reduced(layers=2, batch=1025, h_q=28, h_kv=4, L=48, decode_steps=2)
    assert wl.layers * wl.batch * wl.h_kv > 8192
    Ka, Va = W.make_cache(wl, DEV, canary=False)
    Kb, Vb = Ka.clone(), Va.clone()
    rng = np.random.default_rng(9)
    lens_np = rng.integers(1, 40, (wl.layers, wl.batch, wl.h_kv)).astype(np.int32)
    la, lb = torch.from_numpy(lens_np).to(DEV), torch.from_numpy(lens_np).to(DEV)
    kva, kvb = reco.make_kv(Ka, Va, wl.h_q), reco.make_kv(Kb, Vb, wl.h_q)
    wsa, wsb = reco.workspace(reco.RECO_OP_DECODE, kva, 0, DEV), reco.workspace(reco.RECO_OP_DECODE, kvb, 0, DEV)
    S, n = 2, wl.layers * wl.batch * wl.h_q
    ring = torch.zeros((2 * S, n), device=DEV)
    slot = torch.tensor([1], dtype=torch.int64, device=DEV)
    q_ring = torch.zeros((wl.layers, wl.batch, wl.h_q, S, wl.d), dtype=wl.torch_dtype, device=DEV)
    q, kn, vn = W.make_decode_step(wl, 0, DEV)
    oa, ob = torch.empty(q.shape, device=DEV), torch.empty(q.shape, device=DEV)
    lse = torch.empty(q.shape[:3], device=DEV)
    reco.reco_decode_attn(kva, q, kn, vn, la, wl.scale(), oa, lse, wsa)
    reco.reco_decode_attn_ring(kvb, q, kn, vn, lb, wl.scale(), ob, ring, slot, wsb, q_ring=q_ring)
    reco.reco_check()
    assert torch.equal(oa, ob) and torch.equal(la, lb) and int(slot.item()) == 0
    assert torch.equal(ring[1], lse.view(-1)) and torch.equal(ring[1 + S], lse.view(-1))
    assert torch.equal(ring[0], torch.zeros_like(ring[0])) and torch.equal(ring[S], torch.zeros_like(ring[0]))
    assert torch.equal(q_ring[:, :, :, 1], q) and torch.equal(q_ring[:, :, :, 0], torch.zeros_like(q))
    assert torch.equal(Ka.view(torch.uint8), Kb.view(torch.uint8))
