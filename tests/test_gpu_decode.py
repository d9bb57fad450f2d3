"""reco_decode_attn vs the oracle's softmax attention (float64), element by element,
over ragged per-unit lengths, with and without the fused append."""
import numpy as np
import pytest
import torch

import oracle
from helpers import DECODE_ATOL, gpu_decode, np32
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


def _oracle_decode(wl, K_np, V_np, lens_np, q_np, kn_np=None, vn_np=None):
    K_np, V_np, lens_np = K_np.copy(), V_np.copy(), lens_np.copy()
    if kn_np is not None:
        for l in range(wl.layers):
            for b in range(wl.batch):
                for h in range(wl.h_kv):
                    L = lens_np[l, b, h]
                    K_np[l, b, h, L] = kn_np[l, b, h]
                    V_np[l, b, h, L] = vn_np[l, b, h]
                    lens_np[l, b, h] = L + 1
    out, lse = oracle.decode_batch(q_np, np.nan_to_num(K_np), np.nan_to_num(V_np), lens_np, wl.scale())
    return out, lse, K_np, V_np, lens_np


def _check(wl, lens_np, append: bool, out_dtype=torch.float32, steps=1):
    K, V = W.make_cache(wl, DEV, canary=False)  # the test poisons rows >= its own lengths
    lens = torch.from_numpy(lens_np).to(DEV)
    for l in range(wl.layers):
        for b in range(wl.batch):
            for h in range(wl.h_kv):
                K[l, b, h, int(lens_np[l, b, h]):] = float("nan")
                V[l, b, h, int(lens_np[l, b, h]):] = float("nan")
    K_np, V_np, L_np = np32(K), np32(V), lens_np.copy()
    atol = DECODE_ATOL[wl.dtype]
    for s in range(steps):
        q, kn, vn = W.make_decode_step(wl, s, DEV)
        out, lse = gpu_decode(wl, K, V, lens, q, kn if append else None, vn if append else None, out_dtype)
        reco.reco_check()
        o_ref, lse_ref, K_np, V_np, L_np = _oracle_decode(wl, K_np, V_np, L_np, np32(q),
                                                          np32(kn) if append else None,
                                                          np32(vn) if append else None)
        got = out.float().cpu().numpy()
        tol = atol + (np.abs(o_ref) * 2.0 ** -8 if out_dtype == torch.bfloat16 else 0.0)
        err = np.abs(got - o_ref)
        assert (err <= tol).all(), f"step {s}: worst {np.nanmax(err):.3e}, NaN {np.isnan(err).sum()}"
        lse_got = lse.cpu().numpy()
        fin = np.isfinite(lse_ref)
        assert np.array_equal(np.isfinite(lse_got), fin)
        assert np.abs(lse_got[fin] - lse_ref[fin]).max(initial=0) < 1e-3
        np.testing.assert_array_equal(lens.cpu().numpy(), L_np)
        if append:  # the new rows landed in the cache
            np.testing.assert_array_equal(np.nan_to_num(np32(K)), np.nan_to_num(K_np))
            np.testing.assert_array_equal(np.nan_to_num(np32(V)), np.nan_to_num(V_np))


@pytest.mark.parametrize("name", ["1.5b", "7b", "32b"])
@pytest.mark.parametrize("append", [False, True])
def test_bf16_decode_ragged(name, append):
    base = W.WORKLOADS[name]
    wl = base.reduced(layers=2, batch=2, L=3000, decode_steps=3)
    rng = np.random.default_rng(7)
    hi = wl.L_cap - (3 if append else 0)
    lens = rng.integers(1, hi + 1, (2, 2, wl.h_kv)).astype(np.int32)
    lens[0, 0, 0] = hi
    lens[1, 1, 0] = 1
    _check(wl, lens, append, steps=3 if append else 1)


def test_bf16_decode_bf16_output_and_d64():
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=3, L=900, decode_steps=2)
    _check(wl, np.array([[[900, 1, 17, 899]] * 3], np.int32).reshape(1, 3, 4), True, torch.bfloat16, steps=2)
    wl64 = W.WORKLOADS["7b"].reduced(layers=1, batch=2, h_q=8, h_kv=2, d=64, L=500, decode_steps=1)
    _check(wl64, np.array([[[500, 37], [3, 250]]], np.int32), True)


def test_fp32_decode_tiny_and_d128():
    wl = W.WORKLOADS["tiny"]
    _check(wl, np.array([[[128, 256]]], np.int32), True)
    wl2 = W.WORKLOADS["tiny"].reduced(d=128, h_q=6, h_kv=2, L=300, decode_steps=2, batch=2)
    _check(wl2, np.array([[[300, 5], [1, 150]]], np.int32), True, steps=2)


def test_long_single_unit_many_splits():
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=1, h_q=7, h_kv=1, L=40000, decode_steps=1)
    _check(wl, np.array([[[40000]]], np.int32), True)


def test_empty_unit_and_no_room():
    wl = W.WORKLOADS["7b"].reduced(layers=1, batch=2, h_q=7, h_kv=1, L=64, decode_steps=0)
    K, V = W.make_cache(wl, DEV, canary=False)
    q, _, _ = W.make_decode_step(wl, 0, DEV)
    lens = torch.tensor([[[0], [10]]], dtype=torch.int32, device=DEV)
    out, lse = gpu_decode(wl, K, V, lens, q)
    reco.reco_check()
    assert torch.all(out[0, 0] == 0) and torch.all(torch.isneginf(lse[0, 0]))
    # a full unit cannot take an appended row: error word, zero output, length unchanged
    _, kn, vn = W.make_decode_step(wl.reduced(decode_steps=1), 0, DEV)
    lens = torch.tensor([[[64], [10]]], dtype=torch.int32, device=DEV)
    out, lse = gpu_decode(wl, K, V, lens, q, kn, vn)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    assert torch.all(out[0, 0] == 0) and int(lens[0, 0, 0]) == 64 and int(lens[0, 1, 0]) == 11
    reco.reco_check()


def test_workspace_counters_left_zero_and_reused():
    """Units long enough to be cut between warps (their pieces merge through per-unit
    tickets): two appends in a row on one zero-filled workspace, each checked against the
    oracle, and the counter region is zero again after each call."""
    wl = W.WORKLOADS["7b"].reduced(layers=2, batch=2, L=6000, decode_steps=4)
    K, V = W.make_cache(wl, DEV, canary=False)
    lens_np = np.array([[[6000, 5000, 4100, 3000], [2500, 6000, 5900, 17]]] * 2, np.int32)
    lens = torch.from_numpy(lens_np).to(DEV)
    kv = reco.make_kv(K, V, wl.h_q)
    ws = reco.workspace(reco.RECO_OP_DECODE, kv, 0, DEV)
    units = wl.layers * wl.batch * wl.h_kv
    K_np, V_np = np32(K), np32(V)
    for step in range(2):
        q, kn, vn = W.make_decode_step(wl, 10 + step, DEV)
        out = torch.empty(q.shape, dtype=torch.float32, device=DEV)
        lse = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
        reco.reco_decode_attn(kv, q, kn, vn, lens, wl.scale(), out, lse, ws)
        reco.reco_check()
        ref, lse_ref, K_np, V_np, lens_np = _oracle_decode(wl, K_np, V_np, lens_np, np32(q), np32(kn), np32(vn))
        assert (np.abs(out.cpu().numpy() - ref) <= DECODE_ATOL["bf16"]).all(), step
        assert np.abs(lse.cpu().numpy() - lse_ref).max() < 1e-3
        np.testing.assert_array_equal(lens.cpu().numpy(), lens_np)
        counters = ws[: (2 + units) * 4].view(torch.int32).cpu().numpy()
        assert (counters == 0).all(), counters


def test_deep_ring_partition_ragged():
    """About 96 K blocks of 16 keys: the launch runs 4 warps per CTA with rings twice as deep.
    Ragged lengths (long units cut between warps, short ones whole), two appends in a row."""
    wl = W.WORKLOADS["7b"].reduced(layers=4, batch=8, L=12000, decode_steps=4)
    rng = np.random.default_rng(41)
    lens = rng.integers(9000, 12001, (4, 8, wl.h_kv)).astype(np.int32)
    lens[0, 0, :] = [1, 17, 255, 256]  # short units among the long ones
    assert (lens.astype(np.int64) + 15).__floordiv__(16).sum() >= 64 * 152 * 8
    _check(wl, lens, True, steps=2)


@pytest.mark.parametrize("shape", [(64, 16, 56, 8), (1, 8193, 7, 1), (2, 4100, 8, 1), (1, 4097, 16, 1)])
def test_tma_path_unit_limit(shape):
    """8192 units (the most one TMA launch plans in shared memory), then more: 8193 and 8200
    units run as two launches over unit ranges, and so do 4097 units of 16 heads (two
    virtual units each)."""
    layers, batch, h_q, h_kv = shape
    wl = W.WORKLOADS["7b"].reduced(layers=layers, batch=batch, h_q=h_q, h_kv=h_kv, L=40, decode_steps=4)
    rng = np.random.default_rng(42 + layers)
    lens = rng.integers(1, 41, (layers, batch, h_kv)).astype(np.int32)
    _check(wl, lens, True)


@pytest.mark.parametrize("shape,top", [((28, 14, 28, 4), 255), ((28, 32, 28, 4), 255), ((2, 3, 7, 1), 255),
                                       ((8, 4, 32, 2), 255), ((28, 14, 28, 4), 256)])
def test_short_units_sorted_and_dealt_whole(shape, top):
    """Units of at most 16 blocks after the append are sorted by length and dealt whole to the
    warps in snake order: fewer units than warps, between one and two per warp, more than two,
    two halves of 16 heads per KV head, and (top 256, 17 blocks with the append) the switch back
    to the contiguous deal.  Units without keys (no append) and of one key are among them."""
    layers, batch, h_q, h_kv = shape
    wl = W.WORKLOADS["7b"].reduced(layers=layers, batch=batch, h_q=h_q, h_kv=h_kv, L=300, decode_steps=2)
    rng = np.random.default_rng(layers * batch + top)
    lens = rng.integers(0, top + 1, (layers, batch, h_kv)).astype(np.int32)
    flat = lens.reshape(-1)
    flat[:3] = [0, 1, top]
    flat[-2:] = [0, top]
    _check(wl, lens, False)  # units of length 0 have no keys: zero output, lse -inf
    _check(wl, lens, True, steps=2)


@pytest.mark.parametrize("h_q,h_kv", [(16, 2), (12, 1), (9, 3)])
def test_bf16_decode_more_than_8_heads_per_kv_head(h_q, h_kv):
    """G = 8, 12, 3 ... and 16, 12, 9 heads per KV head: the TMA path takes a unit of more than
    8 heads as two units of ceil(G / 2) heads over the same rows; ragged lengths, appends (the
    new row written once), three steps, bf16 and fp32 output."""
    wl = W.WORKLOADS["7b"].reduced(layers=2, batch=3, h_q=h_q, h_kv=h_kv, L=2000, decode_steps=3)
    rng = np.random.default_rng(h_q)
    hi = wl.L_cap - 3
    lens = rng.integers(1, hi + 1, (2, 3, h_kv)).astype(np.int32)
    lens[0, 0, 0] = hi
    lens[1, 2, -1] = 1
    _check(wl, lens, True, steps=3)
    _check(wl, lens, True, torch.bfloat16, steps=1)


def test_bf16_decode_g16_long_units_cut_between_warps():
    """G = 16 with units long enough to be cut over many warps (partial merges of both halves
    of every unit), in the deep-ring partition."""
    wl = W.WORKLOADS["7b"].reduced(layers=2, batch=4, h_q=32, h_kv=2, L=40000, decode_steps=2)
    rng = np.random.default_rng(77)
    lens = rng.integers(30000, 40001, (2, 4, 2)).astype(np.int32)
    lens[0, 0, 0] = 5
    _check(wl, lens, True, steps=2)
