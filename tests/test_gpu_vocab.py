"""reco_reflect_penalty (bit-exact) and reco_answer_ppl (1e-3 relative) vs the oracle."""
import numpy as np
import pytest
import torch

import oracle
from helpers import PPL_RTOL, np32
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


def test_penalty_bit_exact_7b_vocab():
    wl = W.WORKLOADS["7b"]
    z = W.make_vocab_logits(wl, DEV)
    z0 = z.cpu().numpy().copy()
    ids_np = W.make_reflection_ids(wl)
    ids_np = np.concatenate([ids_np, ids_np[:3]])  # duplicates: still one subtraction each
    rewards_np = np.array([0.0, 0.4, 0.41, 0.79, 0.8, 1.0, 0.55, 0.2], np.float32)
    beta = torch.empty(8, device=DEV)
    reco.reco_reflect_penalty(z, torch.from_numpy(ids_np).to(DEV), torch.from_numpy(rewards_np).to(DEV),
                              0.4, 0.8, 4.0, beta)
    reco.reco_check()
    ref, beta_ref, bad = oracle.reflect_penalty(z0, ids_np, rewards_np, 0.4, 0.8, 4.0)
    assert bad == 0
    np.testing.assert_array_equal(z.cpu().numpy().view(np.uint32), ref.view(np.uint32))
    np.testing.assert_array_equal(beta.cpu().numpy(), beta_ref)


def test_penalty_bad_id_sets_device_error():
    z = torch.zeros((2, 10), device=DEV)
    ids = torch.tensor([3, 10, -1], dtype=torch.int32, device=DEV)
    reco.reco_reflect_penalty(z, ids, torch.tensor([1.0, 0.5], device=DEV))
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    ref, _, bad = oracle.reflect_penalty(np.zeros((2, 10), np.float32), [3, 10, -1], [1.0, 0.5])
    assert bad == 2
    np.testing.assert_array_equal(z.cpu().numpy(), ref)
    reco.reco_check()


def _ppl_case(logits, tokens, n_valid=None, tau_p=1.1):
    B, n, V = logits.shape
    ppl = torch.empty(B, device=DEV)
    stop = torch.empty(B, dtype=torch.uint8, device=DEV)
    ws = reco.workspace(reco.RECO_OP_PPL, None, B * n, DEV)
    nv = None if n_valid is None else torch.from_numpy(np.asarray(n_valid, np.int32)).to(DEV)
    reco.reco_answer_ppl(logits, tokens, nv, tau_p, ppl, stop, ws)
    reco.reco_check()
    ref, stop_ref = oracle.answer_ppl(np32(logits), tokens.cpu().numpy(), n_valid, tau_p)
    got = ppl.cpu().numpy().astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(got), nan)
    assert np.all(np.abs(got[~nan] - ref[~nan]) <= PPL_RTOL * ref[~nan])
    near = np.abs(ref - tau_p) <= 1e-3 * tau_p
    assert np.array_equal(stop.cpu().numpy().astype(bool)[~near], stop_ref[~near])
    return got, stop.cpu().numpy()


def test_ppl_7b_answer_probe():
    wl = W.WORKLOADS["7b"]
    z, tok = W.make_answer(wl, DEV)
    got, stop = _ppl_case(z, tok)
    assert stop[0::2].all() and not stop[1::2].any()  # boosted targets stop, the rest do not


def test_ppl_ragged_lengths_odd_vocab_and_empty():
    rng = np.random.default_rng(3)
    B, n, V = 5, 9, 1001  # V not a multiple of 4: scalar path
    z = torch.from_numpy((rng.standard_normal((B, n, V)) * 2).astype(np.float32)).to(DEV)
    tok = torch.from_numpy(rng.integers(0, V, (B, n)).astype(np.int32)).to(DEV)
    _ppl_case(z, tok, [9, 1, 0, 4, 20])


def test_ppl_golden_two_token():
    z = torch.tensor([[[0.0] * 8, [float(np.log(7.0))] + [0.0] * 7]], device=DEV)
    tok = torch.tensor([[5, 0]], dtype=torch.int32, device=DEV)
    got, stop = _ppl_case(z, tok)
    assert abs(got[0] - 4.0) < 4e-3 and not stop[0]


def test_ppl_bad_token_sets_device_error():
    z = torch.zeros((1, 2, 8), device=DEV)
    tok = torch.tensor([[1, 8]], dtype=torch.int32, device=DEV)
    ppl = torch.empty(1, device=DEV)
    stop = torch.empty(1, dtype=torch.uint8, device=DEV)
    ws = reco.workspace(reco.RECO_OP_PPL, None, 2, DEV)
    reco.reco_answer_ppl(z, tok, None, 1.1, ppl, stop, ws)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    assert torch.isnan(ppl[0]) and int(stop[0]) == 0
    reco.reco_check()
