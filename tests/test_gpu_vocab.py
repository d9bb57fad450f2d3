"""reco_reflect_penalty (bit-exact), reco_penalty_sample (penalty bit-exact, draws equal up to the
boundary band) and reco_answer_ppl (1e-3 relative) vs the oracle."""
import numpy as np
import pytest
import torch

import oracle
from helpers import PPL_RTOL, assert_tokens_valid, np32
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


def test_ppl_logits_not_16_byte_aligned():
    """V a multiple of 4 but the logits one float into their allocation: the kernel must
    not take its 16-byte vector loads (a misaligned vector load faults)."""
    rng = np.random.default_rng(5)
    B, n, V = 3, 7, 2048
    buf = torch.from_numpy((rng.standard_normal(B * n * V + 1) * 2).astype(np.float32)).to(DEV)
    z = buf[1:].view(B, n, V)
    assert z.data_ptr() % 16 == 4 and z.is_contiguous()
    tok = torch.from_numpy(rng.integers(0, V, (B, n)).astype(np.int32)).to(DEV)
    _ppl_case(z, tok, [7, 2, 5])


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


# ---------------------------------------------------------------- penalty + sampling
def _sample_case(z, ids_np, rewards_np, u_np, tau_l=0.4, tau_h=0.8, beta=4.0, max_inexact=None):
    """GPU penalty + draw vs the oracle: penalised logits bit-exact; tokens equal, or (a draw
    within SAMPLE_EPS of a boundary) between the oracle's tokens at u -/+ SAMPLE_EPS and with mass."""
    B, V = z.shape
    z0 = np32(z).copy()
    tok = torch.full((B,), -7, dtype=torch.int32, device=DEV)
    beta_out = torch.empty(B, device=DEV)
    ws = reco.sample_workspace(B, V, DEV)
    reco.reco_penalty_sample(z, torch.from_numpy(np.asarray(ids_np, np.int32)).to(DEV),
                             torch.from_numpy(rewards_np).to(DEV), torch.from_numpy(u_np).to(DEV), tok, ws,
                             tau_l, tau_h, beta, beta_out)
    reco.reco_check()
    zp, ref, _, _, bad = oracle.penalty_sample(z0, ids_np, rewards_np, u_np, tau_l, tau_h, beta)
    assert bad == 0
    np.testing.assert_array_equal(np32(z).view(np.uint32), zp.view(np.uint32))
    beta_ref = np.array([[0.0, beta / 2, beta][oracle.penalty_band(v, tau_l, tau_h)] for v in rewards_np], np.float32)
    np.testing.assert_array_equal(beta_out.cpu().numpy(), beta_ref)
    got = tok.cpu().numpy()
    assert_tokens_valid(got, zp, u_np, ref, max(1, B // 100) if max_inexact is None else max_inexact)
    return got, ref


def test_penalty_sample_7b_vocab():
    wl = W.WORKLOADS["7b"]
    ids_np = W.make_reflection_ids(wl)
    rewards_np = np.array([0.0, 0.4, 0.41, 0.79, 0.8, 1.0, 0.55, 0.2], np.float32)
    for k in range(4):
        z = W.make_vocab_logits(wl, DEV, stream=40 + k)
        _sample_case(z, ids_np, rewards_np, W.make_draws(wl, wl.batch, stream=50 + k))


def test_penalty_sample_moves_mass_off_reflection_tokens():
    """Reflection ids carry most of the mass; the band of the reward decides how much is left."""
    rng = np.random.default_rng(31)
    B, V = 96, 1000
    z = torch.from_numpy((rng.standard_normal((B, V))).astype(np.float32)).to(DEV)
    ids_np = rng.choice(V, 20, replace=False).astype(np.int32)
    z[:, torch.from_numpy(ids_np).long().to(DEV)] += 7.0
    rewards_np = np.repeat(np.array([0.1, 0.6, 0.9], np.float32), B // 3)
    u_np = ((np.arange(B) % 32 + 0.5) / 32).astype(np.float32)
    got, _ = _sample_case(z, ids_np, rewards_np, u_np)
    in_R = np.isin(got, ids_np)
    frac = [in_R[i * 32:(i + 1) * 32].mean() for i in range(3)]
    assert frac[0] > frac[1] > frac[2], frac  # no, half and full penalty


@pytest.mark.parametrize("V", [1, 7, 4095, 4096, 4097, 8193, 100000])
def test_penalty_sample_ragged_vocab_and_edge_draws(V):
    rng = np.random.default_rng(V)
    B = 6
    z = torch.from_numpy((rng.standard_normal((B, V)) * 2).astype(np.float32)).to(DEV)
    ids_np = rng.choice(V, min(V, 5), replace=False).astype(np.int32)
    u_np = np.array([0.0, 0.5, np.float32(1 - 2 ** -24), rng.random(), np.nan, 0.999], np.float32)
    _sample_case(z, ids_np, np.array([1.0, 0.5, 0.0, 0.9, 1.0, 0.3], np.float32), u_np, max_inexact=1)


@pytest.mark.parametrize("V,offset", [(9216, 0), (152064, 0), (393216, 0), (393220, 0), (152064, 1)])
def test_penalty_sample_one_launch_limits(V, offset):
    """Rows drawn in one launch (a cluster per row): CTAs of the cluster left without
    records (V 9216), the largest row (V 393216, 48 records per CTA), then one record past
    it and a row off a 16-byte boundary, both drawn through the workspace."""
    rng = np.random.default_rng(V + offset)
    B = 3
    buf = torch.from_numpy((rng.standard_normal(B * V + offset) * 2).astype(np.float32)).to(DEV)
    z = buf[offset:].view(B, V)
    ids_np = rng.choice(V, 40, replace=False).astype(np.int32)
    ids_np[:8] = np.arange(V - 8, V)  # ids in the last record
    ids_np[8] = ids_np[9]  # a repeated id: one subtraction
    u_np = np.array([0.3, np.float32(1 - 2 ** -24), 0.0], np.float32)
    _sample_case(z, ids_np, np.array([1.0, 0.5, 0.9], np.float32), u_np, max_inexact=1)


def test_penalty_sample_masked_tokens_and_empty_rows():
    rng = np.random.default_rng(33)
    B, V = 8, 9000
    z_np = (rng.standard_normal((B, V)) * 2).astype(np.float32)
    z_np[rng.random((B, V)) < 0.6] = -np.inf  # most tokens masked
    z_np[3] = -np.inf  # no token has mass: -1
    z_np[5, :] = -np.inf
    z_np[5, 8999] = 0.0  # only the last token
    u_np = rng.random(B).astype(np.float32)
    got, _ = _sample_case(torch.from_numpy(z_np).to(DEV), np.zeros(0, np.int32), np.zeros(B, np.float32), u_np)
    assert got[3] == -1 and got[5] == 8999


def test_penalty_sample_stratified_rows_follow_the_distribution():
    """2048 rows of the same logits with stratified draws: every row matches the oracle (up to the
    boundary band), so the token counts are N p to within one plus the band cases."""
    rng = np.random.default_rng(34)
    V, N = 3000, 2048
    z1 = (rng.standard_normal(V) * 2).astype(np.float32)
    u_np = ((np.arange(N) + 0.5) / N).astype(np.float32)
    got, ref = _sample_case(torch.from_numpy(np.repeat(z1[None], N, 0)).to(DEV), np.zeros(0, np.int32),
                            np.zeros(N, np.float32), u_np, max_inexact=4)
    p = np.exp(z1.astype(np.float64) - z1.max())
    p /= p.sum()
    counts = np.bincount(got, minlength=V)
    assert np.abs(counts - N * p).max() <= 1.0 + (got != ref).sum() + 1e-6


def test_penalty_sample_bad_id_sets_device_error():
    z = torch.zeros((2, 10), device=DEV)
    tok = torch.empty(2, dtype=torch.int32, device=DEV)
    ws = reco.sample_workspace(2, 10, DEV)
    reco.reco_penalty_sample(z, torch.tensor([3, 10, -1], dtype=torch.int32, device=DEV),
                             torch.tensor([1.0, 0.5], device=DEV), torch.tensor([0.1, 0.9], device=DEV), tok, ws)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_check()
    assert e.value.status == reco.RECO_EDEVICE
    ref, _, _ = oracle.reflect_penalty(np.zeros((2, 10), np.float32), [3, 10, -1], [1.0, 0.5])
    np.testing.assert_array_equal(z.cpu().numpy(), ref)
    reco.reco_check()


def test_penalty_sample_largest_vocab():
    """V = 4 * 1024 * 1024 logits per row (1024 segments, the most a row may have)."""
    V, B = 4 * 1024 * 1024, 2
    rng = np.random.default_rng(35)
    z = torch.from_numpy((rng.standard_normal((B, V)) * 2).astype(np.float32)).to(DEV)
    ids_np = rng.choice(V, 16, replace=False).astype(np.int32)
    _sample_case(z, ids_np, np.array([1.0, 0.6], np.float32), np.array([0.37, 0.999], np.float32), max_inexact=1)
