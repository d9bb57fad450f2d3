"""Seeded input generators: determinism, shapes and the NaN canary rows (CPU)."""
import numpy as np
import torch

from paper_2608_04771_gb300 import workloads as W


def test_generators_are_deterministic_and_shaped():
    wl = W.WORKLOADS["tiny"]
    K1, V1 = W.make_cache(wl)
    K2, V2 = W.make_cache(wl)
    assert K1.shape == (1, 1, 2, wl.L_cap, 64) and K1.dtype == torch.float32
    assert torch.equal(K1[..., :wl.L, :], K2[..., :wl.L, :])
    assert torch.isnan(K1[..., wl.L:, :]).all() and torch.isnan(V1[..., wl.L:, :]).all()
    assert not torch.equal(K1[..., :wl.L, :], V1[..., :wl.L, :])
    q = W.make_qwin(wl)
    assert q.shape == (1, 1, 8, 16, 64)
    h = W.make_reward_history(wl)
    assert h.shape == (1, 1) and h[0, 0] == np.float32(0.8)


def test_reduced_bf16_cache_and_outliers():
    wl = W.WORKLOADS["1.5b"].reduced(layers=2, batch=1, L=40, decode_steps=2)
    K, V = W.make_cache(wl)
    assert K.dtype == torch.bfloat16 and K.shape == (2, 1, 2, 42, 128)
    ch = W.outlier_channels(wl)
    assert ch.shape == (2, 2, 4)
    for l in range(2):
        for h in range(2):
            assert len(set(ch[l, h].tolist())) == 4
            big = K[l, 0, h, :40].float().abs().mean(0)
            assert big[ch[l, h]].min() > 5 * big.median()


def test_rewards_answer_and_ids():
    wl = W.WORKLOADS["7b"]
    h = W.make_reward_history(wl)
    assert h.shape == (8, 16) and h.min() >= 0 and h.max() <= 1
    ids = W.make_reflection_ids(wl)
    assert len(set(ids.tolist())) == 16 and ids.max() < wl.vocab
    small = wl.reduced(vocab=300, n_answer=5)
    z, tok = W.make_answer(small)
    assert z.shape == (8, 5, 300) and tok.shape == (8, 5)
    picked = z.gather(2, tok.long().unsqueeze(-1)).squeeze(-1)
    assert (picked[0::2] > 10).all()


def test_trace_steps_sum_to_generated():
    steps = W.make_trace_steps(4, 1000, 96, 16, 4)
    for s in steps:
        assert sum(s) == 1000 and min(s[:-1]) >= 16
