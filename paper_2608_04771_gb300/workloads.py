"""Seeded synthetic inputs shaped like the paper's reasoning workloads.

This module only draws random numbers and holds shapes: it contains none of the
method's arithmetic (no retention ratios, scores, selections or penalties), so
the CUDA path and the oracle can both take their inputs from it without sharing
any computation.

The paper's models (R1-Distill-Qwen-7B / Llama-8B, Qwen3-8B), datasets and the
Pilot reward model are not available, so every tensor is synthetic:
  * queries, keys, values ~ N(0, 1); the 1.5B-class stack scales 4 channels per
    (layer, KV head) by 20 in both K and V (outlier channels);
  * step rewards ~ U[0,1] or Beta(2,2) per step; a sequence's history holds
    ``history`` draws, the last one being the current step's reward;
  * vocabulary logits ~ N(0, 4) (sigma 2); reflection ids are distinct seeded ids;
  * answer logits ~ N(0, 4) with the target logit raised by 20 for every other
    sequence, so both outcomes of the stop rule occur.
Small tensors come from numpy's PCG64 (seeded per tensor); large caches come from
torch's generator on the target device (seeded per tensor), so their values depend
on the device they are drawn on.
"""
from __future__ import annotations

import dataclasses
from dataclasses import dataclass

import numpy as np
import torch


@dataclass(frozen=True)
class Workload:
    name: str
    layers: int
    batch: int
    h_q: int
    h_kv: int
    d: int
    dtype: str  # "f32" or "bf16"
    L: int  # cache length at the compression point
    w: int  # observation window
    pool: int  # max-pool kernel
    decode_steps: int
    vocab: int  # 0: no penalty / PPL leg
    n_ids: int  # reflection-token ids
    n_answer: int  # answer tokens for the PPL probe
    reward: str  # "fixed:<v>", "uniform", "beta22"
    history: int  # rewards per sequence
    base: float  # lambda
    delta: float  # delta
    outliers: int  # outlier channels per (layer, KV head), x20
    seed: int
    tau_l: float = 0.4
    tau_h: float = 0.8
    beta: float = 4.0
    tau_p: float = 1.1

    @property
    def G(self) -> int:
        return self.h_q // self.h_kv

    @property
    def L_cap(self) -> int:
        return self.L + self.decode_steps

    @property
    def units(self) -> int:
        return self.layers * self.batch * self.h_kv

    @property
    def torch_dtype(self):
        return torch.float32 if self.dtype == "f32" else torch.bfloat16

    @property
    def elem_bytes(self) -> int:
        return 4 if self.dtype == "f32" else 2

    def scale(self) -> float:
        return 1.0 / float(np.sqrt(self.d))

    def reduced(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)


WORKLOADS = {
    # 1 layer, batch 1, 8/2 heads, d 64, fp32, cache 512, window 16, pool 7, reward 0.8, 1 decode step
    "tiny": Workload("tiny", 1, 1, 8, 2, 64, "f32", 512, 16, 7, 1, 1024, 8, 8, "fixed:0.8", 1,
                     0.25, 0.1, 0, 0),
    # 1.5B-class stack: 28 layers, 12/2 heads, d 128, bf16, batch 4, cache 4096, window 32, 64 steps
    "1.5b": Workload("1.5b", 28, 4, 12, 2, 128, "bf16", 4096, 32, 7, 64, 0, 0, 0, "uniform", 16,
                     0.25, 0.1, 4, 1),
    # 7B-class (Qwen2.5-7B shape): 28 layers, 28/4 heads, batch 8, cache 16384, window 32, 128 steps,
    # vocab 152064 penalty with 16 reflection ids, answer PPL over 32 tokens
    "7b": Workload("7b", 28, 8, 28, 4, 128, "bf16", 16384, 32, 7, 128, 152064, 16, 32, "beta22", 16,
                   0.25, 0.1, 0, 2),
    # 32B-class (Qwen2.5-32B shape): 64 layers, 40/8 heads, batch 4, cache 32768, window 64,
    # ratios spanning 0.2-0.9 (lambda 0.55, delta 0.35), 256 steps
    "32b": Workload("32b", 64, 4, 40, 8, 128, "bf16", 32768, 64, 7, 256, 0, 0, 0, "uniform", 16,
                    0.55, 0.35, 0, 3),
}

# Step-loop trace: 7B-class heads, batch 16, prompt 256, 8192 generated tokens,
# steps of Poisson(96)+16 tokens, Beta(2,2) reward per step.
TRACE = dict(base="7b", batch=16, prompt=256, generated=8192, step_mean=96, step_min=16, seed=4)


def _np_rng(wl: Workload, stream: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64([wl.seed, stream]))


def _torch_gen(wl: Workload, stream: int, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(wl.seed * 1_000_003 + stream)
    return g


def randn(shape, wl: Workload, stream: int, device="cpu", dtype=None) -> torch.Tensor:
    """N(0,1) tensor from a per-(workload, stream) seeded torch generator, rounded to dtype."""
    g = _torch_gen(wl, stream, device)
    x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    return x.to(dtype or wl.torch_dtype)


def outlier_channels(wl: Workload) -> np.ndarray:
    """[layers, h_kv, outliers] channel indices (distinct per row)."""
    rng = _np_rng(wl, 11)
    out = np.zeros((wl.layers, wl.h_kv, wl.outliers), np.int64)
    for l in range(wl.layers):
        for h in range(wl.h_kv):
            out[l, h] = rng.choice(wl.d, wl.outliers, replace=False)
    return out


def _cache_tensor(wl: Workload, stream: int, device, canary: bool) -> torch.Tensor:
    shape = (wl.layers, wl.batch, wl.h_kv, wl.L_cap, wl.d)
    x = randn(shape, wl, stream, device, torch.float32)
    if wl.outliers:
        ch = torch.from_numpy(outlier_channels(wl)).to(device)
        for l in range(wl.layers):
            for h in range(wl.h_kv):
                x[l, :, h, :, ch[l, h]] *= 20.0
    if canary and wl.L_cap > wl.L:
        x[:, :, :, wl.L:, :] = float("nan")
    y = x.to(wl.torch_dtype)
    del x
    return y


def make_cache(wl: Workload, device="cpu", canary: bool = True):
    """K, V of shape [layers, batch, h_kv, L_cap, d]; rows >= L are NaN when ``canary``.
    The outlier channels (if any) are scaled by 20 in both K and V."""
    K = _cache_tensor(wl, 1, device, canary)
    V = _cache_tensor(wl, 2, device, canary)
    return K, V


def make_lens(wl: Workload, device="cpu") -> torch.Tensor:
    return torch.full((wl.layers, wl.batch, wl.h_kv), wl.L, dtype=torch.int32, device=device)


def make_qwin(wl: Workload, device="cpu") -> torch.Tensor:
    """Observation-window queries [layers, batch, h_q, w, d]."""
    return randn((wl.layers, wl.batch, wl.h_q, wl.w, wl.d), wl, 3, device)


def make_reward_history(wl: Workload) -> np.ndarray:
    """[batch, history] float32 step rewards; column -1 is the current step's v_i."""
    if wl.reward.startswith("fixed:"):
        v = np.float32(float(wl.reward.split(":")[1]))
        return np.full((wl.batch, wl.history), v, np.float32)
    rng = _np_rng(wl, 4)
    if wl.reward == "uniform":
        h = rng.random((wl.batch, wl.history))
    elif wl.reward == "beta22":
        h = rng.beta(2.0, 2.0, (wl.batch, wl.history))
    else:
        raise ValueError(wl.reward)
    return h.astype(np.float32)


def make_decode_step(wl: Workload, step: int, device="cpu"):
    """(q [layers,batch,h_q,d], k_new, v_new [layers,batch,h_kv,d]) for decode step ``step``."""
    s = 100 + 3 * step
    q = randn((wl.layers, wl.batch, wl.h_q, wl.d), wl, s, device)
    kn = randn((wl.layers, wl.batch, wl.h_kv, wl.d), wl, s + 1, device)
    vn = randn((wl.layers, wl.batch, wl.h_kv, wl.d), wl, s + 2, device)
    return q, kn, vn


def make_vocab_logits(wl: Workload, device="cpu", stream: int = 5) -> torch.Tensor:
    """[batch, vocab] float32 logits ~ N(0, 4)."""
    return randn((wl.batch, wl.vocab), wl, stream, device, torch.float32) * 2.0


def make_draws(wl: Workload, n: int, stream: int = 13) -> np.ndarray:
    """[n] float32 uniform draws on the 2^-24 grid of [0, 1) (exact in float32)."""
    rng = _np_rng(wl, stream)
    return (rng.integers(0, 1 << 24, n) / float(1 << 24)).astype(np.float32)


def make_reflection_ids(wl: Workload) -> np.ndarray:
    rng = _np_rng(wl, 6)
    return rng.choice(wl.vocab, wl.n_ids, replace=False).astype(np.int32)


def make_answer(wl: Workload, device="cpu"):
    """(logits [batch, n_answer, vocab] f32, tokens [batch, n_answer] i32)."""
    rng = _np_rng(wl, 7)
    tokens = rng.integers(0, wl.vocab, (wl.batch, wl.n_answer)).astype(np.int32)
    z = randn((wl.batch, wl.n_answer, wl.vocab), wl, 8, device, torch.float32) * 2.0
    tok = torch.from_numpy(tokens).to(device).long()
    boost = torch.zeros(wl.batch, device=device)
    boost[0::2] = 20.0
    z.scatter_add_(2, tok.unsqueeze(-1), boost.view(-1, 1, 1).expand(-1, wl.n_answer, 1))
    return z, torch.from_numpy(tokens).to(device)


def make_trace_steps(batch: int, generated: int, step_mean: int, step_min: int, seed: int):
    """Per-sequence step lengths (Poisson(step_mean) + step_min) summing to ``generated``."""
    rng = np.random.Generator(np.random.PCG64([seed, 9]))
    out = []
    for _ in range(batch):
        steps, total = [], 0
        while total < generated:
            s = int(rng.poisson(step_mean)) + step_min
            s = min(s, generated - total)
            steps.append(s)
            total += s
        out.append(steps)
    return out


def make_trace_rewards(steps_per_seq, seed: int):
    rng = np.random.Generator(np.random.PCG64([seed, 10]))
    return [rng.beta(2.0, 2.0, len(s)).astype(np.float32) for s in steps_per_seq]
