"""The step loop of ReCo over a synthetic reasoning trace, through the C ABI.

Each sequence generates tokens one at a time; its trajectory is split into steps of
Poisson(mean) + min tokens (Sec. 3.1 splits at newlines; the lengths here are
synthetic).  Per token, every active sequence decodes one token (append + attention
over its ragged cache, all layers in one call) and the reflection penalty (Eq. 3-4)
is applied to that token's logits with the band of the sequence's latest reward.
When a sequence completes a step it receives a reward v_i (Sec. 3.1), and
  * its cache is compressed to m_i = lambda_i * L (Eq. 1-2, Sec. 3.2) -- all
    sequences are passed to one scoring/selection call, the others with keep = L,
    which leaves them untouched;
  * if v_{i-1} >= tau_h and v_i >= tau_h, the answer probe runs (Eq. 5-6) and a
    sequence that passes PPL <= tau_p stops and leaves the batch.
Budget base L (the paper is silent on repeated compression): reading "A" uses the
current cache length, reading "B" the full uncompressed length so far (the keep
count is then capped at the current length).  Lengths are tracked on the host, so
the loop needs no device read-back except the stop flags of a probe.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

from . import reco
from . import workloads as W


@dataclass
class TraceSpec:
    base: W.Workload
    batch: int
    prompt: int
    generated: int
    step_mean: int
    step_min: int
    seed: int
    reading: str = "A"
    L_cap: int = 0  # rows per unit; 0 = choose from the reading

    def cap(self) -> int:
        if self.L_cap:
            return self.L_cap
        return 1024 if self.reading == "A" else self.prompt + self.generated + 64


def full_trace_spec(reading="A") -> TraceSpec:
    t = W.TRACE
    return TraceSpec(W.WORKLOADS[t["base"]], t["batch"], t["prompt"], t["generated"], t["step_mean"],
                     t["step_min"], t["seed"], reading)


@dataclass
class TraceEvents:
    """What the loop did, for replay and checks."""
    boundaries: list = field(default_factory=list)  # (token, [(seq, reward, keep)], stops)
    probes: list = field(default_factory=list)      # (token, seq, stopped)
    tokens: int = 0


class Trace:
    def __init__(self, spec: TraceSpec, device="cuda", out_dtype=torch.float32):
        self.spec = spec
        wl = spec.base.reduced(batch=spec.batch, L=spec.prompt, decode_steps=spec.cap() - spec.prompt,
                               seed=spec.seed)
        self.wl = wl
        self.device = device
        self.steps = W.make_trace_steps(spec.batch, spec.generated, spec.step_mean, spec.step_min, spec.seed)
        self.rewards = W.make_trace_rewards(self.steps, spec.seed)
        # token index at which each step of each sequence completes
        self.ends = [np.cumsum(s) - 1 for s in self.steps]
        self.K, self.V = W.make_cache(wl, device, canary=False)
        self.active = list(range(spec.batch))  # original sequence ids, in batch order
        self.lens = [spec.prompt] * spec.batch  # per active sequence (all its units share it)
        self.full = [spec.prompt] * spec.batch  # uncompressed length so far
        self.hist = [[] for _ in range(spec.batch)]
        self.step_idx = [0] * spec.batch
        self.out_dtype = out_dtype
        self.ids = torch.from_numpy(W.make_reflection_ids(wl)).to(device) if wl.vocab else None
        self._rebuild()

    # ---------------------------------------------------------------- inputs
    def token_inputs(self, t: int):
        """q [Ly, B, Hq, d], k_new / v_new [Ly, B, Hkv, d] for token t, full batch."""
        return W.make_decode_step(self.wl, 1000 + t, self.device)

    def window_queries(self, t: int):
        wl = self.wl
        return W.randn((wl.layers, wl.batch, wl.h_q, wl.w, wl.d), wl, 5_000_000 + t, self.device)

    def token_logits(self, t: int):
        return W.randn((self.wl.batch, self.wl.vocab), self.wl, 9_000_000 + t, self.device, torch.float32) * 2.0

    def answer(self, t: int, seq: int):
        """Answer logits / tokens of a probe of sequence `seq` at token t (confident on even probes)."""
        wl = self.wl.reduced(batch=1, seed=self.spec.seed * 7919 + t * 31 + seq)
        z, tok = W.make_answer(wl, self.device)
        if (t + seq) % 2:  # every other probe is not confident
            z = W.randn(z.shape, wl, 12, self.device, torch.float32) * 2.0
        return z, tok

    # ---------------------------------------------------------------- plumbing
    def _rebuild(self):
        wl = self.wl
        self.B = len(self.active)
        self.kv = reco.make_kv(self.K, self.V, wl.h_q)
        self.ws_score = reco.workspace(reco.RECO_OP_SCORE, self.kv, wl.w, self.device)
        self.ws_select = reco.workspace(reco.RECO_OP_SELECT, self.kv, wl.w, self.device)
        self.ws_decode = reco.workspace(reco.RECO_OP_DECODE, self.kv, 0, self.device)
        self.scores = torch.zeros(self.K.shape[:4], dtype=torch.float32, device=self.device)
        self.kept = torch.zeros(self.K.shape[:4], dtype=torch.int32, device=self.device)
        self.lens_dev = torch.tensor(self.lens, dtype=torch.int32, device=self.device).view(1, -1, 1).expand(
            wl.layers, -1, wl.h_kv).contiguous()
        self.ws_ppl = reco.workspace(reco.RECO_OP_PPL, None, wl.n_answer, self.device)

    def _drop(self, gone):
        keep_pos = [i for i, s in enumerate(self.active) if s not in gone]
        idx = torch.tensor(keep_pos, device=self.device)
        self.K = self.K.index_select(1, idx).contiguous()
        self.V = self.V.index_select(1, idx).contiguous()
        self.active = [self.active[i] for i in keep_pos]
        self.lens = [self.lens[i] for i in keep_pos]
        self.full = [self.full[i] for i in keep_pos]
        self._rebuild()

    def current_reward(self, s: int) -> float:
        return float(self.hist[s][-1]) if self.hist[s] else 0.0

    # ---------------------------------------------------------------- the loop
    def run(self, max_tokens=None, on_token=None, on_boundary=None) -> TraceEvents:
        spec, wl = self.spec, self.wl
        ev = TraceEvents()
        T = spec.generated if max_tokens is None else min(max_tokens, spec.generated)
        sel = lambda x: x.index_select(1, torch.tensor(self.active, device=self.device)).contiguous()  # noqa: E731
        for t in range(T):
            if not self.active:
                break
            q, kn, vn = self.token_inputs(t)
            q, kn, vn = sel(q), sel(kn), sel(vn)
            out = torch.empty(q.shape, dtype=self.out_dtype, device=self.device)
            lse = torch.empty(q.shape[:3], dtype=torch.float32, device=self.device)
            reco.reco_decode_attn(self.kv, q, kn, vn, self.lens_dev, wl.scale(), out, lse, self.ws_decode)
            self.lens = [L + 1 for L in self.lens]
            self.full = [F + 1 for F in self.full]
            logits = None
            if self.ids is not None:
                logits = self.token_logits(t).index_select(0, torch.tensor(self.active, device=self.device))
                rw = torch.tensor([self.current_reward(s) for s in self.active], dtype=torch.float32,
                                  device=self.device)
                reco.reco_reflect_penalty(logits, self.ids, rw, wl.tau_l, wl.tau_h, wl.beta)
            if on_token:
                on_token(t, self, out, lse, logits)
            ev.tokens += 1
            # step boundaries completed at this token
            done = []
            for i, s in enumerate(self.active):
                k = self.step_idx[s]
                if k < len(self.ends[s]) and self.ends[s][k] == t:
                    self.step_idx[s] += 1
                    self.hist[s].append(self.rewards[s][k])
                    done.append(i)
            if not done:
                continue
            keep = list(self.lens)
            info = []
            for i in done:
                s = self.active[i]
                ratio = reco.reco_retention_ratio(np.array(self.hist[s], np.float32), wl.base, wl.delta)
                base_len = self.lens[i] if spec.reading == "A" else self.full[i]
                m = reco.reco_keep_count(ratio, base_len, wl.w)
                keep[i] = min(m, self.lens[i])
                info.append((s, float(self.hist[s][-1]), keep[i]))
            q_win = sel(self.window_queries(t))
            keep_dev = torch.tensor(keep, dtype=torch.int32, device=self.device)
            reco.reco_score_cache(self.kv, q_win, self.lens_dev, wl.w, wl.pool, wl.scale(), self.scores,
                                  self.ws_score)
            reco.reco_select_compact(self.kv, self.scores, self.lens_dev, keep_dev, wl.w, self.kept,
                                     self.ws_select)
            if on_boundary:
                on_boundary(t, self, done, keep, q_win)
            self.lens = keep
            # early-stop probe (two consecutive top-band rewards)
            gone = set()
            for i in done:
                s = self.active[i]
                h = self.hist[s]
                if len(h) >= 2 and reco.reco_probe_trigger(float(h[-2]), float(h[-1]), wl.tau_h):
                    z, tok = self.answer(t, s)
                    ppl = torch.empty(1, device=self.device)
                    stop = torch.empty(1, dtype=torch.uint8, device=self.device)
                    reco.reco_answer_ppl(z, tok, None, wl.tau_p, ppl, stop, self.ws_ppl)
                    stopped = bool(stop.item())
                    ev.probes.append((t, s, stopped, float(ppl.item())))
                    if stopped:
                        gone.add(s)
            ev.boundaries.append((t, info, sorted(gone)))
            if gone:
                self._drop(gone)
        return ev
