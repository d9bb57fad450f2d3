"""The step loop of ReCo over a synthetic reasoning trace, through the C ABI.

Each sequence generates tokens one at a time; its trajectory is split into steps of
Poisson(mean) + min tokens (Sec. 3.1 splits at newlines; the lengths here are
synthetic).  Per token, every active sequence decodes one token (append + attention
over its ragged cache, all layers in one call) and the reflection penalty (Eq. 3-4)
is applied to that token's logits with the band of the sequence's latest reward.
When a sequence completes a step it receives a reward v_i (Sec. 3.1), and
  * if its cache has grown by at least S tokens since its last compression
    (L - L_{i-1} >= S, Sec. 3.2; L_0 = the prompt; S = 0 compresses at every
    step boundary) it is compressed to m_i = lambda_i * L (Eq. 1-2, Sec. 3.2) --
    all sequences are passed to one scoring/selection call, the others with
    keep = L, which leaves them untouched;
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
    interval: int = 0  # S: minimum growth since the last compression (0: every step boundary)

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
    probes: list = field(default_factory=list)      # (token, seq, stopped, ppl)
    tokens: int = 0            # decode launches (loop iterations)
    generated: int = 0         # tokens generated, summed over sequences
    steps_completed: int = 0   # step boundaries, summed over sequences
    compressions: int = 0      # per-sequence compressions
    peak_cache_bytes: int = 0  # max over tokens of the K+V bytes held by the active sequences
    cache_byte_tokens: float = 0.0  # sum over tokens of the K+V bytes held (for the mean)


class Trace:
    def __init__(self, spec: TraceSpec, device="cuda", out_dtype=torch.float32, input_pool: int = 0):
        """input_pool > 0: per-token inputs are drawn once for that many tokens and reused
        cyclically (timing runs); 0: every token draws its own seeded inputs."""
        self.spec = spec
        self.input_pool = input_pool
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
        self.last_comp = [spec.prompt] * spec.batch  # L_{i-1}: length after the last compression
        self.step_idx = [0] * spec.batch
        self.out_dtype = out_dtype
        self.ids = torch.from_numpy(W.make_reflection_ids(wl)).to(device) if wl.vocab else None
        self._pool = None
        if input_pool:
            self._pool = [(self._token_inputs(t), self._window_queries(t) if t < 8 else None,
                           self._token_logits(t) if wl.vocab else None) for t in range(input_pool)]
        self._rebuild()

    # ---------------------------------------------------------------- inputs
    def _token_inputs(self, t: int):
        return W.make_decode_step(self.wl, 1000 + t, self.device)

    def _window_queries(self, t: int):
        wl = self.wl
        return W.randn((wl.layers, wl.batch, wl.h_q, wl.w, wl.d), wl, 5_000_000 + t, self.device)

    def _token_logits(self, t: int):
        return W.randn((self.wl.batch, self.wl.vocab), self.wl, 9_000_000 + t, self.device, torch.float32) * 2.0

    def token_inputs(self, t: int):
        """q [Ly, B, Hq, d], k_new / v_new [Ly, B, Hkv, d] for token t, full batch."""
        return self._pool[t % self.input_pool][0] if self._pool else self._token_inputs(t)

    def window_queries(self, t: int):
        return self._pool[t % 8][1] if self._pool else self._window_queries(t)

    def token_logits(self, t: int):
        return self._pool[t % self.input_pool][2].clone() if self._pool else self._token_logits(t)

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
        self.last_comp = [self.last_comp[i] for i in keep_pos]
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
            ev.generated += len(self.active)
            row_bytes = 2 * wl.layers * wl.h_kv * wl.d * wl.elem_bytes  # K and V of one token
            held = sum(self.lens) * row_bytes
            ev.peak_cache_bytes = max(ev.peak_cache_bytes, held)
            ev.cache_byte_tokens += held
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
            ev.steps_completed += len(done)
            keep = list(self.lens)
            info = []
            for i in done:
                s = self.active[i]
                if self.lens[i] - self.last_comp[i] < spec.interval:
                    continue  # grown by less than S since the last compression
                ratio = reco.reco_retention_ratio(np.array(self.hist[s], np.float32), wl.base, wl.delta)
                base_len = self.lens[i] if spec.reading == "A" else self.full[i]
                m = reco.reco_keep_count(ratio, base_len, wl.w)
                keep[i] = min(m, self.lens[i])
                self.last_comp[i] = keep[i]
                info.append((s, float(self.hist[s][-1]), keep[i]))
                ev.compressions += 1
            q_win = None
            if info:
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
