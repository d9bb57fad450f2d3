"""One pass of the ReCo hot path over a batch, through the C ABI.

A step is what happens at one reasoning-step boundary and the decode that follows:
  1. Eq. 1 per sequence on the host (library helper) -> keep counts m_b
  2. reco_score_cache      (Eq. 2 scores, all layers in one call)
  3. reco_select_topm, reco_compact  (top-m per KV head, then in-place compaction:
     reco_select_compact's two halves as separate calls, so they can be timed apart)
  4. for each decode step: reco_decode_attn (append + attention over the ragged
     cache, all layers) and reco_reflect_penalty (Eq. 3-4 on the step's logits)
  5. reco_answer_ppl        (Eq. 5-6 probe over the answer logits)
Device state is allocated once; ``reset()`` restores the uncompressed cache so
every step starts from the same input.  PyTorch only provides memory and streams.
"""
from __future__ import annotations

import numpy as np
import torch

from . import reco
from . import workloads as W


class HotPath:
    def __init__(self, wl: W.Workload, device="cuda", out_dtype=torch.bfloat16, canary=False,
                 keep_pristine=True):
        self.wl = wl
        self.device = device
        dev = device
        self.K, self.V = W.make_cache(wl, dev, canary=canary)
        self.K0 = self.K.clone() if keep_pristine else None
        self.V0 = self.V.clone() if keep_pristine else None
        self.lens0 = W.make_lens(wl, dev)
        self.lens = self.lens0.clone()
        self.q_win = W.make_qwin(wl, dev)
        self.hist = W.make_reward_history(wl)
        self.rewards = torch.from_numpy(self.hist[:, -1].copy()).to(dev)
        self.keep_host = np.array(
            [reco.reco_keep_count(reco.reco_retention_ratio(self.hist[b], wl.base, wl.delta), wl.L, wl.w)
             for b in range(wl.batch)], np.int32)
        self.keep = torch.from_numpy(self.keep_host).to(dev)
        steps = wl.decode_steps
        qs, kns, vns = [], [], []
        for s in range(steps):
            q, kn, vn = W.make_decode_step(wl, s, dev)
            qs.append(q)
            kns.append(kn)
            vns.append(vn)
        self.dq = torch.stack(qs) if steps else None
        self.dk = torch.stack(kns) if steps else None
        self.dv = torch.stack(vns) if steps else None
        self.kv = reco.make_kv(self.K, self.V, wl.h_q)
        self.scores = torch.zeros(self.K.shape[:4], dtype=torch.float32, device=dev)
        self.kept = torch.zeros(self.K.shape[:4], dtype=torch.int32, device=dev)
        self.out = torch.empty((max(steps, 1), wl.layers, wl.batch, wl.h_q, wl.d), dtype=out_dtype, device=dev)
        self.lse = torch.empty((max(steps, 1), wl.layers, wl.batch, wl.h_q), dtype=torch.float32, device=dev)
        self.ws_score = reco.workspace(reco.RECO_OP_SCORE, self.kv, wl.w, dev)
        self.ws_select = reco.workspace(reco.RECO_OP_SELECT, self.kv, wl.w, dev)
        self.ws_decode = reco.workspace(reco.RECO_OP_DECODE, self.kv, 0, dev)
        self.has_vocab = wl.vocab > 0
        if self.has_vocab:
            self.logits = W.make_vocab_logits(wl, dev)
            self.ids = torch.from_numpy(W.make_reflection_ids(wl)).to(dev)
            self.beta = torch.empty(wl.batch, dtype=torch.float32, device=dev)
            self.ans_logits, self.ans_tokens = W.make_answer(wl, dev)
            self.ppl = torch.empty(wl.batch, dtype=torch.float32, device=dev)
            self.stop = torch.empty(wl.batch, dtype=torch.uint8, device=dev)
            self.ws_ppl = reco.workspace(reco.RECO_OP_PPL, None, wl.batch * wl.n_answer, dev)

    # ------------------------------------------------------------------ steps
    def reset(self):
        self.K.copy_(self.K0)
        self.V.copy_(self.V0)
        self.lens.copy_(self.lens0)

    def score(self, stream=None):
        wl = self.wl
        reco.reco_score_cache(self.kv, self.q_win, self.lens, wl.w, wl.pool, wl.scale(), self.scores,
                              self.ws_score, stream=stream)

    def select(self, stream=None):
        reco.reco_select_topm(self.kv, self.scores, self.lens, self.keep, self.wl.w, self.kept, self.ws_select,
                              stream)

    def compact(self, stream=None):
        reco.reco_compact(self.kv, self.kept, self.lens, self.keep, self.wl.w, stream)

    def compress(self, stream=None):
        self.score(stream)
        self.select(stream)
        self.compact(stream)

    def decode(self, s: int, stream=None):
        reco.reco_decode_attn(self.kv, self.dq[s], self.dk[s], self.dv[s], self.lens, self.wl.scale(),
                              self.out[s], self.lse[s], self.ws_decode, stream)

    def penalty(self, stream=None):
        wl = self.wl
        reco.reco_reflect_penalty(self.logits, self.ids, self.rewards, wl.tau_l, wl.tau_h, wl.beta,
                                  self.beta, stream)

    def probe(self, stream=None):
        reco.reco_answer_ppl(self.ans_logits, self.ans_tokens, None, self.wl.tau_p, self.ppl, self.stop,
                             self.ws_ppl, stream)

    def step(self, stream=None, decode_events=None):
        """The whole hot path once.  decode_events: optional list of (start, end) CUDA
        event pairs recorded around each decode launch."""
        self.compress(stream)
        for s in range(self.wl.decode_steps):
            if decode_events is not None:
                decode_events[s][0].record(stream)
            self.decode(s, stream)
            if decode_events is not None:
                decode_events[s][1].record(stream)
            if self.has_vocab:
                self.penalty(stream)
        if self.has_vocab:
            self.probe(stream)

    def launches_per_step(self) -> int:
        """Library kernels launched by one step."""
        n = 4 + 3  # score: pass 1, combine, pass 2, pool; select; compact and its length update
        n += self.wl.decode_steps * (1 + (1 if self.has_vocab else 0))
        n += 2 if self.has_vocab else 0
        return n
