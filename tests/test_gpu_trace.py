"""The step-loop trace (ragged step boundaries, compression at every boundary,
decode between, penalty and a draw every token, answer probe on two top-band rewards,
stopped sequences leaving the batch) replayed in lock-step by the oracle.  Eq. 2's window
queries are the last w decoded tokens' queries; the library scores a boundary in one pass
from their decode lse when it can, and the oracle always from its own normalisers.

The oracle keeps its own float64-computed cache state from the same seeded inputs
(never from the GPU's results) and checks, at every token, every decode output, the
penalised logits and the sampled tokens (equal up to the boundary band), at every
boundary the scores and kept sets of the sequences that compress, and every probe's
PPL and stop decision."""
import numpy as np
import pytest
import torch

import oracle
from helpers import DECODE_ATOL, PPL_RTOL, assert_kept_match, assert_scores_close, assert_tokens_valid, np32
from paper_2608_04771_gb300 import reco, trace
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


class OracleReplay:
    """Follows the sequences in `track` (all by default); each sequence's cache evolves
    independently of the others, so a subset can be replayed on its own."""

    def __init__(self, tr: trace.Trace, track=None, decode_every=1):
        wl = tr.wl
        self.wl = wl
        self.track = set(range(tr.spec.batch)) if track is None else set(track)
        self.decode_every = decode_every
        self.K = np32(tr.K).astype(np.float32)  # [Ly, B, Hkv, L_cap, d], original batch order
        self.V = np32(tr.V).astype(np.float32)
        self.lens = {s: tr.spec.prompt for s in range(tr.spec.batch)}
        self.last_comp = {s: tr.spec.prompt for s in range(tr.spec.batch)}
        self.hist = {s: [] for s in range(tr.spec.batch)}
        self.ids = W.make_reflection_ids(wl)
        self.checked_tokens = 0
        self.checked_boundaries = 0
        self.tie_diffs = 0
        self.diverged = set()  # (seq, layer, kv head) whose kept set differed within the tie band
        self.expected_probes = set()
        self.sampled = 0  # draws checked
        # cache bytes held after every token, from the replay's own lengths (Table 3's
        # memory, cache only): K and V rows of every layer and KV head of the active sequences
        self.row_bytes = 2 * wl.layers * wl.h_kv * wl.d * wl.elem_bytes
        self.peak_bytes = 0
        self.byte_tokens = 0

    def on_token(self, t, tr, out, lse, logits):
        wl = self.wl
        pos = [i for i, s in enumerate(tr.active) if s in self.track]  # batch positions followed
        act = [tr.active[i] for i in pos]
        if not act:
            return
        q, kn, vn = (np32(x) for x in tr.token_inputs(t))
        for s in act:
            L = self.lens[s]
            self.K[:, s, :, L] = kn[:, s]
            self.V[:, s, :, L] = vn[:, s]
            self.lens[s] = L + 1
        held = sum(self.lens[s] for s in act) * self.row_bytes
        self.peak_bytes = max(self.peak_bytes, held)
        self.byte_tokens += held
        # the device's lengths after the decode's append are the replay's, on every layer and head
        dev_lens = tr.lens_dev.cpu().numpy()
        for i, s in zip(pos, act):
            assert (dev_lens[:, i, :] == self.lens[s]).all(), (t, s, self.lens[s])
        if t % self.decode_every == 0:
            lens = np.array([[[self.lens[s]] * wl.h_kv for s in act]] * wl.layers, np.int32)
            o_ref, lse_ref = oracle.decode_batch(q[:, act], self.K[:, act], self.V[:, act], lens, wl.scale())
            got = out[:, pos].float().cpu().numpy()
            ok = np.ones(got.shape[:3], bool)  # [layer, seq, query head]: skip diverged units
            for j, s in enumerate(act):
                for (s2, l, h) in self.diverged:
                    if s2 == s:
                        ok[l, j, h * wl.G:(h + 1) * wl.G] = False
            assert (np.abs(got - o_ref)[ok] <= DECODE_ATOL[wl.dtype]).all(), f"token {t}: decode"
            assert np.abs(lse[:, pos].cpu().numpy() - lse_ref)[ok].max(initial=0) < 1e-3
            if logits is not None:
                z = np32(tr.token_logits(t))[act]
                rw = np.array([self.hist[s][-1] if self.hist[s] else 0.0 for s in act], np.float32)
                ref, _, _ = oracle.reflect_penalty(z, self.ids, rw, wl.tau_l, wl.tau_h, wl.beta)
                np.testing.assert_array_equal(logits[pos].cpu().numpy().view(np.uint32), ref.view(np.uint32))
                u = tr.token_draws(t).cpu().numpy()[act]
                _, tref, _, _, _ = oracle.penalty_sample(z, self.ids, rw, u, wl.tau_l, wl.tau_h, wl.beta)
                assert_tokens_valid(tr.tokens[pos].cpu().numpy(), ref, u, tref, max_inexact=1)
                self.sampled += len(act)
            self.checked_tokens += 1

    def on_boundary(self, t, tr, done, keep, q_win):
        wl = self.wl
        act = list(tr.active)
        qw = np32(q_win) if q_win is not None else None
        got_kept = tr.kept.cpu().numpy()
        got_scores = tr.scores.cpu().numpy()
        for i in done:
            s = act[i]
            if s not in self.track:
                continue
            self.hist[s].append(tr.rewards[s][len(self.hist[s])])  # the generator's k-th step reward
            hs = self.hist[s]
            if len(hs) >= 2 and oracle.probe_trigger(hs[-2], hs[-1], wl.tau_h):
                self.expected_probes.add((t, s))
            L = self.lens[s]
            if L - self.last_comp[s] < tr.spec.interval:  # grown by less than S: no compression
                assert keep[i] == L
                continue
            ratio = oracle.retention_ratio(np.array(hs, np.float32), wl.base, wl.delta)
            base_len = L if tr.spec.reading == "A" else tr.spec.prompt + t + 1
            m = min(oracle.keep_count(ratio, base_len, wl.w), L)
            assert m == keep[i], (t, s, m, keep[i])
            lens1 = np.full((wl.layers, 1, wl.h_kv), L, np.int32)
            pooled_all = oracle.score_cache(qw[:, i:i + 1], self.K[:, s:s + 1], lens1, wl.w, wl.pool, wl.scale())
            for l in range(wl.layers):
                for h in range(wl.h_kv):
                    pooled = pooled_all[l, 0, h, :L - wl.w]
                    idx = oracle.select_unit(pooled.astype(np.float32), L, wl.w, m)
                    if (s, l, h) not in self.diverged:
                        if m < L:  # m == L keeps everything: the library skips that sequence's scoring
                            assert_scores_close(got_scores[l, i, h, :L - wl.w], pooled, f"t {t} seq {s}")
                        nd = assert_kept_match(got_kept[l, i, h], idx, pooled, L, wl.w, m)
                        if nd:  # a near-tie decided the other way: this unit's two caches now differ
                            self.tie_diffs += nd
                            self.diverged.add((s, l, h))
                    self.K[l, s, h, :m] = oracle.gather_unit(self.K[l, s, h, :L], idx)
                    self.V[l, s, h, :m] = oracle.gather_unit(self.V[l, s, h, :L], idx)
            self.lens[s] = m
            self.last_comp[s] = m
        self.checked_boundaries += 1


def _run(spec, track=None, decode_every=1, use_graph=False, input_pool=0):
    tr = trace.Trace(spec, DEV, use_graph=use_graph, input_pool=input_pool)
    rep = OracleReplay(tr, track, decode_every)
    ev = tr.run(on_token=rep.on_token, on_boundary=rep.on_boundary)
    reco.reco_check()
    assert {(t, s) for (t, s, _, _) in ev.probes if s in rep.track} == rep.expected_probes
    # every probe: PPL and the stop decision against the oracle
    for (t, s, stopped, ppl) in ev.probes:
        z, tok = tr.answer(t, s)
        p_ref, stop_ref = oracle.answer_ppl(np32(z), tok.cpu().numpy(), None, spec.base.tau_p)
        assert abs(ppl - p_ref[0]) <= PPL_RTOL * p_ref[0]
        assert stopped == bool(stop_ref[0])
    if track is None:  # every sequence followed: the trace's cache-bytes counters are the replay's
        assert ev.peak_cache_bytes == rep.peak_bytes > 0
        assert ev.cache_byte_tokens == rep.byte_tokens
    return tr, rep, ev


@pytest.mark.parametrize("use_graph,input_pool", [(False, 0), (True, 0), (True, 32)])
def test_trace_reading_A_reduced(use_graph, input_pool):
    # tau_h 0.6 so that this seed's Beta(2,2) rewards trigger probes (4 probes, 3 stops)
    base = W.WORKLOADS["7b"].reduced(layers=2, vocab=5000, tau_h=0.6)
    spec = trace.TraceSpec(base, batch=4, prompt=128, generated=400, step_mean=40, step_min=8, seed=4,
                           reading="A")
    tr, rep, ev = _run(spec, use_graph=use_graph, input_pool=input_pool)
    assert rep.tie_diffs == 0  # no near-tie flips on this seed: every unit compared throughout
    assert rep.checked_tokens >= 150 and rep.checked_boundaries >= 15
    assert len(ev.probes) == 4 and sum(st for (_, _, st, _) in ev.probes) == 3
    # steps of at least w tokens score in one pass from the decode's lse, shorter ones in two
    assert ev.lse_scorings > 0 and ev.two_pass_scorings > 0


def test_trace_interval_trigger():
    """Compress only once the cache has grown by S = 100 tokens since the last compression."""
    base = W.WORKLOADS["7b"].reduced(layers=1, vocab=2000)
    spec = trace.TraceSpec(base, batch=3, prompt=64, generated=420, step_mean=30, step_min=8, seed=7,
                           reading="A", interval=100)
    tr, rep, ev = _run(spec)
    assert rep.tie_diffs == 0
    assert 0 < ev.compressions < ev.steps_completed  # some boundaries skip compression
    assert ev.generated > 0


def test_trace_reading_B_reduced_with_stops():
    base = W.WORKLOADS["7b"].reduced(layers=1, vocab=3000, tau_h=0.55)  # lower tau_h: more probes, stops
    spec = trace.TraceSpec(base, batch=4, prompt=96, generated=500, step_mean=30, step_min=8, seed=6,
                           reading="B")
    tr, rep, ev = _run(spec)
    assert rep.tie_diffs == 0
    assert any(stopped for (_, _, stopped, _) in ev.probes), "expected at least one early stop"
    assert len(tr.active) < 4


def test_trace_full_size_sampled():
    """The full step-loop workload (7B-class heads, 28 layers, batch 16, prompt 256, 8192
    generated tokens, steps of Poisson(96)+16, Beta(2,2) rewards, reading A) with the
    oracle following two whole sequences (decode checked every 8th token, every boundary)."""
    spec = trace.full_trace_spec("A")
    tr, rep, ev = _run(spec, track=[0, 9], decode_every=8, use_graph=True)
    assert rep.checked_boundaries >= 100 and rep.checked_tokens >= 100
    # near-tie flips (fp32 vs fp64 scores within 1e-5 of the cut) stop the comparison of that unit only
    assert len(rep.diverged) <= 0.05 * 2 * spec.base.layers * spec.base.h_kv, rep.diverged
    assert ev.lse_scorings > 10 * ev.two_pass_scorings  # steps are Poisson(96)+16 >> w tokens


def test_trace_cache_bytes_without_compression():
    """With compression switched off by the interval trigger (S larger than any growth) the
    cache holds every token: the peak is the closed form B * (prompt + generated) rows and the
    per-token sum is B * sum_t (prompt + t + 1) rows."""
    base = W.WORKLOADS["7b"].reduced(layers=1, vocab=2000, tau_h=1.5)  # no probe: every sequence runs on
    spec = trace.TraceSpec(base, batch=3, prompt=64, generated=150, step_mean=30, step_min=8, seed=7,
                           reading="A", interval=10_000)
    tr, rep, ev = _run(spec, decode_every=50)
    assert ev.compressions == 0
    row = 2 * base.layers * base.h_kv * base.d * base.elem_bytes
    assert ev.peak_cache_bytes == 3 * (64 + 150) * row
    assert ev.cache_byte_tokens == 3 * sum(64 + t + 1 for t in range(150)) * row
