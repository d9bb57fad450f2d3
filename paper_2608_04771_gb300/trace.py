"""The step loop of ReCo over a synthetic reasoning trace, through the C ABI.

Each sequence generates tokens one at a time; its trajectory is split into steps of
Poisson(mean) + min tokens (Sec. 3.1 splits at newlines; the lengths here are
synthetic).  Per token, every active sequence decodes one token (append + attention
over its ragged cache, all layers in one call), the reflection penalty (Eq. 3-4) is
applied to that token's logits with the band of the sequence's latest reward, and the
next token is drawn from softmax of the penalised logits (Sec. 3.3) at a seeded
uniform draw.
When a sequence completes a step it receives a reward v_i (Sec. 3.1), and
  * if its cache has grown by at least S tokens since its last compression
    (L - L_{i-1} >= S, Sec. 3.2; L_0 = the prompt; S = 0 compresses at every
    step boundary) it is compressed to m_i = lambda_i * L (Eq. 1-2, Sec. 3.2) --
    all sequences are passed to one scoring/selection call, the others with
    keep = L, which skips their scoring and leaves them untouched;
  * if v_{i-1} >= tau_h and v_i >= tau_h, the answer probe runs (Eq. 5-6) and a
    sequence that passes PPL <= tau_p stops and leaves the batch.
Eq. 2's observation window is the queries of the last w decoded tokens.  Those queries
and the lse each decode returns are kept in device rings of w slots, written by every
token; when none of the sequences compressed at a boundary was compressed within its
window, those lse are the window rows' normalisers and the scores take one pass over K
(reco_score_cache_lse), else two (reco_score_cache).
Budget base L (the paper is silent on repeated compression): reading "A" uses the
current cache length, reading "B" the full uncompressed length so far (the keep
count is then capped at the current length).  Lengths are tracked on the host, so
the loop needs no device read-back except the stop flags of a probe.

With use_graph, a token's decode, penalty, draw and lse push are one captured CUDA
graph over static input buffers (captured again whenever the batch shrinks), so the
per-token host work is one graph launch (with an input pool, the graph also gathers
the token's inputs); a boundary uploads keep counts and rewards and launches the
scoring and selection, with no host-side gather of the window.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np
import torch

from . import reco
from . import workloads as W


def _pack(parts, out=None):
    """Lay tensors end to end in one uint8 buffer (each part 256-byte aligned); returns the
    buffer and a view of each part in it.  With `out`, views into `out` are made instead
    (the parts then only give shapes and dtypes)."""
    offs, n = [], 0
    for x in parts:
        offs.append(n)
        n += (x.numel() * x.element_size() + 255) // 256 * 256
    buf = out if out is not None else torch.empty(n, dtype=torch.uint8, device=parts[0].device)
    views = []
    for x, o in zip(parts, offs):
        v = buf[o:o + x.numel() * x.element_size()].view(x.dtype).view(x.shape)
        if out is None:
            v.copy_(x)
        views.append(v)
    return buf, views


class _Staging:
    """Small host -> device copies (keep counts, rewards) through a ring of pinned host
    slots.  A slot is written again only after the copy that last read it has completed
    (one event per slot), so the host never blocks on a busy GPU queue and never
    allocates pinned memory in the loop.  A device slot is reused only by a later copy on
    the same stream, after every kernel that read it."""

    def __init__(self, n_max: int, device, n_slots: int = 64):
        self.host = torch.zeros((n_slots, n_max), dtype=torch.int32).pin_memory()
        self.host_np = self.host.numpy()
        self.dev = torch.zeros((n_slots, n_max), dtype=torch.int32, device=device)
        self.events = [torch.cuda.Event() for _ in range(n_slots)]
        self.stream = torch.cuda.current_stream(device)
        self.used = [False] * n_slots
        self.next = 0

    def put(self, values, dtype, out=None) -> torch.Tensor:
        """Copy `values` to the device (into `out` if given, else a ring slot)."""
        i = self.next
        self.next = (i + 1) % len(self.events)
        if self.used[i]:
            self.events[i].synchronize()
        n = len(values)
        self.host_np[i, :n] = np.asarray(values, dtype=np.int32 if dtype == torch.int32 else np.float32).view(np.int32)
        src = self.host[i, :n].view(dtype)
        dst = out if out is not None else self.dev[i, :n].view(dtype)
        dst.copy_(src, non_blocking=True)
        self.events[i].record(self.stream)
        self.used[i] = True
        return dst


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
    lse_scorings: int = 0      # boundary scorings in one pass, normalisers from the decode
    two_pass_scorings: int = 0  # boundary scorings in two passes (a window not all decoded since)


class Trace:
    def __init__(self, spec: TraceSpec, device="cuda", out_dtype=torch.float32, input_pool: int = 0,
                 use_graph: bool = False):
        """input_pool = w (the window): per-token inputs are drawn once for w tokens and
        reused cyclically (timing runs); 0: every token draws its own seeded inputs.
        use_graph: the per-token decode + penalty runs as a captured CUDA graph."""
        self.spec = spec
        self.input_pool = input_pool
        self.use_graph = use_graph
        self.graph = None
        wl = spec.base.reduced(batch=spec.batch, L=spec.prompt, decode_steps=spec.cap() - spec.prompt,
                               seed=spec.seed)
        self.wl = wl
        self.device = device
        self.steps = W.make_trace_steps(spec.batch, spec.generated, spec.step_mean, spec.step_min, spec.seed)
        self.rewards = W.make_trace_rewards(self.steps, spec.seed)
        # token index at which each step of each sequence completes, and its inverse
        # (token -> the sequences that complete a step there)
        self.ends = [np.cumsum(s) - 1 for s in self.steps]
        self.ends_at = {}
        for sq, e in enumerate(self.ends):
            for tok in e.tolist():
                self.ends_at.setdefault(tok, []).append(sq)
        self.K, self.V = W.make_cache(wl, device, canary=False)
        self.active = list(range(spec.batch))  # original sequence ids, in batch order
        self.lens = [spec.prompt] * spec.batch  # per active sequence (all its units share it)
        self.full = [spec.prompt] * spec.batch  # uncompressed length so far
        self.hist = [[] for _ in range(spec.batch)]
        self.last_comp = [spec.prompt] * spec.batch  # L_{i-1}: length after the last compression
        self.step_idx = [0] * spec.batch
        self.out_dtype = out_dtype
        self.ids = torch.from_numpy(W.make_reflection_ids(wl)).to(device) if wl.vocab else None
        self.staging = _Staging(3 * spec.batch + wl.w, device)
        self._pool = None
        self._answers = {}
        if input_pool:
            # every slot's inputs stacked on a leading slot axis: [P, Ly, B, ...], [P, B, V]
            ins = [self._token_inputs(t) for t in range(input_pool)]
            self._pool = (torch.stack([x[0] for x in ins]), torch.stack([x[1] for x in ins]),
                          torch.stack([x[2] for x in ins]),
                          torch.stack([self._token_logits(t) for t in range(input_pool)]) if wl.vocab else None,
                          torch.stack([self._token_draws(t) for t in range(input_pool)]) if wl.vocab else None)
            del ins
            # the answers of every probe the rewards can trigger, drawn before the loop runs
            for sq in range(spec.batch):
                r = np.asarray(self.rewards[sq], np.float32)
                for k in range(1, len(r)):
                    t = int(self.ends[sq][k])
                    if t < spec.generated and r[k - 1] >= np.float32(wl.tau_h) and r[k] >= np.float32(wl.tau_h):
                        self._answers[(t, sq)] = self._answer(t, sq)
        # The window ring: the queries (q_win, slot t % w of every head's w rows) and the
        # decode's lse (ring row t % w, mirrored in row t % w + w) of the last w tokens, kept
        # by every token on the device; one device counter (slot_dev = t % w) also selects
        # the input-pool slot.  Per active sequence, `since` counts the tokens decoded since
        # its last compression: Eq. 2's window rows are those tokens' queries, and their lse
        # are the rows' normalisers while the cache has not been compressed since they were
        # decoded.  In that one-pass form Eq. 2 sums the same rows whatever their order (every
        # candidate key precedes the whole window), so the ring is scored in slot order; the
        # two-pass form (causal row normalisers) gets the window rotated into token order.
        self.R = wl.w
        if input_pool and input_pool != self.R:
            raise ValueError(f"input_pool must be 0 or the window w = {self.R} (one counter selects both)")
        self.lse_ring = torch.zeros((2 * self.R, wl.layers, spec.batch, wl.h_q), dtype=torch.float32,
                                    device=device)
        self.slot_dev = torch.zeros(1, dtype=torch.long, device=device)
        self._slot_t = -1  # the token whose ring slot slot_dev holds
        self.since = [0] * spec.batch
        self._rebuild()

    # ---------------------------------------------------------------- inputs
    def _token_inputs(self, t: int):
        return W.make_decode_step(self.wl, 1000 + t, self.device)

    def _token_logits(self, t: int):
        return W.randn((self.wl.batch, self.wl.vocab), self.wl, 9_000_000 + t, self.device, torch.float32) * 2.0

    def token_inputs(self, t: int):
        """q [Ly, B, Hq, d], k_new / v_new [Ly, B, Hkv, d] for token t, full batch."""
        if self._pool:
            i = t % self.input_pool
            return self._pool[0][i], self._pool[1][i], self._pool[2][i]
        return self._token_inputs(t)

    def token_logits(self, t: int):
        return self._pool[3][t % self.input_pool].clone() if self._pool else self._token_logits(t)

    def _token_draws(self, t: int):
        return torch.from_numpy(W.make_draws(self.wl, self.wl.batch, 7_000_000 + t)).to(self.device)

    def token_draws(self, t: int):
        """[B] uniform draws of token t's sampling step, full batch."""
        return self._pool[4][t % self.input_pool] if self._pool else self._token_draws(t)

    def answer(self, t: int, seq: int):
        """Answer logits / tokens of a probe of sequence `seq` at token t (confident on even probes)."""
        got = self._answers.get((t, seq))
        return got if got is not None else self._answer(t, seq)

    def _answer(self, t: int, seq: int):
        wl = self.wl.reduced(batch=1, seed=self.spec.seed * 7919 + t * 31 + seq)
        z, tok = W.make_answer(wl, self.device)
        if (t + seq) % 2:  # every other probe is not confident
            z = W.randn(z.shape, wl, 12, self.device, torch.float32) * 2.0
        return z, tok

    def _full_batch(self) -> bool:
        return len(self.active) == self.spec.batch

    def _sel(self, x, dim=1):
        """Rows of the active sequences (batch dimension `dim`), in batch order."""
        return x if self._full_batch() else x.index_select(dim, self.idx_dev).contiguous()

    def active_inputs(self, t: int):
        """Token t's q, k_new, v_new for the active sequences."""
        if self._apool is not None:
            return tuple(self._slot_view(t % self.input_pool, k) for k in range(3))
        q, kn, vn = self._token_inputs(t)
        return self._sel(q), self._sel(kn), self._sel(vn)

    def active_logits(self, t: int):
        """A fresh copy of token t's logits rows of the active sequences."""
        if self._apool is not None:
            return self._slot_view(t % self.input_pool, 3).clone()
        return self._sel(self._token_logits(t), 0)

    def active_draws(self, t: int):
        if self._apool is not None:
            return self._slot_view(t % self.input_pool, 4)
        return self._sel(self._token_draws(t), 0)

    def _window_in_token_order(self, t: int):
        """q_win rotated so that row k holds the query of token t - w + 1 + k (the two-pass
        scoring's causal row normalisers depend on the row's position)."""
        return torch.roll(self.q_win, shifts=-((t + 1) % self.R), dims=3)

    # ---------------------------------------------------------------- plumbing
    def _active_pool(self):
        """The input pool restricted to the active sequences (one gather per input over all
        slots).  Slot i's q | k_new | v_new | logits are packed in row i of one byte matrix,
        laid out like the captured graph's static inputs (each part 256-byte aligned), so a
        token's inputs arrive in a single copy."""
        if not self._pool:
            return None
        P = self.input_pool
        Q, KN, VN, Z, U = self._pool
        sel = (lambda x, d: x) if self._full_batch() else (lambda x, d: x.index_select(d, self.idx_dev))
        parts = [sel(Q, 2), sel(KN, 2), sel(VN, 2)] + ([] if Z is None else [sel(Z, 1), sel(U, 1)])
        self._slot_meta, cols, off = [], [], 0
        for x in parts:
            nb = x[0].numel() * x.element_size()
            cols.append(x.reshape(P, -1).contiguous().view(torch.uint8))
            pad = (nb + 255) // 256 * 256 - nb
            if pad:
                cols.append(torch.zeros((P, pad), dtype=torch.uint8, device=x.device))
            self._slot_meta.append((off, nb, x.dtype, tuple(x.shape[1:])))
            off += nb + pad
        return torch.cat(cols, dim=1)

    def _slot_view(self, i: int, k: int):
        off, nb, dt, shape = self._slot_meta[k]
        return self._apool[i, off:off + nb].view(dt).view(shape)

    def _rebuild(self):
        wl = self.wl
        self.B = len(self.active)
        self.pos = {sq: i for i, sq in enumerate(self.active)}  # sequence id -> batch position
        self.idx_dev = torch.tensor(self.active, dtype=torch.long, device=self.device)
        self._apool = None
        self._apool = self._active_pool()
        self.kv = reco.make_kv(self.K, self.V, wl.h_q)
        self.ws_score = reco.workspace(reco.RECO_OP_SCORE, self.kv, wl.w, self.device)
        self.ws_select = reco.workspace(reco.RECO_OP_SELECT, self.kv, wl.w, self.device)
        self.ws_decode = reco.workspace(reco.RECO_OP_DECODE, self.kv, 0, self.device)
        self.scores = torch.zeros(self.K.shape[:4], dtype=torch.float32, device=self.device)
        self.kept = torch.zeros(self.K.shape[:4], dtype=torch.int32, device=self.device)
        self.q_win = torch.zeros((wl.layers, self.B, wl.h_q, wl.w, wl.d), dtype=wl.torch_dtype, device=self.device)
        self.lens_dev = torch.tensor(self.lens, dtype=torch.int32, device=self.device).view(1, -1, 1).expand(
            wl.layers, -1, wl.h_kv).contiguous()
        self.ws_ppl = reco.workspace(reco.RECO_OP_PPL, None, wl.n_answer, self.device)
        self.ws_sample = reco.sample_workspace(self.B, wl.vocab, self.device) if wl.vocab else None
        self.tokens = None  # the last token's draws, [active] int32
        self.graph = None  # buffers and pointers changed: capture again before the next token

    def _drop(self, gone):
        keep_pos = [i for i, s in enumerate(self.active) if s not in gone]
        idx = torch.tensor(keep_pos, device=self.device)
        self.K = self.K.index_select(1, idx).contiguous()
        self.V = self.V.index_select(1, idx).contiguous()
        self.active = [self.active[i] for i in keep_pos]
        self.lens = [self.lens[i] for i in keep_pos]
        self.full = [self.full[i] for i in keep_pos]
        self.last_comp = [self.last_comp[i] for i in keep_pos]
        self.since = [self.since[i] for i in keep_pos]
        self.lse_ring = self.lse_ring.index_select(2, idx).contiguous()
        q_win = self.q_win.index_select(1, idx)
        self._rebuild()
        self.q_win.copy_(q_win)

    def _capture(self, t: int):
        """Static input/output buffers and one CUDA graph of a token's decode + penalty.
        With an input pool the graph also gathers its token's inputs (slot slot_dev of
        the packed pool) and advances slot_dev, so a token costs the host one launch."""
        wl, dev, B = self.wl, self.device, len(self.active)
        shapes = [((wl.layers, B, wl.h_q, wl.d), wl.torch_dtype), ((wl.layers, B, wl.h_kv, wl.d), wl.torch_dtype),
                  ((wl.layers, B, wl.h_kv, wl.d), wl.torch_dtype)]
        if self.ids is not None:
            shapes += [((B, wl.vocab), torch.float32), ((B,), torch.float32)]
        protos = [torch.empty(sh, dtype=dt, device="meta") for sh, dt in shapes]
        n = sum((x.numel() * x.element_size() + 255) // 256 * 256 for x in protos)
        self.g_in = torch.zeros(n, dtype=torch.uint8, device=dev)  # q | k_new | v_new | logits
        _, views = _pack(protos, out=self.g_in)
        self.g_q, self.g_kn, self.g_vn = views[:3]
        self.g_logits = views[3] if self.ids is not None else None
        self.g_u = views[4] if self.ids is not None else None
        self.g_tok = torch.full((B,), -1, dtype=torch.int32, device=dev)
        self.g_out = torch.empty(self.g_q.shape, dtype=self.out_dtype, device=dev)
        self.g_lse = torch.empty(self.g_q.shape[:3], dtype=torch.float32, device=dev)
        # keep counts | current rewards (float32 bits) | window slots and rows: one upload
        self.g_small = torch.zeros(3 * B + wl.w, dtype=torch.int32, device=dev)
        self.g_rw = self.g_small[B:2 * B].view(torch.float32)
        self._put_small(list(self.lens))
        # one call outside the capture, without an append (cache and lens stay as they are)
        reco.reco_decode_attn(self.kv, self.g_q, None, None, self.lens_dev, wl.scale(), self.g_out, self.g_lse,
                              self.ws_decode)
        torch.cuda.synchronize()
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, capture_error_mode="relaxed"):
            if self._apool is not None:
                # the token's packed inputs: pool row slot_dev (every part a multiple of
                # 256 bytes), selected on the device
                reco.reco_copy_row(self._apool, self.slot_dev, self.g_in)
            # the token's lse and queries go straight into the window rings, and the decode
            # advances the slot (the next token's pool slot)
            reco.reco_decode_attn_ring(self.kv, self.g_q, self.g_kn, self.g_vn, self.lens_dev, wl.scale(), self.g_out,
                                       self.lse_ring, self.slot_dev, self.ws_decode, q_ring=self.q_win)
            if self.g_logits is not None:
                reco.reco_penalty_sample(self.g_logits, self.ids, self.g_rw, self.g_u, self.g_tok, self.ws_sample,
                                         wl.tau_l, wl.tau_h, wl.beta)
        self.slot_dev.fill_(t % self.R)
        self._slot_t = t
        self.graph = g

    def _put_small(self, keep):
        """Upload keep counts and the active sequences' current rewards into g_small in one
        copy; returns the device view written."""
        rw = np.asarray([self.current_reward(s) for s in self.active], np.float32).view(np.int32)
        vals = np.concatenate([np.asarray(keep, np.int32), rw])
        return self.staging.put(vals, torch.int32, out=self.g_small[:len(vals)])

    def current_reward(self, s: int) -> float:
        return float(self.hist[s][-1]) if self.hist[s] else 0.0

    # ---------------------------------------------------------------- the loop
    def _token(self, t: int):
        """Decode (append + attention) and penalty of token t; returns out, lse, logits."""
        wl = self.wl
        if self._slot_t != t:  # first token after a (re)build
            self.slot_dev.fill_(t % self.R)
            self._slot_t = t
        if self.use_graph:
            if self.graph is None:
                self._capture(t)
            if self._apool is None:
                q, kn, vn = self.active_inputs(t)
                self.g_q.copy_(q)
                self.g_kn.copy_(kn)
                self.g_vn.copy_(vn)
                if self.g_logits is not None:
                    self.g_logits.copy_(self.active_logits(t))
                    self.g_u.copy_(self.active_draws(t))
            self.graph.replay()
            self._slot_t = t + 1
            self.tokens = self.g_tok
            return self.g_out, self.lse_ring[t % self.R], self.g_logits
        q, kn, vn = self.active_inputs(t)
        out = torch.empty(q.shape, dtype=self.out_dtype, device=self.device)
        reco.reco_decode_attn_ring(self.kv, q, kn, vn, self.lens_dev, wl.scale(), out, self.lse_ring, self.slot_dev,
                                   self.ws_decode, q_ring=self.q_win)
        lse = self.lse_ring[t % self.R]
        self._slot_t = t + 1
        logits = None
        if self.ids is not None:
            logits = self.active_logits(t)
            rw = self.staging.put([self.current_reward(s) for s in self.active], torch.float32)
            self.tokens = torch.empty(len(self.active), dtype=torch.int32, device=self.device)
            reco.reco_penalty_sample(logits, self.ids, rw, self.active_draws(t), self.tokens, self.ws_sample,
                                     wl.tau_l, wl.tau_h, wl.beta)
        return out, lse, logits

    def run(self, max_tokens=None, on_token=None, on_boundary=None) -> TraceEvents:
        spec, wl = self.spec, self.wl
        ev = TraceEvents()
        T = spec.generated if max_tokens is None else min(max_tokens, spec.generated)
        row_bytes = 2 * wl.layers * wl.h_kv * wl.d * wl.elem_bytes  # K and V of one token
        for t in range(T):
            if not self.active:
                break
            out, lse, logits = self._token(t)
            self.lens = [L + 1 for L in self.lens]
            self.full = [F + 1 for F in self.full]
            self.since = [x + 1 for x in self.since]
            ev.generated += len(self.active)
            held = sum(self.lens) * row_bytes
            ev.peak_cache_bytes = max(ev.peak_cache_bytes, held)
            ev.cache_byte_tokens += held
            if on_token:
                on_token(t, self, out, lse, logits)
            ev.tokens += 1
            # step boundaries completed at this token (batch positions, in batch order)
            done = []
            for s in self.ends_at.get(t, ()):
                if s not in self.pos:
                    continue  # stopped earlier
                self.hist[s].append(self.rewards[s][self.step_idx[s]])
                self.step_idx[s] += 1
                done.append(self.pos[s])
            if not done:
                continue
            done.sort()
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
                comp = [self.pos[s] for s, _, _ in info]
                if self.use_graph and self.graph is not None:
                    keep_dev = self._put_small(keep)[:self.B]  # with the new rewards
                else:
                    keep_dev = self.staging.put(list(keep), torch.int32)
                # only the sequences compressed now are scored (keep == L skips the rest)
                if all(self.since[i] >= wl.w for i in comp):
                    # every window token was decoded on the cache as it is now, so the lse
                    # its decode returned is its row's normaliser: one pass over K, with the
                    # rings' rows in slot order
                    q_win = self.q_win
                    reco.reco_score_cache_lse(self.kv, q_win, self.lens_dev, self.lse_ring[:wl.w], wl.w,
                                              wl.pool, wl.scale(), self.scores, self.ws_score, keep=keep_dev)
                    ev.lse_scorings += 1
                else:
                    q_win = self._window_in_token_order(t)
                    reco.reco_score_cache(self.kv, q_win, self.lens_dev, wl.w, wl.pool, wl.scale(), self.scores,
                                          self.ws_score, keep=keep_dev)
                    ev.two_pass_scorings += 1
                reco.reco_select_compact(self.kv, self.scores, self.lens_dev, keep_dev, wl.w, self.kept,
                                         self.ws_select)
                if on_boundary and q_win is self.q_win:
                    q_win = self._window_in_token_order(t)  # the caller sees token order
            if on_boundary:
                on_boundary(t, self, done, keep, q_win)
            for i in range(len(keep)):
                if keep[i] < self.lens[i]:
                    self.since[i] = 0  # compressed: its earlier lse no longer match its cache
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
            elif self.use_graph and self.graph is not None and not info:
                self._put_small(keep)  # the new rewards (the keep row is not read)
        return ev
