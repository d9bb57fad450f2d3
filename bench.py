"""Benchmark of the ReCo hot path on GB300: compress + decode tokens/s.

One step = one reasoning-step boundary of a workload and the decode that follows.
The default is the largest single-GPU one, the 32B-class stack (Qwen2.5-32B shape:
64 layers, 40/8 heads, d 128, bf16, batch 4, cache 32768, window 64, Eq. 1 ratios
spanning 0.2-0.9): Eq. 1 keep counts, Eq. 2 scores, top-m select, in-place
compaction, then 256 decode steps (append + attention over the ragged compacted
cache, all layers per launch).  The 7B-class workload adds the Eq. 3-4 reflection
penalty on [8, 152064] logits after every decode step and the Eq. 5-6 answer-PPL
probe over 32 answer tokens.  Tokens per step = B*L cached tokens compressed +
B*steps decoded; the line also carries the two rates apart (compress_tokens_s over
score + select + compact, decode_tokens_s over the decode launches).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload 32b|7b|1.5b|tiny|trace]
    python bench.py --impl reference ...   # the fp64 CPU oracle on the host cores

Under torchrun each rank runs an independent replica (the path shards by sequence
with no data exchange); rank 0 prints one JSON line.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)
os.environ.setdefault("OMP_NUM_THREADS", str(os.cpu_count() or 1))

import numpy as np  # noqa: E402
import torch  # noqa: E402

METRIC = "compress+decode tokens/s and achieved HBM GB/s (fraction of ~8 TB/s), 1×GB300"
UNIT = "tokens/s"


def log(*a):
    print(*a, file=sys.stderr, flush=True)


# ------------------------------------------------------------------ distributed plumbing
def dist_setup(n_gpus):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------ peaks, clocks, profiles
def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


class ClockSampler:
    """nvidia-smi samples (200 ms) of SM clock and throttle reasons during the timed region."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device):
        self.proc = None
        self.path = tempfile.mktemp(prefix="reco_clocks_", suffix=".csv")
        try:
            self.gpu = "GPU-" + str(torch.cuda.get_device_properties(device).uuid)
        except Exception:
            vis = os.environ.get("CUDA_VISIBLE_DEVICES", "").split(",")[0].strip()
            self.gpu = vis if vis else "0"

    def __enter__(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return None
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                rows.append((float(parts[1]), float(parts[2]), float(parts[3]), parts[5:9]))
            except ValueError:
                continue
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i, v in enumerate(r[3]) if v.lower() == "active"})
        loaded = [r[0] for r in rows if r[2] > 200.0] or [r[0] for r in rows]
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


def decode_code_hash(src: str) -> str:
    """sha256 (16 hex digits) of a CUDA source with its comments and blank lines removed:
    a profile stays valid across edits that change no code."""
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    lines = [re.sub(r"//.*$", "", ln).rstrip() for ln in src.splitlines()]
    return hashlib.sha256("\n".join(ln for ln in lines if ln.strip()).encode()).hexdigest()[:16]


def decode_traffic(wl):
    """DRAM bytes per decode launch of this workload from the committed ncu summary
    profiles/decode_attn_<workload>.md, if it was taken on the current decode kernel
    source (checked by hash).  Returns (bytes or None, where the figure comes from)."""
    name = f"decode_attn_{wl.name}.md"
    path = os.path.join(ROOT, "profiles", name)
    if not os.path.exists(path):
        return None, f"none: no ncu summary profiles/{name}"
    text = open(path).read()
    m = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
    h = re.search(r"decode_source_sha256:\s*([0-9a-f]+)", text)
    c = re.search(r"capture:\s*(.+)", text)
    if not m or not h:
        return None, f"none: profiles/{name} carries no per-launch DRAM bytes"
    src = open(os.path.join(ROOT, "paper_2608_04771_gb300", "csrc", "decode.cu")).read()
    if decode_code_hash(src) != h.group(1)[:16]:
        return None, f"none: profiles/{name} was taken on another decode.cu"
    return float(m.group(1)), (f"profile-derived, not measured in this run: profiles/{name} "
                               f"(ncu dram__bytes_read.sum + dram__bytes_write.sum; {c.group(1).strip() if c else ''})")


# ------------------------------------------------------------------ algorithmic work
def algorithmic(wl, keep_host):
    """Per-launch algorithmic bytes / flops of each kernel group for one step."""
    es = wl.elem_bytes
    units_per_b = wl.layers * wl.h_kv
    d = wl.d
    G = wl.G
    rows_q = wl.layers * wl.batch * wl.h_q
    score_bytes = wl.units * (wl.L * d * es + 4 * (wl.L - wl.w)) + rows_q * wl.w * d * es
    score_flops = wl.units * 2.0 * G * wl.w * wl.L * d
    kept_total = sum(int(m) for m in keep_host) * units_per_b
    select_bytes = wl.units * 4 * (wl.L - wl.w) + 4 * kept_total  # scores read + indices written
    compact_bytes = 4.0 * kept_total * d * es  # read + write K and V for every kept row (upper bound)
    dec = []
    for s in range(wl.decode_steps):
        rows = sum((int(m) + s + 1) for m in keep_host) * units_per_b
        b = 2.0 * rows * d * es  # K and V rows read
        b += rows_q * d * es + 2.0 * wl.units * d * es * 2  # q read; k_new/v_new read and written
        b += rows_q * d * 2 + rows_q * 4  # bf16 out + lse
        dec.append(b)
    pen_bytes = 2.0 * wl.batch * wl.n_ids * 4 if wl.vocab else 0.0
    ppl_bytes = 4.0 * wl.batch * wl.n_answer * wl.vocab if wl.vocab else 0.0
    return dict(score_bytes=score_bytes, score_flops=score_flops, select_bytes=select_bytes,
                compact_bytes=compact_bytes, decode_bytes=dec, penalty_bytes=pen_bytes, ppl_bytes=ppl_bytes)


# ------------------------------------------------------------------ oracle timing (CPU)
class OracleSample:
    """The fp64 oracle timed on a bounded sample of a workload on the host cores: the
    first `units` units (whole layers of the batch, or part of layer 0) at full length
    for score + select + compact, then `dec_steps` decode steps over them; for workloads
    with a vocabulary, the penalty once on the full logits and the PPL on the sampled
    sequences.  Inputs are drawn once; run() times one pass over the sample.  Nothing is
    extrapolated inside run(): project() scales the measured pieces linearly to one full
    step (all units, all decode steps, a penalty per decode step, the PPL of every sequence)."""

    def __init__(self, wl, units: int, dec_steps: int):
        import oracle
        from paper_2608_04771_gb300 import workloads as W
        oracle.build()
        self.wl = wl
        per_layer = wl.batch * wl.h_kv
        if units >= per_layer:
            Ls, Bs = min(wl.layers, -(-units // per_layer)), wl.batch
        else:
            Ls, Bs = 1, max(1, min(wl.batch, -(-units // wl.h_kv)))
        self.sw = sw = wl.reduced(layers=Ls, batch=Bs)
        K, V = W.make_cache(sw, "cpu", canary=False)
        self.K, self.V = K.float().numpy(), V.float().numpy()
        self.q = W.make_qwin(sw, "cpu").float().numpy()
        self.lens = np.full((Ls, Bs, sw.h_kv), sw.L, np.int32)
        hist = W.make_reward_history(wl)[:Bs]
        self.keep = np.array([oracle.keep_count(oracle.retention_ratio(hist[b], wl.base, wl.delta), wl.L, wl.w)
                              for b in range(Bs)], np.int32)
        self.n_dec = min(dec_steps, wl.decode_steps)
        self.dec = []
        for s in range(self.n_dec):
            qd, kn, vn = W.make_decode_step(sw, s, "cpu")
            self.dec.append((qd.float().numpy(), kn.float().numpy(), vn.float().numpy()))
        if wl.vocab:
            self.z = W.make_vocab_logits(wl, "cpu").numpy()
            self.ids = W.make_reflection_ids(wl)
            self.rw = W.make_reward_history(wl)[:, -1].copy()
            za, tok = W.make_answer(wl.reduced(batch=Bs), "cpu")
            self.za, self.tok = za.numpy(), tok.numpy()

    def run(self):
        import oracle
        sw, wl = self.sw, self.wl
        t0 = time.perf_counter()
        sc = oracle.score_cache(self.q, self.K, self.lens, sw.w, sw.pool, sw.scale())
        idx = oracle.select_batch(sc.astype(np.float32), self.lens, self.keep, sw.w)
        Kc, Vc = np.zeros_like(self.K), np.zeros_like(self.V)
        for l in range(sw.layers):
            for b in range(sw.batch):
                m = int(self.keep[b])
                for h in range(sw.h_kv):
                    Kc[l, b, h, :m] = oracle.gather_unit(self.K[l, b, h], idx[l, b, h, :m])
                    Vc[l, b, h, :m] = oracle.gather_unit(self.V[l, b, h], idx[l, b, h, :m])
        t_comp = time.perf_counter() - t0
        lens_c = np.broadcast_to(self.keep.reshape(1, -1, 1), self.lens.shape).copy()
        t0 = time.perf_counter()
        for qd, kn, vn in self.dec:
            for l in range(sw.layers):
                for b in range(sw.batch):
                    for h in range(sw.h_kv):
                        Lc = lens_c[l, b, h]
                        Kc[l, b, h, Lc], Vc[l, b, h, Lc] = kn[l, b, h], vn[l, b, h]
            lens_c += 1
            oracle.decode_batch(qd, Kc, Vc, lens_c, sw.scale())
        t_dec = time.perf_counter() - t0
        t_pen = t_ppl = 0.0
        if wl.vocab:
            t0 = time.perf_counter()
            oracle.reflect_penalty(self.z, self.ids, self.rw, wl.tau_l, wl.tau_h, wl.beta)
            t_pen = time.perf_counter() - t0
            t0 = time.perf_counter()
            oracle.answer_ppl(self.za, self.tok, None, wl.tau_p)
            t_ppl = time.perf_counter() - t0
        return {"compress_s": t_comp, "decode_s": t_dec, "penalty_s": t_pen, "ppl_s": t_ppl,
                "total_s": t_comp + t_dec + t_pen + t_ppl}

    def project(self, m):
        """Measured pieces -> one full step (linear in units, decode steps and rows)."""
        wl, sw = self.wl, self.sw
        f = sw.units / wl.units
        t_comp = m["compress_s"] / f
        t_dec = (m["decode_s"] / max(self.n_dec, 1)) * wl.decode_steps / f if self.n_dec else 0.0
        t_voc = m["penalty_s"] * wl.decode_steps + m["ppl_s"] * wl.batch / sw.batch if wl.vocab else 0.0
        full = t_comp + t_dec + t_voc
        tokens = wl.batch * (wl.L + wl.decode_steps)
        return {"full_step_s": full, "value": tokens / full,
                "compress_tokens_s": wl.batch * wl.L / t_comp,
                "decode_tokens_s": wl.batch * wl.decode_steps / t_dec if t_dec > 0 else None,
                "sample_tokens": tokens * m["total_s"] / full}

    def describe(self):
        wl, sw = self.wl, self.sw
        return (f"{sw.units} of {wl.units} units ({sw.layers} layer(s) x {sw.batch} sequences x {sw.h_kv} KV heads) "
                f"at full length: score+select+compact, then {self.n_dec} of {wl.decode_steps} decode steps over them"
                + ("; penalty once on the full logits; PPL on the sampled sequences" if wl.vocab else "")
                + "; measured pieces scaled linearly to one full step")


def cpu_rate(wl, units, dec_steps, threads=None):
    """One timed pass of the oracle sample; returns the cpu_baseline-style record."""
    import oracle
    smp = OracleSample(wl, units, dec_steps)
    if threads:
        oracle.set_threads(threads)
    try:
        m = smp.run()
        cores = oracle.threads()
    finally:
        if threads:
            oracle.set_threads(int(os.environ["OMP_NUM_THREADS"]))
    p = smp.project(m)
    return {"value": p["value"], "unit": UNIT, "cores": cores, "kind": "oracle", "sample": smp.describe(),
            "extrapolated": smp.sw.units < wl.units or smp.n_dec < wl.decode_steps,
            "units_timed": smp.sw.units, "units_total": wl.units, "decode_steps_timed": smp.n_dec,
            "decode_steps_total": wl.decode_steps, "measured_s": m, "projected_full_step_s": p["full_step_s"],
            "compress_tokens_s": p["compress_tokens_s"], "decode_tokens_s": p["decode_tokens_s"]}


def run_reference(args, wl):
    """The reference arm: the oracle as it stands, each step one pass over the bounded sample
    (timed as it ran); value = the sample's token-equivalents per second of its run."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    import oracle
    smp = OracleSample(wl, args.ref_units, args.ref_dec_steps)
    oracle.set_threads(int(os.environ["OMP_NUM_THREADS"]))
    runs = []
    for i in range(args.warmup + args.steps):
        m = smp.run()
        if i >= args.warmup:
            runs.append(m)
    mean = {k: statistics.mean(r[k] for r in runs) for k in runs[0]}
    p = smp.project(mean)
    ms = mean["total_s"] * 1e3
    cores = oracle.threads()
    desc = smp.describe()
    line = {"impl": "reference", "metric": METRIC, "value": p["value"], "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": workload_name(wl), "tokens_per_step": p["sample_tokens"],
                       "step": "one pass of the oracle over the bounded sample below (not a full step): "
                               "ms_per_step is that pass as measured, tokens_per_step its token-equivalents "
                               "(the full step's tokens times its share of the projected full-step time)",
                       "full_step_tokens": wl.batch * (wl.L + wl.decode_steps),
                       "projected_full_step_ms": p["full_step_s"] * 1e3},
            "compress_tokens_s": p["compress_tokens_s"], "decode_tokens_s": p["decode_tokens_s"],
            "cpu_baseline": {"value": p["value"], "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc,
                             "extrapolated": smp.sw.units < wl.units or smp.n_dec < wl.decode_steps,
                             "units_timed": smp.sw.units, "units_total": wl.units,
                             "decode_steps_timed": smp.n_dec, "decode_steps_total": wl.decode_steps,
                             "measured_s": mean},
            "e2e": {"value": p["value"], "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def workload_name(wl):
    return (f"{wl.name}-class: {wl.layers} layers, {wl.h_q}/{wl.h_kv} heads, d {wl.d}, {wl.dtype}, batch "
            f"{wl.batch}, cache {wl.L}, window {wl.w}, pool {wl.pool}, {wl.decode_steps} decode steps"
            + (f", vocab {wl.vocab} penalty ({wl.n_ids} ids) + answer PPL ({wl.n_answer} tokens)" if wl.vocab else ""))


# ------------------------------------------------------------------ GPU arm
def time_penalty(hp, n=128, reps=4):
    """reco_reflect_penalty on the step's logits, ids and rewards (a copy of the logits),
    timed apart from the step so that no event pair sits between the step's launches:
    n launches captured in one CUDA graph, the way the step issues them after each decode."""
    from paper_2608_04771_gb300 import reco
    wl = hp.wl
    z = hp.logits.clone()
    beta = torch.empty_like(hp.beta)
    reco.reco_reflect_penalty(z, hp.ids, hp.rewards, wl.tau_l, wl.tau_h, wl.beta, beta)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="relaxed"):
        for _ in range(n):
            reco.reco_reflect_penalty(z, hp.ids, hp.rewards, wl.tau_l, wl.tau_h, wl.beta, beta)
    g.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        g.replay()
    b.record()
    b.synchronize()
    reco.reco_check()
    return {"ms_per_launch": a.elapsed_time(b) / (reps * n),
            "timing": f"{n} launches on the step's buffers captured in one CUDA graph, outside the timed step"}


def time_score_lse(hp, alg, reps=5):
    """Eq. 2 with the window rows' normalisers from the decode (reco_score_cache_lse) on the
    step's pristine cache, beside the two-pass reco_score_cache, both timed apart from the
    step.  The normalisers are the lse outputs of the library's decode of each window query
    over the keys Eq. 2 lets it see (lens L-w+t+1, no append), as the decode of the window
    tokens would have returned them.  Both results are compared element by element."""
    from paper_2608_04771_gb300 import reco
    wl, dev = hp.wl, hp.K.device
    hp.reset()
    ws_dec = reco.workspace(reco.RECO_OP_DECODE, hp.kv, 0, dev)
    row_lse = torch.empty((wl.w, wl.layers, wl.batch, wl.h_q), dtype=torch.float32, device=dev)
    out = torch.empty((wl.layers, wl.batch, wl.h_q, wl.d), dtype=torch.bfloat16, device=dev)
    for t in range(wl.w):
        lens_t = hp.lens0 - (wl.w - 1 - t)
        reco.reco_decode_attn(hp.kv, hp.q_win[:, :, :, t, :].contiguous(), None, None, lens_t, wl.scale(), out,
                              row_lse[t], ws_dec)
    two = torch.empty_like(hp.scores)
    one = torch.empty_like(hp.scores)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(4)]
    t2, t1 = [], []
    for _ in range(reps):
        ev[0].record()
        reco.reco_score_cache(hp.kv, hp.q_win, hp.lens, wl.w, wl.pool, wl.scale(), two, hp.ws_score)
        ev[1].record()
        reco.reco_score_cache_lse(hp.kv, hp.q_win, hp.lens, row_lse, wl.w, wl.pool, wl.scale(), one, hp.ws_score)
        ev[2].record()
        ev[2].synchronize()
        t2.append(ev[0].elapsed_time(ev[1]))
        t1.append(ev[1].elapsed_time(ev[2]))
    reco.reco_check()
    nc = wl.L - wl.w
    a, b = two[..., :nc].double(), one[..., :nc].double()
    rel = float(((a - b).abs() / a.abs().clamp_min(1e-30)).max())
    ms1, ms2 = statistics.median(t1), statistics.median(t2)
    k_bytes = wl.units * wl.L * wl.d * wl.elem_bytes
    return {"ms": ms1, "two_pass_ms": ms2, "TFLOP/s": alg["score_flops"] / ms1 / 1e9,
            "K GB/s": k_bytes / ms1 / 1e6, "max_rel_diff_vs_two_pass": rel,
            "timing": "median of 5 calls on the pristine cache, outside the timed step; normalisers from the "
                      "decode of each window query (no append)"}


def time_penalty_sample(wl, dev, n_buf=32, reps=4):
    """The penalty followed by one draw per sequence (reco_penalty_sample) on the workload's
    vocabulary, timed apart from the step: n_buf logits buffers (more bytes than L2) are
    visited in turn so every launch reads its logits from HBM.  Algorithmic bytes per launch:
    the logits once, plus one segment per row read again and the penalised ids written."""
    from paper_2608_04771_gb300 import reco
    from paper_2608_04771_gb300 import workloads as W
    zs = [W.make_vocab_logits(wl, dev, stream=60 + i) for i in range(n_buf)]
    ids = torch.from_numpy(W.make_reflection_ids(wl)).to(dev)
    rw = torch.from_numpy(W.make_reward_history(wl)[:, -1].copy()).to(dev)
    u = torch.from_numpy(W.make_draws(wl, wl.batch)).to(dev)
    tok = torch.empty(wl.batch, dtype=torch.int32, device=dev)
    ws = reco.sample_workspace(wl.batch, wl.vocab, dev)
    for z in zs[:4]:
        reco.reco_penalty_sample(z, ids, rw, u, tok, ws, wl.tau_l, wl.tau_h, wl.beta)
    torch.cuda.synchronize()
    # the n_buf calls as one CUDA graph, so the launches are not paced by the host
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="relaxed"):
        for z in zs:
            reco.reco_penalty_sample(z, ids, rw, u, tok, ws, wl.tau_l, wl.tau_h, wl.beta)
    g.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(reps):
        g.replay()
    b.record()
    b.synchronize()
    reco.reco_check()
    ms = a.elapsed_time(b) / (reps * n_buf)
    byts = 4.0 * wl.batch * wl.vocab + 4.0 * wl.batch * min(wl.vocab, 4096) + 8.0 * wl.batch * wl.n_ids
    return {"ms_per_launch": ms, "GB/s": byts / ms / 1e6, "rows": wl.batch, "vocab": wl.vocab,
            "timing": f"{n_buf} logits buffers visited in turn ({n_buf * 4 * wl.batch * wl.vocab / 1e6:.0f} MB > L2) "
                      "by one captured graph, outside the timed step"}


def run_gpu(args, wl):
    from paper_2608_04771_gb300 import build as B
    from paper_2608_04771_gb300 import driver, reco
    world, rank, local = dist_setup(args.gpus)
    B.build()
    dev = f"cuda:{local}"
    torch.cuda.set_device(dev)
    hp = driver.HotPath(wl, dev, out_dtype=torch.bfloat16, keep_pristine=True)
    stream = torch.cuda.current_stream()
    steps, warm = args.steps, max(args.warmup, 3)
    ev = lambda: torch.cuda.Event(enable_timing=True)  # noqa: E731
    for _ in range(warm):
        hp.reset()
        hp.step()
    reco.reco_check()
    torch.cuda.synchronize()

    ph = {k: [] for k in ("score", "select", "compact", "decode", "decode_phase", "ppl", "step")}
    # an event pair around every 4th decode launch: the sampled launches give the average
    # launch time (their own algorithmic bytes over their own durations), with a quarter
    # of the event gaps inside the step
    sampled = list(range(0, wl.decode_steps, 4))
    dec_ev = {s: (ev(), ev()) for s in sampled}
    barrier(world)
    torch.cuda.synchronize()
    with ClockSampler(torch.cuda.current_device()) as clk:
        for _ in range(steps):
            hp.reset()
            e = [ev() for _ in range(6)]
            e[0].record(stream)
            hp.score()
            e[1].record(stream)
            hp.select()
            e[2].record(stream)
            hp.compact()
            e[3].record(stream)
            for s in range(wl.decode_steps):
                if s in dec_ev:
                    dec_ev[s][0].record(stream)
                hp.decode(s)
                if s in dec_ev:
                    dec_ev[s][1].record(stream)
                if hp.has_vocab:
                    hp.penalty()
            e[4].record(stream)
            if hp.has_vocab:
                hp.probe()
            e[5].record(stream)
            e[5].synchronize()
            ph["score"].append(e[0].elapsed_time(e[1]))
            ph["select"].append(e[1].elapsed_time(e[2]))
            ph["compact"].append(e[2].elapsed_time(e[3]))
            ph["decode"].append([dec_ev[s][0].elapsed_time(dec_ev[s][1]) for s in sampled])
            ph["decode_phase"].append(e[3].elapsed_time(e[4]))
            ph["ppl"].append(e[4].elapsed_time(e[5]))
            ph["step"].append(e[0].elapsed_time(e[5]))
        torch.cuda.synchronize()
        barrier(world)
    reco.reco_check()
    ms_step = max_over_ranks(statistics.mean(ph["step"]), world)
    tokens = wl.batch * (wl.L + wl.decode_steps)
    value = world * tokens / (ms_step / 1e3)

    hbm, tc_burst, tc_sust, peak_kind = measured_peaks()
    alg = algorithmic(wl, hp.keep_host)
    dec_ms = np.array(ph["decode"]).mean(axis=0)  # per sampled decode launch, averaged over steps
    dec_bytes = np.array(alg["decode_bytes"])[sampled]
    dec_avg_ms = float(dec_ms.mean())
    dec_achieved = float(dec_bytes.mean() / (dec_avg_ms / 1e3) / 1e9)
    traffic, traffic_src = decode_traffic(wl)
    score_ms = statistics.mean(ph["score"])
    select_ms = statistics.mean(ph["select"])
    compact_ms = statistics.mean(ph["compact"])
    compress_ms = max_over_ranks(score_ms + select_ms + compact_ms, world)
    decode_ms = max_over_ranks(dec_avg_ms * wl.decode_steps, world)
    mx = int(hp.keep_host.max())  # rows whose source is another row (kept[r] != r): the ones that move
    r_ = torch.arange(mx, device=dev, dtype=torch.int32)
    moved = int(((hp.kept[..., :mx] != r_) & (r_.view(1, 1, 1, -1) < hp.keep.view(1, -1, 1, 1))).sum())
    compact_gbs = alg["compact_bytes"] / compact_ms / 1e6
    kernels = {
        "score": {"ms": score_ms, "GB/s": alg["score_bytes"] / score_ms / 1e6,
                  "TFLOP/s": alg["score_flops"] / score_ms / 1e9,
                  "tensor_frac": alg["score_flops"] / score_ms / 1e9 / tc_burst,
                  "note": "one logical QK^T pass of flops; the kernel runs two passes over K"},
        "select": {"ms": select_ms, "GB/s": alg["select_bytes"] / select_ms / 1e6},
        "compact": {"ms": compact_ms, "GB/s": compact_gbs, "frac": compact_gbs / hbm, "peak": hbm,
                    "peak_kind": peak_kind, "frac_of_8TBs": compact_gbs / 8000.0,
                    "algorithmic_bytes": alg["compact_bytes"],
                    "rows_moved_frac": moved / max(1, int(hp.keep_host.sum()) * wl.layers * wl.h_kv),
                    "timing": "own event pair in the step (reco_compact after reco_select_topm)"},
        "decode": {"ms_per_launch": dec_avg_ms, "GB/s": dec_achieved, "launches": wl.decode_steps,
                   "phase_ms": statistics.mean(ph["decode_phase"]),
                   "timed_launches": f"every 4th ({len(sampled)} of {wl.decode_steps}) between CUDA events"},
    }
    if hp.has_vocab:
        kernels["penalty"] = time_penalty(hp)
        kernels["ppl"] = {"ms": statistics.mean(ph["ppl"]),
                          "GB/s": alg["ppl_bytes"] / statistics.mean(ph["ppl"]) / 1e6}
        kernels["penalty_sample"] = time_penalty_sample(wl, dev)
    kernels["score_lse"] = time_score_lse(hp, alg)

    e2e = run_e2e(hp, wl, args, world) if not args.no_e2e else None
    clocks = clk.summary()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from paper_2608_04771_gb300 import workloads as W
        cpu = cpu_rate(wl, args.ref_units, args.ref_dec_steps)
        # one host core, on the Tiny workload (whole) and on a sample of the 1.5B-class stack
        cpu["one_core"] = {name: cpu_rate(W.WORKLOADS[name], u, n, threads=1)
                           for name, u, n in (("tiny", 2, 1), ("1.5b", 8, 8))}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": steps, "warmup": warm,
            "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if wl.dtype == "bf16" else "f32", "data": "synthetic",
            "compress_tokens_s": world * wl.batch * wl.L / (compress_ms / 1e3),
            "decode_tokens_s": world * wl.batch * wl.decode_steps / (decode_ms / 1e3),
            "config": {"workload": workload_name(wl), "tokens_per_step": tokens,
                       "parallelism": f"replicas x{world} (sequences sharded, no collective)",
                       "l2": f"inputs larger than L2 (K/V {2 * hp.K.numel() * hp.K.element_size() / 1e9:.1f} GB); "
                             "the cache restore before each step (outside the timed events) also overwrites L2",
                       "rates": "compress_tokens_s = B*L / (score + select + compact); decode_tokens_s = "
                                "B*steps / (steps * mean decode launch), attention only",
                       "kernels": kernels, "keep_counts": [int(x) for x in hp.keep_host]},
            "roofline": {"bound": "hbm", "kernel": "decode_tma (reco_decode_attn)", "achieved": dec_achieved,
                         "peak": hbm, "unit": "GB/s", "frac": dec_achieved / hbm, "peak_kind": peak_kind,
                         "frac_of_8TBs": dec_achieved / 8000.0,
                         "traffic": traffic, "traffic_source": traffic_src,
                         "algorithmic_bytes_per_launch": float(dec_bytes.mean())},
            "cpu_baseline": cpu,
            "e2e": e2e,
            "gpu_launches": hp.launches_per_step() * steps,
            "clocks": clocks,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def gpu_local_cpus(dev):
    """Host CPUs attached to the GPU's NUMA node (from sysfs), or None if not visible."""
    try:
        pr = torch.cuda.get_device_properties(dev)
        bus = f"{pr.pci_domain_id:04x}:{pr.pci_bus_id:02x}:{pr.pci_device_id:02x}.0"
        text = open(f"/sys/bus/pci/devices/{bus}/local_cpulist").read().strip()
    except Exception:
        return None
    cpus = set()
    for part in text.split(","):
        if "-" in part:
            lo, hi = part.split("-")
            cpus.update(range(int(lo), int(hi) + 1))
        elif part:
            cpus.add(int(part))
    allowed = os.sched_getaffinity(0)
    return (cpus & allowed) or None


def run_e2e(hp, wl, args, world):
    """Same metric through the C ABI with host buffers: every step copies all of its inputs
    from pinned host memory, runs the hot path and reads its results back, all inside the
    timed region.  The steps are pipelined over two device buffer sets: step i+1's inputs
    travel on a copy stream while step i computes, and a set is overwritten only after the
    step that last used it has finished (its results read back).  The pinned buffers are
    allocated and first touched from the CPUs local to the GPU when sysfs names them, so
    their pages sit on the GPU's own host memory node."""
    from paper_2608_04771_gb300 import driver
    dev = hp.K.device
    local = gpu_local_cpus(dev)
    prev_aff = os.sched_getaffinity(0)
    if local:
        os.sched_setaffinity(0, local)
    try:
        def pin(t):  # device tensor -> a pinned host copy, with no pageable intermediate
            h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
            h.copy_(t)
            return h
        host = dict(K=pin(hp.K0), V=pin(hp.V0), lens=pin(hp.lens0), q_win=pin(hp.q_win), keep=pin(hp.keep),
                    dq=pin(hp.dq), dk=pin(hp.dk), dv=pin(hp.dv))
        if hp.has_vocab:
            host.update(logits=pin(hp.logits), ids=pin(hp.ids), rewards=pin(hp.rewards),
                        ans_logits=pin(hp.ans_logits), ans_tokens=pin(hp.ans_tokens))
        out_names = ["out"] + (["ppl", "stop"] if hp.has_vocab else [])
        host_out = {k: torch.empty(getattr(hp, k).shape, dtype=getattr(hp, k).dtype, pin_memory=True)
                    for k in out_names}
    finally:
        os.sched_setaffinity(0, prev_aff)
    sets = [hp, driver.HotPath(wl, dev, out_dtype=hp.out.dtype, keep_pristine=False)]
    h2d = sum(h.numel() * h.element_size() for h in host.values())
    d2h = sum(h.numel() * h.element_size() for h in host_out.values())
    comp = torch.cuda.current_stream()
    ncs = 2  # host-to-device copy streams (copy engines working at once)
    cps = torch.cuda.Stream(device=dev)  # host-to-device copies (the first copy stream)
    cpx = [cps] + [torch.cuda.Stream(device=dev) for _ in range(ncs - 1)]
    dps = torch.cuda.Stream(device=dev)  # device-to-host copies
    ready = [torch.cuda.Event() for _ in sets]
    done = [torch.cuda.Event() for _ in sets]
    free = [torch.cuda.Event() for _ in sets]
    cp_ev = []

    def enqueue(i, timed=False):
        s = sets[i % 2]
        with torch.cuda.stream(cps):
            if i >= 2:
                cps.wait_event(free[i % 2])  # the step that last used this set has finished
            c0 = torch.cuda.Event(enable_timing=timed)
            c0.record(cps)
            for x in cpx[1:]:
                x.wait_event(c0)
            # copies of at most 1 GiB each, dealt in turn to the copy streams (several copy engines)
            j = 0
            for k, h in host.items():
                dst = getattr(s, k).view(-1).view(torch.uint8)
                src = h.view(-1).view(torch.uint8)
                for o in range(0, src.numel(), 1 << 30):
                    with torch.cuda.stream(cpx[j % ncs]):
                        dst[o:o + (1 << 30)].copy_(src[o:o + (1 << 30)], non_blocking=True)
                    j += 1
            for x in cpx[1:]:
                cps.wait_stream(x)
            ready[i % 2].record(cps)
            if timed:
                c1 = torch.cuda.Event(enable_timing=True)
                c1.record(cps)
                cp_ev.append((c0, c1))
        comp.wait_event(ready[i % 2])
        s.step()
        done[i % 2].record(comp)
        with torch.cuda.stream(dps):
            dps.wait_event(done[i % 2])
            for k, h in host_out.items():
                h.copy_(getattr(s, k), non_blocking=True)
            free[i % 2].record(dps)

    enqueue(0)  # warm-up of the second set and the streams (untimed)
    enqueue(1)
    torch.cuda.synchronize()
    n = max(4, args.steps)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(comp)
    cps.wait_event(a)
    for i in range(n):
        enqueue(i, timed=True)
    comp.wait_stream(dps)  # the last results read back
    b.record(comp)
    b.synchronize()
    ms = max_over_ranks(a.elapsed_time(b) / n, world)
    cp_ms = statistics.median(c0.elapsed_time(c1) for c0, c1 in cp_ev)
    tokens = wl.batch * (wl.L + wl.decode_steps)
    return {"value": world * tokens / (ms / 1e3), "unit": UNIT, "ms_per_step": ms,
            "h2d_bytes_per_step": int(h2d), "d2h_bytes_per_step": int(d2h), "steps": n,
            "h2d_GBps": h2d / cp_ms / 1e6, "h2d_ms_per_step": cp_ms,
            "pinned_near_gpu": bool(local),
            "schedule": "two device buffer sets; step i+1's host-to-device copies (pieces of at most 1 GiB over two "
                        "copy streams) and step i-1's read-back overlap step i's compute"}


def run_trace(args):
    """The step-loop trace (batch 16, 8192 generated tokens, 7B-class heads): one run, timed."""
    from paper_2608_04771_gb300 import build as B
    from paper_2608_04771_gb300 import reco, trace
    B.build()
    spec = trace.full_trace_spec(args.reading)
    if args.generated:
        spec.generated = args.generated
    use_graph = not args.no_graph
    warm = trace.Trace(spec, "cuda", torch.bfloat16, input_pool=32, use_graph=use_graph)
    warm.run(max_tokens=320)  # past the first probe (and its stop): every kernel and path warm
    torch.cuda.synchronize()
    tr = trace.Trace(spec, "cuda", torch.bfloat16, input_pool=32, use_graph=use_graph)
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0 = time.perf_counter()
    a.record()
    ev = tr.run()
    b.record()
    b.synchronize()
    wall = time.perf_counter() - t0
    reco.reco_check()
    ms = a.elapsed_time(b)
    wl = tr.wl
    row_bytes = 2 * wl.layers * wl.h_kv * wl.d * wl.elem_bytes
    full_peak = spec.batch * (spec.prompt + spec.generated) * row_bytes
    line = {
        "metric": "step-loop trace: generated tokens/s (decode + penalty + draw every token, compression at step "
                  "boundaries, answer probes), 1xGB300",
        "value": ev.generated / (ms / 1e3), "unit": "tokens/s", "n_gpus": 1, "ms_total": ms, "wall_s": wall,
        "higher_is_better": True, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"trace: 7B-class heads, 28 layers, batch {spec.batch}, prompt {spec.prompt}, "
                               f"{spec.generated} generated tokens, steps Poisson({spec.step_mean})+{spec.step_min}, "
                               f"Beta(2,2) rewards, reading {spec.reading}, interval S={spec.interval}",
                   "inputs": "per-token synthetic inputs drawn once for w = 32 tokens and reused cyclically",
                   "window": "Eq. 2's window queries are the last w decoded tokens' queries; their queries and "
                             "decode lse are kept in device rings of w slots by every token, and a boundary "
                             "scores in one pass with those lse when none of the compressing sequences was "
                             "compressed within the window, else in two passes",
                   "per_token_launch": "captured CUDA graph (input gather from the pool + query into the window "
                                       "ring + decode writing its lse into the ring + penalty and draw in one "
                                       "launch)" if use_graph else "direct calls"},
        "trace": {"generated": ev.generated, "decode_launches": ev.tokens, "steps_completed": ev.steps_completed,
                  "compressions": ev.compressions, "probes": len(ev.probes),
                  "boundary_scorings": {"one_pass_decode_lse": ev.lse_scorings, "two_pass": ev.two_pass_scorings},
                  "stops": sum(1 for p in ev.probes if p[2]),
                  "peak_cache_bytes": ev.peak_cache_bytes,
                  "mean_cache_bytes": ev.cache_byte_tokens / max(ev.tokens, 1),
                  "uncompressed_peak_cache_bytes": full_peak},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["gb300", "reference"], default="gb300")
    ap.add_argument("--workload", default="32b", choices=["tiny", "1.5b", "7b", "32b", "trace"])
    ap.add_argument("--reading", default="A", choices=["A", "B"], help="trace: budget base reading")
    ap.add_argument("--generated", type=int, default=0, help="trace: generated tokens (default 8192)")
    ap.add_argument("--no-graph", action="store_true", help="trace: per-token calls without a CUDA graph")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--ref-units", type=int, default=16, help="oracle sample: units (whole layers, or part of layer 0)")
    ap.add_argument("--ref-dec-steps", type=int, default=8, help="oracle sample: decode steps")
    ap.add_argument("--layers", type=int, help="override the layer count (profiling a smaller case)")
    ap.add_argument("--batch", type=int, help="override the batch (profiling a smaller case)")
    ap.add_argument("--decode-steps", type=int, help="override the decode steps (profiling a smaller case)")
    args = ap.parse_args()
    from paper_2608_04771_gb300 import workloads as W
    if args.workload == "trace":
        return run_trace(args)
    wl = W.WORKLOADS[args.workload]
    over = {k: v for k, v in (("layers", args.layers), ("batch", args.batch),
                               ("decode_steps", args.decode_steps)) if v is not None}
    if over:
        wl = wl.reduced(**over)
    if args.impl == "reference":
        run_reference(args, wl)
    else:
        run_gpu(args, wl)


if __name__ == "__main__":
    main()
