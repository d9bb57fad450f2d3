"""The C-ABI library on the CPU: it builds, loads, exports every symbol include/reco.h
declares, its host helpers agree with the oracle, and host-side argument checks
reject bad calls before any launch (no GPU needed, no compute calls)."""
import ctypes
import json
import os
import re

import numpy as np
import pytest

import oracle
from paper_2608_04771_gb300 import build as B
from paper_2608_04771_gb300 import reco

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    B.build()
    return reco.lib()


def declared_functions():
    text = open(os.path.join(ROOT, "include", "reco.h")).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*(reco_[a-z_0-9]+)\s*\(", text, flags=re.M)))


def test_every_declared_symbol_is_exported(L):
    names = declared_functions()
    assert len(names) >= 12
    assert set(names) == set(reco.EXPORTS)
    for n in names:
        assert hasattr(L, n), n
    out = os.popen(f"nm -D --defined-only {B.LIB}").read()
    for n in names:
        assert re.search(rf"\bT {n}\b", out), n


def test_retention_ratio_and_keep_count_match_oracle(L):
    g = json.load(open(os.path.join(ROOT, "tests", "golden", "eq1_retention.json")))
    for c in g["cases"]:
        r = reco.reco_retention_ratio(c["history"], c["base"], c["delta"])
        assert r == oracle.retention_ratio(c["history"], c["base"], c["delta"])
        assert reco.reco_keep_count(r, c["L"], c["w"]) == c["m"]
    rng = np.random.default_rng(0)
    for _ in range(2000):
        h = rng.random(int(rng.integers(1, 30))).astype(np.float32)
        base, delta = float(rng.uniform(0.1, 0.6)), float(rng.uniform(0, 0.35))
        r = reco.reco_retention_ratio(h, base, delta)
        assert r == oracle.retention_ratio(h, base, delta)  # bit-exact (same definition, same order)
        Lc = int(rng.integers(1, 40000))
        w = int(rng.integers(1, Lc + 1))
        assert reco.reco_keep_count(r, Lc, w) == oracle.keep_count(r, Lc, w)


def test_band_and_trigger_match_oracle(L):
    g = json.load(open(os.path.join(ROOT, "tests", "golden", "eq34_penalty.json")))
    for c in g["bands"]:
        assert reco.reco_penalty_band(c["v"], g["tau_l"], g["tau_h"]) == c["band"]
    for c in g["probe_trigger"]:
        assert reco.reco_probe_trigger(c["v_prev"], c["v_cur"], 0.8) == c["fire"]
    for v in np.linspace(0, 1, 1001, dtype=np.float32):
        assert reco.reco_penalty_band(float(v)) == oracle.penalty_band(float(v))


def test_host_helpers_reject_bad_input(L):
    with pytest.raises(reco.RecoError) as e:
        reco.reco_retention_ratio([], 0.25, 0.1)
    assert e.value.status == reco.RECO_EINVAL
    with pytest.raises(reco.RecoError):
        reco.reco_keep_count(0.25, 10, 11)  # w > L
    with pytest.raises(reco.RecoError):
        reco.reco_keep_count(0.25, 10, 0)


def _kv(**kw):
    d = dict(k=16, v=32, n_layers=2, B=3, H_q=8, H_kv=2, L_cap=100, d=128, dtype=reco.RECO_BF16)
    d.update(kw)
    return reco.reco_kv(d["k"], d["v"], d["n_layers"], d["B"], d["H_q"], d["H_kv"], d["L_cap"], d["d"],
                        d["dtype"])


def test_workspace_sizes(L):
    kv = _kv()
    s = reco.reco_workspace_bytes(reco.RECO_OP_SCORE, kv, 16)
    units, R = 2 * 3 * 2, 4 * 16
    assert s >= units * 100 * 4 + units * R * 4
    assert reco.reco_workspace_bytes(reco.RECO_OP_SELECT, kv) >= units * 100 * 4
    assert reco.reco_workspace_bytes(reco.RECO_OP_DECODE, kv) > 0
    assert reco.reco_workspace_bytes(reco.RECO_OP_PPL, None, 64) == 256
    # sampling: (max, sum) float pairs per 4096-logit segment of one row
    assert reco.reco_workspace_bytes(reco.RECO_OP_SAMPLE, None, 152064) == 38 * 8
    assert reco.reco_workspace_bytes(reco.RECO_OP_SAMPLE, None, 1) == 8
    with pytest.raises(reco.RecoError):
        reco.reco_workspace_bytes(reco.RECO_OP_SAMPLE, None, 0)
    with pytest.raises(reco.RecoError):
        reco.reco_workspace_bytes(reco.RECO_OP_SCORE, _kv(d=96), 16)
    with pytest.raises(reco.RecoError):
        reco.reco_workspace_bytes(reco.RECO_OP_SCORE, _kv(H_q=7), 16)


def test_device_calls_validate_before_launch(L):
    """Bad shapes, NULLs, misalignment and short workspaces fail with EINVAL/EUNSUPPORTED
    on the host; no kernel is launched (this machine has no GPU)."""
    kv = _kv()
    vp = ctypes.c_void_p
    ws = vp(256 * 1000)
    st = L.reco_score_cache(ctypes.byref(kv), vp(16), vp(16), None, 0, 7, 0.1, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"window" in L.reco_last_error()
    st = L.reco_score_cache(ctypes.byref(kv), vp(16), vp(16), None, 16, 4, 0.1, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"pool_kernel" in L.reco_last_error()
    st = L.reco_score_cache(ctypes.byref(kv), vp(16), vp(16), None, 16, 7, 0.1, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"workspace" in L.reco_last_error()
    st = L.reco_score_cache(ctypes.byref(_kv(k=17)), vp(16), vp(16), None, 16, 7, 0.1, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"aligned" in L.reco_last_error()
    # the lse form of Eq. 2 checks its row normalisers on top of reco_score_cache's checks
    st = L.reco_score_cache_lse(ctypes.byref(kv), vp(16), vp(16), None, None, 16, 7, 0.1, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"row_lse" in L.reco_last_error()
    st = L.reco_score_cache_lse(ctypes.byref(kv), vp(16), vp(16), None, vp(18), 16, 7, 0.1, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"aligned" in L.reco_last_error()
    st = L.reco_score_cache_lse(ctypes.byref(kv), vp(16), vp(16), None, vp(16), 0, 7, 0.1, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"window" in L.reco_last_error()
    st = L.reco_score_cache_lse(ctypes.byref(kv), vp(16), vp(16), None, vp(16), 16, 7, 0.1, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"workspace" in L.reco_last_error()
    st = L.reco_lse_push(vp(16), 0, vp(16), 4, vp(16), None)
    assert st == reco.RECO_EINVAL
    st = L.reco_lse_push(vp(16), 10, vp(16), 4, None, None)
    assert st == reco.RECO_EINVAL and b"NULL" in L.reco_last_error()
    st = L.reco_lse_push(vp(16), 10, vp(16), 4, vp(20), None)
    assert st == reco.RECO_EINVAL and b"aligned" in L.reco_last_error()
    st = L.reco_select_compact(ctypes.byref(kv), None, vp(16), vp(16), 16, None, ws, 10, None)
    assert st == reco.RECO_EINVAL
    st = L.reco_decode_attn(ctypes.byref(kv), vp(16), vp(16), None, vp(16), 0.1, vp(16), 0, None, ws, 10, None)
    assert st == reco.RECO_EINVAL and b"k_new" in L.reco_last_error()
    st = L.reco_decode_attn(ctypes.byref(_kv(H_q=34, H_kv=2)), vp(16), None, None, vp(16), 0.1, vp(16), 0,
                            None, ws, 10, None)
    assert st == reco.RECO_EUNSUPPORTED
    st = L.reco_reflect_penalty(vp(16), 0, 10, vp(16), 1, vp(16), 0.4, 0.8, 4.0, None, None)
    assert st == reco.RECO_EINVAL
    st = L.reco_answer_ppl(vp(16), vp(16), None, 2, 4, 10, 1.1, vp(16), vp(16), None, 0, None)
    assert st == reco.RECO_EINVAL and b"workspace" in L.reco_last_error()


def test_penalty_sample_validates_before_launch(L):
    vp = ctypes.c_void_p
    ws = vp(256 * 1000)
    args = dict(logits=vp(256), B=4, V=1000, ids=vp(512), n_ids=2, rewards=vp(768), tau_l=0.4, tau_h=0.8, beta=4.0,
                uniforms=vp(1024), tokens=vp(1280), beta_out=None, ws=ws, ws_bytes=4 * 8, stream=None)

    def call(**kw):
        a = dict(args, **kw)
        return L.reco_penalty_sample(a["logits"], a["B"], a["V"], a["ids"], a["n_ids"], a["rewards"], a["tau_l"],
                                     a["tau_h"], a["beta"], a["uniforms"], a["tokens"], a["beta_out"], a["ws"],
                                     a["ws_bytes"], a["stream"])
    assert call(uniforms=None) == reco.RECO_EINVAL and b"NULL" in L.reco_last_error()
    assert call(tokens=vp(1281)) == reco.RECO_EINVAL and b"aligned" in L.reco_last_error()
    assert call(ws_bytes=4 * 8 - 1) == reco.RECO_EINVAL and b"workspace" in L.reco_last_error()
    assert call(V=4096 * 1024 + 1) == reco.RECO_EUNSUPPORTED
    assert call(beta=-1.0) == reco.RECO_EINVAL
    assert call(B=0) == reco.RECO_EINVAL


def test_split_select_compact_and_ring_decode_validate_before_launch(L):
    """reco_select_topm, reco_compact and reco_decode_attn_ring (also a q_ring off a 16-byte
    boundary) reject bad arguments on the host, before any launch."""
    kv = _kv()
    vp = ctypes.c_void_p
    ws = vp(256 * 1000)
    big = 1 << 30
    st = L.reco_select_topm(ctypes.byref(kv), vp(16), vp(16), vp(16), 16, None, ws, big, None)
    assert st == reco.RECO_EINVAL and b"kept_idx" in L.reco_last_error()
    st = L.reco_select_topm(ctypes.byref(kv), vp(16), vp(16), vp(16), 0, vp(16), ws, big, None)
    assert st == reco.RECO_EINVAL and b"window" in L.reco_last_error()
    st = L.reco_select_topm(ctypes.byref(kv), vp(16), vp(16), vp(18), 16, vp(16), ws, big, None)
    assert st == reco.RECO_EINVAL and b"aligned" in L.reco_last_error()
    st = L.reco_select_topm(ctypes.byref(kv), vp(16), vp(16), vp(16), 16, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"workspace" in L.reco_last_error()
    # the selection alone does not touch the cache: NULL K/V pointers are accepted there ...
    st = L.reco_select_topm(ctypes.byref(_kv(k=0, v=0)), vp(16), vp(16), vp(16), 16, vp(16), ws, 10, None)
    assert st == reco.RECO_EINVAL and b"workspace" in L.reco_last_error()
    # ... but not by the compaction
    st = L.reco_compact(ctypes.byref(_kv(k=0, v=0)), vp(16), vp(16), vp(16), 16, None)
    assert st == reco.RECO_EINVAL and b"NULL" in L.reco_last_error()
    st = L.reco_compact(ctypes.byref(kv), vp(16), vp(16), None, 16, None)
    assert st == reco.RECO_EINVAL and b"keep" in L.reco_last_error()
    st = L.reco_compact(ctypes.byref(kv), vp(17), vp(16), vp(16), 16, None)
    assert st == reco.RECO_EINVAL and b"aligned" in L.reco_last_error()
    st = L.reco_compact(ctypes.byref(kv), vp(16), vp(16), vp(16), 101, None)
    assert st == reco.RECO_EINVAL and b"window" in L.reco_last_error()
    dec = lambda kv_, ring, slots, slot, q_ring=None: L.reco_decode_attn_ring(  # noqa: E731
        ctypes.byref(kv_), vp(16), None, None, vp(16), 0.1, vp(16), 0, ring, slots, slot, q_ring, ws, 10, None)
    assert dec(kv, vp(16), 0, vp(16)) == reco.RECO_EINVAL and b"slots" in L.reco_last_error()
    assert dec(kv, None, 4, vp(16)) == reco.RECO_EINVAL
    assert dec(kv, vp(16), 4, vp(20)) == reco.RECO_EINVAL and b"aligned" in L.reco_last_error()
    assert dec(kv, vp(16), 4, vp(16), vp(24)) == reco.RECO_EINVAL and b"q_ring" in L.reco_last_error()
    # past its own checks it applies reco_decode_attn's (here: the workspace is too short)
    assert dec(kv, vp(16), 4, vp(16)) == reco.RECO_EINVAL and b"workspace" in L.reco_last_error()
    assert dec(_kv(H_q=34, H_kv=2), vp(16), 4, vp(16)) == reco.RECO_EUNSUPPORTED


def test_copy_row_validates_before_launch(L):
    vp = ctypes.c_void_p
    assert L.reco_copy_row(vp(256), 0, 64, vp(8), vp(256), None) == reco.RECO_EINVAL
    assert L.reco_copy_row(vp(256), 4, 72 + 1, vp(8), vp(256), None) == reco.RECO_EINVAL
    assert L.reco_copy_row(vp(256), 4, 0, vp(8), vp(256), None) == reco.RECO_EINVAL
    assert L.reco_copy_row(vp(264), 4, 64, vp(8), vp(256), None) == reco.RECO_EINVAL
    assert b"aligned" in L.reco_last_error()
    assert L.reco_copy_row(vp(256), 4, 64, vp(12), vp(256), None) == reco.RECO_EINVAL
    assert L.reco_copy_row(vp(256), 4, 64, None, vp(256), None) == reco.RECO_EINVAL
    assert L.reco_copy_row(vp(256), 4, 64, vp(8), vp(260), None) == reco.RECO_EINVAL


def test_decode_workspace_counts_a_ticket_per_half_unit_above_8_heads(L):
    """A unit of more than 8 query heads per KV head runs as two units on the tensor path, with
    a merge ticket each: the workspace holds one more int per unit."""
    w8 = reco.reco_workspace_bytes(reco.RECO_OP_DECODE, _kv(H_q=16, H_kv=2))
    w16 = reco.reco_workspace_bytes(reco.RECO_OP_DECODE, _kv(H_q=32, H_kv=2))
    parts = 4096  # partial slots, each G x (2 + d) floats
    assert w16 - w8 >= parts * 8 * (2 + 128) * 4  # the partials of 8 more heads per slot
    kv = _kv(H_q=32, H_kv=2, n_layers=64, B=16)  # 2048 units: the counters alone differ by 8 KB
    kv8 = _kv(H_q=16, H_kv=2, n_layers=64, B=16)
    g = reco.reco_workspace_bytes(reco.RECO_OP_DECODE, kv) - reco.reco_workspace_bytes(reco.RECO_OP_DECODE, kv8)
    assert g >= parts * 8 * (2 + 128) * 4 + 2048 * 4 - 512
