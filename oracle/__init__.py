"""fp64 CPU oracle for the ReCo hot path -- TEST INFRASTRUCTURE ONLY.

Only the test suite, ``__graft_entry__.smoke()`` and the benchmark's CPU-baseline
and reference arm may import this package.  The CUDA library under
``paper_2608_04771_gb300`` never imports it, and this package imports nothing
from there: the two share no code.  The arithmetic lives in ``reco_oracle.c``
(plain C, double precision); this module only compiles it with gcc and passes
numpy arrays to it.

Each wrapper names the paper passage it follows:
  retention_ratio / keep_count  -- Eq. 1, Sec. 3.2
  score_unit / score_cache      -- Eq. 2, Sec. 3.2 (plus the readings on scale,
                                   causal window, GQA mean and max-pool)
  select_unit / select_batch    -- top-m with the window kept, Sec. 3.2
  gather_unit                   -- compaction to m rows, Sec. 3.2
  decode_unit / decode_batch    -- softmax attention over the compacted cache
  penalty_band / reflect_penalty-- Eq. 3 and Eq. 4, Sec. 3.3
  penalty_sample                -- Eq. 3-4, then a draw from softmax(z~) (Sec. 3.3)
  probe_trigger                 -- two consecutive top-band rewards, Sec. 3.3
  answer_ppl                    -- Eq. 5 and Eq. 6, Sec. 3.3
"""
from __future__ import annotations

import ctypes
import os
import subprocess
from pathlib import Path

import numpy as np

_HERE = Path(__file__).resolve().parent
_SRC = _HERE / "reco_oracle.c"
_LIB_PATH = _HERE / "_build" / "liboracle.so"
_lib = None

_f32p = np.ctypeslib.ndpointer(dtype=np.float32, flags="C_CONTIGUOUS")
_f64p = np.ctypeslib.ndpointer(dtype=np.float64, flags="C_CONTIGUOUS")
_i32p = np.ctypeslib.ndpointer(dtype=np.int32, flags="C_CONTIGUOUS")
_u8p = np.ctypeslib.ndpointer(dtype=np.uint8, flags="C_CONTIGUOUS")


def build(force: bool = False) -> Path:
    """Compile reco_oracle.c into _build/liboracle.so (gcc, -O2, OpenMP, IEEE math)."""
    _LIB_PATH.parent.mkdir(exist_ok=True)
    if force or not _LIB_PATH.exists() or _LIB_PATH.stat().st_mtime < _SRC.stat().st_mtime:
        tmp = _LIB_PATH.with_suffix(".so.tmp%d" % os.getpid())
        cmd = ["gcc", "-O2", "-std=c11", "-fPIC", "-shared", "-fopenmp", "-fno-fast-math",
               "-ffp-contract=off", str(_SRC), "-o", str(tmp), "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    _lib = _bind(ctypes.CDLL(str(_LIB_PATH)))
    return _lib


def _bind(lib):
    """Declare the C signatures on a loaded oracle library."""
    c_int, c_double, c_float = ctypes.c_int, ctypes.c_double, ctypes.c_float
    lib.oracle_set_threads.argtypes = [c_int]
    lib.oracle_set_threads.restype = None
    lib.oracle_threads.argtypes = []
    lib.oracle_threads.restype = c_int
    lib.oracle_retention_ratio.argtypes = [_f32p, c_int, c_double, c_double]
    lib.oracle_retention_ratio.restype = c_double
    lib.oracle_keep_count.argtypes = [c_double, c_int, c_int]
    lib.oracle_keep_count.restype = c_int
    lib.oracle_score_unit.argtypes = [_f32p, _f32p, c_int, c_int, c_int, c_int, c_double, c_int,
                                      _f64p, ctypes.c_void_p]
    lib.oracle_score_unit.restype = None
    lib.oracle_score_cache.argtypes = [_f32p, _f32p, _i32p, c_int, c_int, c_int, c_int, c_int,
                                       c_int, c_int, c_int, c_double, _f64p]
    lib.oracle_score_cache.restype = None
    lib.oracle_select_unit.argtypes = [_f32p, c_int, c_int, c_int, _i32p]
    lib.oracle_select_unit.restype = c_int
    lib.oracle_select_batch.argtypes = [_f32p, _i32p, _i32p, c_int, c_int, c_int, c_int, c_int, _i32p]
    lib.oracle_select_batch.restype = None
    lib.oracle_gather_unit.argtypes = [_f32p, _i32p, c_int, c_int, _f32p]
    lib.oracle_gather_unit.restype = None
    lib.oracle_decode_unit.argtypes = [_f32p, _f32p, _f32p, c_int, c_int, c_double, _f64p,
                                       ctypes.c_void_p]
    lib.oracle_decode_unit.restype = None
    lib.oracle_decode_batch.argtypes = [_f32p, _f32p, _f32p, _i32p, c_int, c_int, c_int, c_int,
                                        c_int, c_int, c_double, _f64p, ctypes.c_void_p]
    lib.oracle_decode_batch.restype = None
    lib.oracle_penalty_band.argtypes = [c_float, c_float, c_float]
    lib.oracle_penalty_band.restype = c_int
    lib.oracle_reflect_penalty.argtypes = [_f32p, c_int, c_int, _i32p, c_int, _f32p, c_float,
                                           c_float, c_float, ctypes.c_void_p]
    lib.oracle_reflect_penalty.restype = c_int
    lib.oracle_penalty_sample.argtypes = [_f32p, c_int, c_int, _i32p, c_int, _f32p, c_float, c_float, c_float,
                                          _f32p, _i32p, _f64p, _f64p]
    lib.oracle_penalty_sample.restype = c_int
    lib.oracle_probe_trigger.argtypes = [c_float, c_float, c_float]
    lib.oracle_probe_trigger.restype = c_int
    lib.oracle_answer_ppl.argtypes = [_f32p, _i32p, ctypes.c_void_p, c_int, c_int, c_int, c_float,
                                      _f64p, _u8p]
    lib.oracle_answer_ppl.restype = None
    return lib


def _f32(a):
    return np.ascontiguousarray(a, dtype=np.float32)


def _i32(a):
    return np.ascontiguousarray(a, dtype=np.int32)


# ---- Eq. 1 -----------------------------------------------------------------
def set_threads(n: int) -> None:
    """Threads of the OpenMP loops over units (timing plumbing; results do not depend on it)."""
    _load().oracle_set_threads(int(n))


def threads() -> int:
    return int(_load().oracle_threads())


def retention_ratio(rewards, base: float = 0.25, delta: float = 0.1) -> float:
    r = _f32(rewards).ravel()
    return float(_load().oracle_retention_ratio(r, int(r.size), float(base), float(delta)))


def keep_count(ratio: float, L: int, w: int) -> int:
    return int(_load().oracle_keep_count(float(ratio), int(L), int(w)))


# ---- Eq. 2 -----------------------------------------------------------------
def score_unit(q, k, w: int, scale: float, pool: int = 1):
    """q: [G, w, d], k: [L, d].  Returns (raw [L], pooled [L-w]) in float64."""
    q = _f32(q)
    k = _f32(k)
    G, wq, d = q.shape
    assert wq == w and k.shape[1] == d
    L = k.shape[0]
    raw = np.zeros(L, np.float64)
    pooled = np.zeros(max(L - w, 0), np.float64)
    _load().oracle_score_unit(q, k, G, w, L, d, float(scale), int(pool), raw,
                              pooled.ctypes.data if pooled.size else None)
    return raw, pooled


def score_cache(q_win, K, lens, w: int, pool: int, scale: float):
    """q_win [Ly,B,Hq,w,d], K [Ly,B,Hkv,Lcap,d], lens [Ly,B,Hkv] -> pooled [Ly,B,Hkv,Lcap] f64."""
    q_win = _f32(q_win)
    K = _f32(K)
    lens = _i32(lens)
    Ly, B, Hq, wq, d = q_win.shape
    _, _, Hkv, Lcap, _ = K.shape
    out = np.zeros((Ly, B, Hkv, Lcap), np.float64)
    _load().oracle_score_cache(q_win, K, lens, Ly, B, Hq, Hkv, Lcap, d, w, int(pool), float(scale), out)
    return out


# ---- top-m and compaction ----------------------------------------------------
def select_unit(scores_f32, L: int, w: int, m: int):
    s = _f32(scores_f32).ravel()
    idx = np.zeros(max(m, 1), np.int32)
    got = _load().oracle_select_unit(s, int(L), int(w), int(m), idx)
    if got < 0:
        raise ValueError("bad sizes for selection")
    return idx[:got]


def select_batch(scores_f32, lens, keep, w: int):
    s = _f32(scores_f32)
    Ly, B, Hkv, Lcap = s.shape
    idx = np.full((Ly, B, Hkv, Lcap), -1, np.int32)
    _load().oracle_select_batch(s, _i32(lens), _i32(keep), Ly, B, Hkv, Lcap, int(w), idx)
    return idx


def gather_unit(rows, idx):
    rows = _f32(rows)
    idx = _i32(idx)
    out = np.zeros((idx.size, rows.shape[1]), np.float32)
    _load().oracle_gather_unit(rows, idx, int(idx.size), int(rows.shape[1]), out)
    return out


# ---- decode attention ---------------------------------------------------------
def decode_unit(q, k, v, length: int, scale: float):
    q = _f32(q).ravel()
    d = q.size
    out = np.zeros(d, np.float64)
    lse = np.zeros(1, np.float64)
    _load().oracle_decode_unit(q, _f32(k), _f32(v), int(length), d, float(scale), out, lse.ctypes.data)
    return out, float(lse[0])


def decode_batch(q, K, V, lens, scale: float):
    """q [Ly,B,Hq,d]; K,V [Ly,B,Hkv,Lcap,d]; lens [Ly,B,Hkv] -> (out f64, lse f64)."""
    q = _f32(q)
    K = _f32(K)
    V = _f32(V)
    Ly, B, Hq, d = q.shape
    Hkv, Lcap = K.shape[2], K.shape[3]
    out = np.zeros((Ly, B, Hq, d), np.float64)
    lse = np.zeros((Ly, B, Hq), np.float64)
    _load().oracle_decode_batch(q, K, V, _i32(lens), Ly, B, Hq, Hkv, Lcap, d, float(scale), out,
                                lse.ctypes.data)
    return out, lse


# ---- Eq. 3 / Eq. 4 ----------------------------------------------------------------
def penalty_band(v: float, tau_l: float = 0.4, tau_h: float = 0.8) -> int:
    return int(_load().oracle_penalty_band(float(np.float32(v)), float(np.float32(tau_l)),
                                           float(np.float32(tau_h))))


def reflect_penalty(logits, ids, rewards, tau_l=0.4, tau_h=0.8, beta=4.0):
    """Returns (penalised logits copy [B,V] f32, beta_i [B] f32, #ignored ids)."""
    z = _f32(logits).copy()
    B, V = z.shape
    ids = _i32(ids).ravel()
    r = _f32(rewards).ravel()
    beta_out = np.zeros(B, np.float32)
    bad = _load().oracle_reflect_penalty(z, B, V, ids, int(ids.size), r, float(tau_l), float(tau_h),
                                         float(beta), beta_out.ctypes.data)
    return z, beta_out, int(bad)


def penalty_sample(logits, ids, rewards, uniforms, tau_l=0.4, tau_h=0.8, beta=4.0):
    """Eq. 3-4 on a copy of logits [B,V], then one inversion draw per row at uniforms [B].
    Returns (penalised logits, tokens [B] int32, cdf_lo [B], cdf_hi [B], #ignored ids)."""
    z = _f32(logits).copy()
    B, V = z.shape
    ids = _i32(ids).ravel()
    tok = np.zeros(B, np.int32)
    lo = np.zeros(B, np.float64)
    hi = np.zeros(B, np.float64)
    bad = _load().oracle_penalty_sample(z, B, V, ids, int(ids.size), _f32(rewards).ravel(), float(tau_l),
                                        float(tau_h), float(beta), _f32(uniforms).ravel(), tok, lo, hi)
    return z, tok, lo, hi, int(bad)


def probe_trigger(v_prev: float, v_cur: float, tau_h: float = 0.8) -> bool:
    return bool(_load().oracle_probe_trigger(float(v_prev), float(v_cur), float(tau_h)))


# ---- Eq. 5 / Eq. 6 ----------------------------------------------------------------
def answer_ppl(logits, tokens, n_valid=None, tau_p: float = 1.1):
    z = _f32(logits)
    B, n, V = z.shape
    tok = _i32(tokens)
    nv = None if n_valid is None else _i32(n_valid)
    ppl = np.zeros(B, np.float64)
    stop = np.zeros(B, np.uint8)
    _load().oracle_answer_ppl(z, tok, None if nv is None else nv.ctypes.data, B, n, V,
                              float(tau_p), ppl, stop)
    return ppl, stop.astype(bool)
