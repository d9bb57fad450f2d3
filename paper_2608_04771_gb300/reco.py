"""Thin ctypes binding over libreco.so, with the C ABI's names (include/reco.h).

Only argument marshalling happens here: torch tensors supply device pointers and
the current CUDA stream; every step of the hot path runs in the library's kernels.
There is no fallback: if the library is missing or a call fails, this module raises.
"""
from __future__ import annotations

import ctypes
from pathlib import Path

import torch

_LIB_PATH = Path(__file__).resolve().parent / "_build" / "libreco.so"
_lib = None

RECO_OK, RECO_EINVAL, RECO_EUNSUPPORTED, RECO_ECUDA, RECO_EDEVICE = range(5)
RECO_F32, RECO_BF16 = 0, 1
RECO_OP_SCORE, RECO_OP_SELECT, RECO_OP_DECODE, RECO_OP_PPL, RECO_OP_SAMPLE = range(5)

EXPORTS = ("reco_retention_ratio", "reco_keep_count", "reco_penalty_band", "reco_probe_trigger",
           "reco_workspace_bytes", "reco_last_error", "reco_check", "reco_score_cache",
           "reco_score_cache_lse", "reco_lse_push", "reco_copy_row", "reco_select_compact", "reco_select_topm", "reco_compact",
           "reco_decode_attn", "reco_decode_attn_ring", "reco_reflect_penalty", "reco_penalty_sample", "reco_answer_ppl",
           "reco_answer_ppl_static")
RECO_PPL_STATIC_MAX_ROWS = 65536


class RecoError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"reco status {status}: {msg}")
        self.status = status


class reco_kv(ctypes.Structure):
    _fields_ = [("k", ctypes.c_void_p), ("v", ctypes.c_void_p), ("n_layers", ctypes.c_int),
                ("B", ctypes.c_int), ("H_q", ctypes.c_int), ("H_kv", ctypes.c_int),
                ("L_cap", ctypes.c_int), ("d", ctypes.c_int), ("dtype", ctypes.c_int)]


def library_path() -> Path:
    return _LIB_PATH


def lib():
    """Load libreco.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not _LIB_PATH.exists():
        raise RuntimeError(f"{_LIB_PATH} is missing: build it with __graft_entry__.build() "
                           "or `python -m paper_2608_04771_gb300.build`")
    L = ctypes.CDLL(str(_LIB_PATH))
    vp, i32, f32, f64, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_float, ctypes.c_double, ctypes.c_size_t
    kvp = ctypes.POINTER(reco_kv)
    L.reco_retention_ratio.argtypes = [vp, i32, f64, f64, ctypes.POINTER(f64)]
    L.reco_keep_count.argtypes = [f64, i32, i32, ctypes.POINTER(ctypes.c_int32)]
    L.reco_penalty_band.argtypes = [f32, f32, f32]
    L.reco_penalty_band.restype = i32
    L.reco_probe_trigger.argtypes = [f32, f32, f32]
    L.reco_probe_trigger.restype = i32
    L.reco_workspace_bytes.argtypes = [i32, kvp, i32, ctypes.POINTER(sz)]
    L.reco_last_error.argtypes = []
    L.reco_last_error.restype = ctypes.c_char_p
    L.reco_check.argtypes = [vp]
    L.reco_score_cache.argtypes = [kvp, vp, vp, vp, i32, i32, f32, vp, vp, sz, vp]
    L.reco_score_cache_lse.argtypes = [kvp, vp, vp, vp, vp, i32, i32, f32, vp, vp, sz, vp]
    L.reco_lse_push.argtypes = [vp, ctypes.c_int64, vp, i32, vp, vp]
    L.reco_copy_row.argtypes = [vp, ctypes.c_int64, ctypes.c_int64, vp, vp, vp]
    L.reco_select_compact.argtypes = [kvp, vp, vp, vp, i32, vp, vp, sz, vp]
    L.reco_select_topm.argtypes = [kvp, vp, vp, vp, i32, vp, vp, sz, vp]
    L.reco_compact.argtypes = [kvp, vp, vp, vp, i32, vp]
    L.reco_decode_attn.argtypes = [kvp, vp, vp, vp, vp, f32, vp, i32, vp, vp, sz, vp]
    L.reco_decode_attn_ring.argtypes = [kvp, vp, vp, vp, vp, f32, vp, i32, vp, i32, vp, vp, vp, sz, vp]
    L.reco_reflect_penalty.argtypes = [vp, i32, i32, vp, i32, vp, f32, f32, f32, vp, vp]
    L.reco_penalty_sample.argtypes = [vp, i32, i32, vp, i32, vp, f32, f32, f32, vp, vp, vp, vp, sz, vp]
    L.reco_answer_ppl.argtypes = [vp, vp, vp, i32, i32, i32, f32, vp, vp, vp, sz, vp]
    L.reco_answer_ppl_static.argtypes = [vp, vp, vp, i32, i32, i32, f32, vp, vp, vp]
    for name in ("reco_retention_ratio", "reco_keep_count", "reco_workspace_bytes", "reco_check",
                 "reco_score_cache", "reco_score_cache_lse", "reco_lse_push", "reco_copy_row", "reco_select_compact",
                 "reco_select_topm", "reco_compact",
                 "reco_decode_attn", "reco_decode_attn_ring", "reco_reflect_penalty", "reco_penalty_sample",
                 "reco_answer_ppl",
                 "reco_answer_ppl_static"):
        getattr(L, name).restype = i32
    _lib = L
    return L


def _ok(status: int):
    if status != RECO_OK:
        raise RecoError(status, lib().reco_last_error().decode())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


_raw_stream = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream(stream):
    if stream is None:
        if _raw_stream is not None:  # the current stream's handle without building a Stream object
            return ctypes.c_void_p(_raw_stream(torch.cuda.current_device()))
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype_code(dt):
    if dt == torch.float32:
        return RECO_F32
    if dt == torch.bfloat16:
        return RECO_BF16
    raise TypeError(f"unsupported dtype {dt}")


def make_kv(K: torch.Tensor, V: torch.Tensor, H_q: int) -> reco_kv:
    """Describe contiguous [layers, B, H_kv, L_cap, d] K and V tensors."""
    if K.shape != V.shape or K.dtype != V.dtype or K.dim() != 5:
        raise ValueError("K and V must be [layers, B, H_kv, L_cap, d] with equal shape and dtype")
    if not (K.is_contiguous() and V.is_contiguous()):
        raise ValueError("K and V must be contiguous")
    Ly, B, Hkv, Lcap, d = K.shape
    return reco_kv(K.data_ptr(), V.data_ptr(), Ly, B, H_q, Hkv, Lcap, d, _dtype_code(K.dtype))


# ---------------------------------------------------------------- host helpers
def reco_retention_ratio(rewards, base: float = 0.25, delta: float = 0.1) -> float:
    import numpy as np
    r = np.ascontiguousarray(rewards, dtype=np.float32).ravel()
    out = ctypes.c_double()
    _ok(lib().reco_retention_ratio(r.ctypes.data, int(r.size), float(base), float(delta), ctypes.byref(out)))
    return out.value


def reco_keep_count(ratio: float, L: int, w: int) -> int:
    out = ctypes.c_int32()
    _ok(lib().reco_keep_count(float(ratio), int(L), int(w), ctypes.byref(out)))
    return out.value


def reco_penalty_band(v: float, tau_l: float = 0.4, tau_h: float = 0.8) -> int:
    return lib().reco_penalty_band(v, tau_l, tau_h)


def reco_probe_trigger(v_prev: float, v_cur: float, tau_h: float = 0.8) -> bool:
    return bool(lib().reco_probe_trigger(v_prev, v_cur, tau_h))


def reco_workspace_bytes(op: int, kv: reco_kv | None, w: int = 0) -> int:
    out = ctypes.c_size_t()
    _ok(lib().reco_workspace_bytes(op, ctypes.byref(kv) if kv is not None else None, int(w),
                                   ctypes.byref(out)))
    return out.value


def workspace(op: int, kv: reco_kv | None, w: int = 0, device="cuda") -> torch.Tensor:
    """A zero-filled workspace (the decode call needs its counters zero before first use)."""
    n = reco_workspace_bytes(op, kv, w)
    return torch.zeros(max(n, 256), dtype=torch.uint8, device=device)


def reco_check(stream=None):
    _ok(lib().reco_check(_stream(stream)))


# ---------------------------------------------------------------- device calls
def reco_score_cache(kv: reco_kv, q_win, lens, w: int, pool_kernel: int, scale: float, scores, ws, keep=None,
                     stream=None):
    """keep (optional [B] int32): skip the units of sequences with keep[b] >= lens."""
    _ok(lib().reco_score_cache(ctypes.byref(kv), _ptr(q_win), _ptr(lens), _ptr(keep), int(w), int(pool_kernel),
                               float(scale), _ptr(scores), _ptr(ws), ws.numel(), _stream(stream)))


def reco_lse_push(lse, ring, slot, stream=None):
    """ring[slot] = ring[slot + S] = lse (flattened); slot = (slot + 1) % S, on the device.
    ring [2 * S, n] float32 (the second half mirrors the first), slot a one-element int64
    device tensor."""
    n = lse.numel()
    if ring.dim() < 2 or ring[0].numel() != n or ring.shape[0] % 2:
        raise ValueError("ring must have an even number of rows of lse.numel() floats")
    _ok(lib().reco_lse_push(_ptr(lse), n, _ptr(ring), int(ring.shape[0]) // 2, _ptr(slot), _stream(stream)))


def reco_copy_row(src, index, dst, stream=None):
    """dst = src[index] on the device: src [rows, ...] (each row a multiple of 16 bytes),
    index a one-element int64 device tensor, dst a tensor of one row's bytes."""
    rows = src.shape[0]
    row_bytes = src[0].numel() * src.element_size()
    if not src.is_contiguous() or not dst.is_contiguous() or dst.numel() * dst.element_size() != row_bytes:
        raise ValueError("src and dst must be contiguous and dst one row of src")
    if index.dtype != torch.int64 or index.numel() != 1:
        raise ValueError("index must be a one-element int64 tensor")
    _ok(lib().reco_copy_row(_ptr(src), rows, row_bytes, _ptr(index), _ptr(dst), _stream(stream)))


def reco_score_cache_lse(kv: reco_kv, q_win, lens, row_lse, w: int, pool_kernel: int, scale: float, scores, ws,
                         keep=None, stream=None):
    """Eq. 2 with the window rows' normalisers from the decode: row_lse [w, Ly, B, Hq]
    float32 holds the lse reco_decode_attn returned for each window token's query."""
    _ok(lib().reco_score_cache_lse(ctypes.byref(kv), _ptr(q_win), _ptr(lens), _ptr(keep), _ptr(row_lse), int(w),
                                   int(pool_kernel), float(scale), _ptr(scores), _ptr(ws), ws.numel(),
                                   _stream(stream)))


def reco_select_compact(kv: reco_kv, scores, lens, keep, w: int, kept_idx, ws, stream=None):
    _ok(lib().reco_select_compact(ctypes.byref(kv), _ptr(scores), _ptr(lens), _ptr(keep), int(w),
                                  _ptr(kept_idx), _ptr(ws), ws.numel(), _stream(stream)))


def reco_select_topm(kv: reco_kv, scores, lens, keep, w: int, kept_idx, ws, stream=None):
    """The selection of reco_select_compact alone: kept indices written, cache and lens untouched."""
    _ok(lib().reco_select_topm(ctypes.byref(kv), _ptr(scores), _ptr(lens), _ptr(keep), int(w), _ptr(kept_idx),
                               _ptr(ws), ws.numel(), _stream(stream)))


def reco_compact(kv: reco_kv, kept_idx, lens, keep, w: int, stream=None):
    """The compaction of reco_select_compact alone, to the rows kept_idx names."""
    _ok(lib().reco_compact(ctypes.byref(kv), _ptr(kept_idx), _ptr(lens), _ptr(keep), int(w), _stream(stream)))


def reco_decode_attn(kv: reco_kv, q, k_new, v_new, lens, scale: float, out, lse, ws, stream=None):
    _ok(lib().reco_decode_attn(ctypes.byref(kv), _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(lens),
                               float(scale), _ptr(out), _dtype_code(out.dtype), _ptr(lse), _ptr(ws),
                               ws.numel(), _stream(stream)))


def reco_decode_attn_ring(kv: reco_kv, q, k_new, v_new, lens, scale: float, out, ring, slot, ws, stream=None,
                          q_ring=None):
    """reco_decode_attn with the lse written into ring rows slot and slot + S (ring [2 * S, n]
    float32) and slot (one-element int64 device tensor) advanced, on the device; with
    q_ring ([Ly, B, Hq, S, d], q's dtype) each head's query also goes to its row slot."""
    if ring.dim() < 2 or ring.shape[0] % 2:
        raise ValueError("ring must have an even number of rows")
    S = int(ring.shape[0]) // 2
    if q_ring is not None and (q_ring.dim() != 5 or q_ring.shape[3] != S or q_ring.dtype != q.dtype
                               or tuple(q_ring.shape[:3]) + (q_ring.shape[4],) != tuple(q.shape)
                               or not q_ring.is_contiguous()):
        raise ValueError("q_ring must be a contiguous [Ly, B, Hq, S, d] tensor of q's dtype")
    _ok(lib().reco_decode_attn_ring(ctypes.byref(kv), _ptr(q), _ptr(k_new), _ptr(v_new), _ptr(lens), float(scale),
                                    _ptr(out), _dtype_code(out.dtype), _ptr(ring), S, _ptr(slot), _ptr(q_ring),
                                    _ptr(ws), ws.numel(), _stream(stream)))


def reco_reflect_penalty(logits, ids, rewards, tau_l=0.4, tau_h=0.8, beta=4.0, beta_out=None,
                         stream=None):
    B, V = logits.shape
    _ok(lib().reco_reflect_penalty(_ptr(logits), B, V, _ptr(ids), ids.numel(), _ptr(rewards),
                                   float(tau_l), float(tau_h), float(beta), _ptr(beta_out),
                                   _stream(stream)))


def sample_workspace(B: int, V: int, device="cuda") -> torch.Tensor:
    """Workspace for reco_penalty_sample over B rows of V logits."""
    n = B * reco_workspace_bytes(RECO_OP_SAMPLE, None, V)
    return torch.empty(max(n, 256), dtype=torch.uint8, device=device)


def reco_penalty_sample(logits, ids, rewards, uniforms, tokens, ws, tau_l=0.4, tau_h=0.8, beta=4.0, beta_out=None,
                        stream=None):
    B, V = logits.shape
    _ok(lib().reco_penalty_sample(_ptr(logits), B, V, _ptr(ids), ids.numel(), _ptr(rewards), float(tau_l),
                                  float(tau_h), float(beta), _ptr(uniforms), _ptr(tokens), _ptr(beta_out), _ptr(ws),
                                  ws.numel(), _stream(stream)))


def _ppl_args(logits, tokens, n_valid):
    """[B, n, V] float32 logits and [B, n] int32 tokens, both contiguous (strides are not passed)."""
    if logits.dim() != 3 or logits.dtype != torch.float32 or not logits.is_contiguous():
        raise ValueError("logits must be a contiguous float32 [B, n, V] tensor")
    B, n, V = logits.shape
    if tokens.shape != (B, n) or tokens.dtype != torch.int32 or not tokens.is_contiguous():
        raise ValueError("tokens must be a contiguous int32 [B, n] tensor")
    if n_valid is not None and (n_valid.numel() != B or n_valid.dtype != torch.int32 or not n_valid.is_contiguous()):
        raise ValueError("n_valid must be a contiguous int32 [B] tensor")
    return B, n, V


def reco_answer_ppl(logits, tokens, n_valid, tau_p, ppl, stop, ws, stream=None):
    B, n, V = _ppl_args(logits, tokens, n_valid)
    _ok(lib().reco_answer_ppl(_ptr(logits), _ptr(tokens), _ptr(n_valid), B, n, V, float(tau_p),
                              _ptr(ppl), _ptr(stop), _ptr(ws), ws.numel(), _stream(stream)))


def reco_answer_ppl_static(logits, tokens, n_valid, tau_p, ppl, stop, stream=None):
    """reco_answer_ppl without a workspace: the library's fixed scratch array is used."""
    B, n, V = _ppl_args(logits, tokens, n_valid)
    _ok(lib().reco_answer_ppl_static(_ptr(logits), _ptr(tokens), _ptr(n_valid), B, n, V, float(tau_p),
                                     _ptr(ppl), _ptr(stop), _stream(stream)))
