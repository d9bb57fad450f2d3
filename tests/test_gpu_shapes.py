"""Head shapes, windows, pool widths and dtypes beyond the named workloads, each run
score -> select/compact -> decode against the oracle (see test_gpu_pipeline)."""
import ctypes

import pytest
import torch

from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W
from test_gpu_pipeline import run_pipeline

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


BASE = W.WORKLOADS["7b"]
CASES = {
    # name: overrides                                       path exercised
    "mha_g1": dict(h_q=4, h_kv=4, w=16, L=900),            # G = 1
    "g3_d64_pool3": dict(h_q=6, h_kv=2, w=8, d=64, pool=3, L=700),
    "g4_d64_r160": dict(h_q=8, h_kv=2, w=40, d=64, L=1100),  # 2 query tiles at d = 64: pass 1 on 256-key tiles
    "g7_short_units": dict(L=200),                           # 2 query tiles, every unit inside one 256-key tile
    "g8_r256": dict(h_q=16, h_kv=2, w=32, L=1300),         # tensor decode at G = 8; pass 2 N = 256
    "g16_split_decode": dict(h_q=16, h_kv=1, w=16, L=800),  # G = 16: the TMA decode as two 8-head units
    "w1_pool1": dict(w=1, pool=1, L=600),                  # one window query, Eq. 2 without pooling
    "r320_pool9": dict(h_q=10, h_kv=2, w=64, pool=9, L=1500),  # 32B-class window: 3 query tiles, 4 x 80 columns
    "r384": dict(h_q=12, h_kv=2, w=64, L=1000),            # 3 query tiles, full
    "r448_7b_heads_w64": dict(w=64, L=1200),               # G = 7 with w = 64: 4 query tiles, 4 x 112 columns
    "r512_max": dict(h_q=8, h_kv=1, w=64, L=1000),         # largest tensor-core window
    "fp32_d128": dict(dtype="f32", d=128, L=600),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_pipeline_shape(name):
    wl = BASE.reduced(layers=1, batch=2, decode_steps=2, **CASES[name])
    run_pipeline(wl)


def test_window_rows_beyond_both_scoring_paths_are_rejected():
    wl = BASE.reduced(layers=1, batch=1, h_q=8, h_kv=1, w=66, L=300, decode_steps=0)  # G*w = 528
    K, V = W.make_cache(wl, "cuda", canary=False)
    kv = reco.make_kv(K, V, wl.h_q)
    st = reco.lib().reco_score_cache(ctypes.byref(kv), ctypes.c_void_p(K.data_ptr()), ctypes.c_void_p(16),
                                     None, wl.w, 7, 0.1, ctypes.c_void_p(16), ctypes.c_void_p(256 * 4096), 1 << 40, None)
    assert st == reco.RECO_EUNSUPPORTED
