"""The allocation-free answer-PPL entry point against the workspace one.

reco_answer_ppl_static serves callers that cannot give the library device memory
(a plug-in whose host engine has reserved the whole GPU, C code without a device
allocator): its scratch is a fixed array inside the library.  This file is
collected last so that a failure here leaves every other test already run."""
import numpy as np
import pytest
import torch

from helpers import PPL_RTOL
from paper_2608_04771_gb300 import reco
from paper_2608_04771_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    from paper_2608_04771_gb300 import build
    build.build()
    reco.lib()


def _both(z, tok, n_valid, tau_p=1.1):
    B, n, V = z.shape
    nv = None if n_valid is None else torch.tensor(n_valid, dtype=torch.int32, device=DEV)
    p_ws, s_ws = torch.empty(B, device=DEV), torch.empty(B, dtype=torch.uint8, device=DEV)
    ws = reco.workspace(reco.RECO_OP_PPL, None, B * n, DEV)
    reco.reco_answer_ppl(z, tok, nv, tau_p, p_ws, s_ws, ws)
    p_st, s_st = torch.full((B,), -1.0, device=DEV), torch.full((B,), 7, dtype=torch.uint8, device=DEV)
    reco.reco_answer_ppl_static(z, tok, nv, tau_p, p_st, s_st)
    reco.reco_check()
    a, b = p_ws.cpu().numpy().astype(np.float64), p_st.cpu().numpy().astype(np.float64)
    nan = np.isnan(a)
    assert np.array_equal(nan, np.isnan(b))
    assert np.all(np.abs(a[~nan] - b[~nan]) <= PPL_RTOL * np.abs(a[~nan]))
    assert torch.equal(s_ws, s_st)


def test_static_matches_workspace_entry_point_twice():
    wl = W.WORKLOADS["7b"].reduced(vocab=30000)
    z, tok = W.make_answer(wl, DEV)  # 8 x 32 rows: half the batch confident
    _both(z, tok, None)
    # a second call in a row, different sizes and ragged lengths, reusing the same array
    rng = np.random.default_rng(11)
    z2 = torch.from_numpy((rng.standard_normal((5, 40, 1001)) * 2).astype(np.float32)).to(DEV)
    tok2 = torch.from_numpy(rng.integers(0, 1001, (5, 40)).astype(np.int32)).to(DEV)
    _both(z2, tok2, [40, 3, 0, 17, 40])


def test_static_allocates_no_device_memory():
    """The defining property: no device memory is taken by the calls themselves.
    Inputs, outputs and a first call (which loads the kernels) come before the count."""
    wl = W.WORKLOADS["7b"].reduced(vocab=30000)
    z, tok = W.make_answer(wl, DEV)
    B = z.shape[0]
    ppl, stop = torch.empty(B, device=DEV), torch.empty(B, dtype=torch.uint8, device=DEV)
    reco.reco_answer_ppl_static(z, tok, None, 1.1, ppl, stop)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    reserved0 = torch.cuda.memory_reserved()
    for _ in range(2):
        reco.reco_answer_ppl_static(z, tok, None, 1.1, ppl, stop)
    torch.cuda.synchronize()
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0 and torch.cuda.memory_reserved() == reserved0
    reco.reco_check()


def test_static_rejects_more_rows_than_its_array():
    n = reco.RECO_PPL_STATIC_MAX_ROWS // 4 + 1
    z = torch.zeros((4, n, 4), device=DEV)
    tok = torch.zeros((4, n), dtype=torch.int32, device=DEV)
    ppl = torch.empty(4, device=DEV)
    stop = torch.empty(4, dtype=torch.uint8, device=DEV)
    with pytest.raises(reco.RecoError) as e:
        reco.reco_answer_ppl_static(z, tok, None, 1.1, ppl, stop)
    assert e.value.status == reco.RECO_EINVAL and "static scratch" in str(e.value)
    # the grid limits of the workspace entry point hold here too: same inputs, same status
    for B, n in ((65536, 1), (70000, 0)):
        z = torch.zeros((B, n, 4), device=DEV)
        tok = torch.zeros((B, n), dtype=torch.int32, device=DEV)
        ppl = torch.empty(B, device=DEV)
        stop = torch.empty(B, dtype=torch.uint8, device=DEV)
        ws = reco.workspace(reco.RECO_OP_PPL, None, B * n, DEV)
        with pytest.raises(reco.RecoError) as e1:
            reco.reco_answer_ppl(z, tok, None, 1.1, ppl, stop, ws)
        with pytest.raises(reco.RecoError) as e2:
            reco.reco_answer_ppl_static(z, tok, None, 1.1, ppl, stop)
        assert e1.value.status == e2.value.status == reco.RECO_EUNSUPPORTED
