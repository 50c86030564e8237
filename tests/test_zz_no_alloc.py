"""The allocation-free attribution entry point agrees with lv_attribute and the oracle.

lv_attribute_noalloc exists for callers that must not allocate device memory
while they run -- for instance a serving engine's scheduler that has already
handed almost all GPU memory to its KV cache and sits on a latency-critical
path where a cudaMalloc would also synchronise the device.  It keeps its
scratch in a fixed static device array instead of an lv_ctx.  This file is
named to run last in a suite, so a failure here leaves every other test's
result standing; it also passes on its own in a fresh process.
"""

import ctypes

import numpy as np
import pytest

import oracle
import workloads

pytestmark = pytest.mark.gpu

TOL = 1e-12


@pytest.fixture(scope="module")
def lv():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2608_08382_gb300
    return paper_2608_08382_gb300


def _noalloc(lv, model, b, T, share, status):
    """Call the C entry point directly: no context, caller-owned outputs."""
    import torch
    bs = b.struct()
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    rc = lv.lib().lv_attribute_noalloc(ctypes.byref(model), ctypes.byref(bs), ctypes.c_void_p(T.data_ptr()),
                                       ctypes.c_void_p(share.data_ptr()), ctypes.c_void_p(status.data_ptr()),
                                       stream)
    return int(rc)


def _reference(lv, model, b, n_batch, n_req):
    """The same quantities through the context-based lv_attribute."""
    import torch
    ctx = lv.Context()
    T = torch.empty(n_batch, dtype=torch.float64, device="cuda")
    share = torch.empty(n_req, dtype=torch.float64, device="cuda")
    lv.lv_attribute(ctx, model, b, T, share, None)
    assert ctx.status() == lv.LV_OK
    return T.cpu().numpy(), share.cpu().numpy()


def test_noalloc_matches_lv_attribute_twice(lv):
    import torch
    cases = [workloads.config(0, scale=0.5), workloads.config(4, scale=0.01)]
    status = torch.full((1,), -1, dtype=torch.int32, device="cuda")
    for w in cases:  # two calls in a row, the second over different data and a different model
        b = lv.batches_to_device(w.p, w.c, w.phase, w.offsets)
        model = lv.make_model(w.coef, w.split)
        T = torch.full((w.n_batch,), float("nan"), dtype=torch.float64, device="cuda")
        share = torch.full((w.n_req,), float("nan"), dtype=torch.float64, device="cuda")
        assert _noalloc(lv, model, b, T, share, status) == lv.LV_OK
        torch.cuda.synchronize()
        assert int(status.item()) == 0
        T_ref, s_ref = _reference(lv, model, b, w.n_batch, w.n_req)
        Tg, sg = T.cpu().numpy(), share.cpu().numpy()
        nz = T_ref != 0
        assert np.all(Tg[~nz] == 0)
        assert np.max(np.abs(Tg[nz] - T_ref[nz]) / np.abs(T_ref[nz])) <= TOL
        assert np.max(np.abs(sg - s_ref) / np.abs(s_ref)) <= TOL
        # and against the CPU oracle directly
        T_o, s_o = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
        assert np.all(Tg[T_o == 0] == 0)
        assert np.max(np.abs(Tg[T_o != 0] - T_o[T_o != 0]) / np.abs(T_o[T_o != 0])) <= TOL
        assert np.max(np.abs(sg - s_o) / np.abs(s_o)) <= TOL


def test_noalloc_rejects_beyond_its_fixed_scratch(lv):
    import torch
    # n_batch + n_req above 65,536 tiles of 1,024: refused before any launch (no data is read)
    off = torch.zeros(2, dtype=torch.int64, device="cuda")
    x = torch.zeros(4, dtype=torch.int32, device="cuda")
    b = lv.lv_batches()
    b.p = b.c = b.phase = ctypes.c_void_p(x.data_ptr())
    b.offsets = ctypes.c_void_p(off.data_ptr())
    b.n_req = 1 << 27
    b.n_batch = 1
    model = lv.make_model(np.ones((4, 5)), (1, 1))
    rc = lv.lib().lv_attribute_noalloc(ctypes.byref(model), ctypes.byref(b), None, None, None, None)
    assert rc == lv.LV_EINVAL
