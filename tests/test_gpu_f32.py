"""GPU parity of the single-precision variant (lv_attribute_f32) against the
fp64 oracle: T, shares and tenant totals within 1e-5 relative (plain relative
error, every coefficient positive); the tenant totals are also the exact sums of
the fp32 shares the call returned (each rounded to 2^-72 s)."""

from fractions import Fraction

import numpy as np
import pytest

import oracle
import workloads

pytestmark = pytest.mark.gpu
TOL = 1e-5


@pytest.fixture(scope="module")
def lv():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2608_08382_gb300
    return paper_2608_08382_gb300


def _run(lv, w):
    import torch
    ctx = lv.Context()
    b = lv.batches_to_device(w.p, w.c, w.phase, w.offsets, w.tenant, w.n_tenants)
    model = lv.make_model(w.coef, w.split)
    T = torch.full((w.n_batch,), float("nan"), dtype=torch.float32, device="cuda")
    S = torch.full((w.n_req,), float("nan"), dtype=torch.float32, device="cuda")
    acc = lv.TenantAcc(ctx, w.n_tenants)
    lv.lv_attribute_f32(ctx, model, b, T, S, acc)
    L = torch.empty(w.n_tenants, dtype=torch.float64, device="cuda")
    lv.lv_tenant_totals(ctx, acc, L)
    st = ctx.status()
    return T.cpu().numpy().astype(np.float64), S.cpu().numpy().astype(np.float64), L.cpu().numpy(), st


@pytest.mark.parametrize("cfg,scale", [(0, 1.0), (1, 0.01), (4, 0.01)])
def test_f32_parity(lv, cfg, scale):
    w = workloads.config(cfg, scale=scale)
    T, S, L, st = _run(lv, w)
    assert st == lv.LV_OK
    T_o, s_o = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
    nz = T_o != 0
    assert np.all(T[~nz] == 0)
    assert np.max(np.abs(T[nz] - T_o[nz]) / np.abs(T_o[nz])) <= TOL
    assert np.max(np.abs(S - s_o) / np.abs(s_o)) <= TOL
    L_o = oracle.tenant_totals(s_o, w.tenant, w.n_tenants)
    m = L_o != 0
    assert np.max(np.abs(L[m] - L_o[m]) / np.abs(L_o[m])) <= TOL
    for u in np.unique(w.tenant)[:16]:
        tot = sum(round(Fraction(v) * 2**72) for v in S[w.tenant == u].tolist())
        assert L[u] == float(Fraction(tot, 2**72))
