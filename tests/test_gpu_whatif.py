"""GPU parity of lv_whatif against the oracle, which materialises every batch B + {j}.

Tolerance 1e-12 relative for T_new; shares relative to max(|oracle|, T_new/n').
The fp64 arithmetic mode follows the oracle's rounding sequence bit for bit.
"""

import json
import os

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


@pytest.fixture(scope="module")
def ctx(lv):
    return lv.Context()


def _run(lv, ctx, off, p, c, ph, pn, cn, phn, coef, split, arith=0):
    import torch
    ctx.set_arith(arith)
    cand = lv.batches_to_device(p, c, ph, off)
    t = lambda a: torch.as_tensor(np.ascontiguousarray(a, dtype=np.int32), device="cuda")  # noqa: E731
    npd, nc = len(pn), len(off) - 1
    T = torch.full((npd, nc), float("nan"), dtype=torch.float64, device="cuda")
    S = torch.full((npd, nc), float("nan"), dtype=torch.float64, device="cuda")
    lv.lv_whatif(ctx, lv.make_model(coef, split), cand, t(pn), t(cn), t(phn), T, S)
    st = ctx.status()
    ctx.set_arith(0)
    return T.cpu().numpy(), S.cpu().numpy(), st


def _check(off, p, c, ph, pn, cn, phn, coef, split, T, S):
    To, So = oracle.whatif(off, p, c, ph, pn, cn, phn, split, coef)
    assert np.max(np.abs(T - To) / np.abs(To)) <= TOL
    assert np.max(np.abs(S - So) / np.abs(So)) <= TOL
    return To, So


def test_whatif_hand_case(lv, ctx, golden_dir):
    g = json.load(open(os.path.join(golden_dir, "eq1_hand_cases.json")))
    w = g["whatif"]
    for arith in (0, 1):
        T, S, st = _run(lv, ctx, w["cand_offsets"], w["cand_p"], w["cand_c"], w["cand_phase"], w["p_new"], w["c_new"],
                        w["phase_new"], np.array(g["coef"], dtype=float), g["split"], arith)
        assert st == lv.LV_OK
        assert T.tolist() == w["T_new"] and S.tolist() == w["share_new"]


@pytest.mark.parametrize("arith", [0, 1])
def test_whatif_config3_full(lv, ctx, arith):
    q = workloads.whatif_config()
    c = q.cand
    T, S, st = _run(lv, ctx, c.offsets, c.p, c.c, c.phase, q.p_new, q.c_new, q.phase_new, q.coef, q.split, arith)
    assert st == lv.LV_OK
    To, So = _check(c.offsets, c.p, c.c, c.phase, q.p_new, q.c_new, q.phase_new, q.coef, q.split, T, S)
    if arith == 1:
        assert np.array_equal(T, To) and np.array_equal(S, So)


def test_whatif_adversarial(lv, ctx):
    """Empty candidates, single requests, splits hit exactly, decode/prefill mixes, one pending row, ragged sizes."""
    rng = np.random.default_rng(4)
    sizes = np.array([0, 1, 2, 255, 256, 0, 3, 300, 1, 0] + list(rng.integers(0, 40, 190)))
    off = np.zeros(len(sizes) + 1, np.int64)
    np.cumsum(sizes, out=off[1:])
    n = int(off[-1])
    ph = (rng.random(n) < 0.3).astype(np.int32)
    p = np.where(ph == 1, rng.integers(1, 5000, n), 1).astype(np.int32)
    c = np.where(ph == 1, 0, rng.integers(0, 131072, n)).astype(np.int32)
    coef, _ = workloads.draw_coefficients(rng, "qwen2.5-32b")
    split = np.array([256, 300])
    for npd in (1, 33, 257):
        phn = (rng.random(npd) < 0.5).astype(np.int32)
        pn = np.where(phn == 1, rng.integers(1, 300, npd), 1).astype(np.int32)
        cn = np.where(phn == 1, 0, rng.integers(0, 100000, npd)).astype(np.int32)
        T, S, st = _run(lv, ctx, off, p, c, ph, pn, cn, phn, coef, split)
        assert st == lv.LV_OK
        _check(off, p, c, ph, pn, cn, phn, coef, split, T, S)


def test_whatif_deterministic_and_outputs_optional(lv, ctx):
    import torch
    q = workloads.whatif_config(scale=0.1, n_pending=100)
    c = q.cand
    a = _run(lv, ctx, c.offsets, c.p, c.c, c.phase, q.p_new, q.c_new, q.phase_new, q.coef, q.split)
    b = _run(lv, ctx, c.offsets, c.p, c.c, c.phase, q.p_new, q.c_new, q.phase_new, q.coef, q.split)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])
    cand = lv.batches_to_device(c.p, c.c, c.phase, c.offsets)
    t = lambda x: torch.as_tensor(x, device="cuda")  # noqa: E731
    S = torch.empty((q.n_pending, c.n_batch), dtype=torch.float64, device="cuda")
    lv.lv_whatif(ctx, lv.make_model(q.coef, q.split), cand, t(q.p_new), t(q.c_new), t(q.phase_new), None, S)
    assert np.array_equal(S.cpu().numpy(), a[1])


def _admit_inputs(q, n_tenants=8, seed=3):
    """Tenants of the pending requests, running totals, budgets and an SLO around
    the workload's own magnitudes, so that both outcomes occur often."""
    rng = np.random.default_rng(seed)
    To, So = oracle.whatif(q.cand.offsets, q.cand.p, q.cand.c, q.cand.phase, q.p_new, q.c_new, q.phase_new,
                           q.split, q.coef)
    u = rng.integers(0, n_tenants, q.n_pending).astype(np.int32)
    L = rng.uniform(0.0, 1.0, n_tenants) * float(np.median(So)) * 100
    B = L + rng.uniform(0.0, 2.0, n_tenants) * float(np.median(So))
    slo = float(np.median(To))
    return u, L, B, slo, To, So


@pytest.mark.parametrize("scale", [0.25, 1.0])
def test_whatif_admit_config3(lv, ctx, scale):
    """admit equals the oracle's predicate on the device's own T_new and shares
    bit for bit, and on the oracle's everywhere but at exact-margin ties; the
    admit-only call (no T_new, share_new) gives the same mask."""
    import torch
    q = workloads.whatif_config(scale=scale)
    c = q.cand
    u, L, B, slo, To, So = _admit_inputs(q)
    cand = lv.batches_to_device(c.p, c.c, c.phase, c.offsets)
    t = lambda a: torch.as_tensor(np.ascontiguousarray(a, dtype=np.int32), device="cuda")  # noqa: E731
    d = lambda a: torch.as_tensor(np.ascontiguousarray(a, dtype=np.float64), device="cuda")  # noqa: E731
    npd, nc = q.n_pending, c.n_batch
    T = torch.full((npd, nc), float("nan"), dtype=torch.float64, device="cuda")
    S = torch.full((npd, nc), float("nan"), dtype=torch.float64, device="cuda")
    A = torch.full((npd, nc), 7, dtype=torch.uint8, device="cuda")
    model = lv.make_model(q.coef, q.split)
    lv.lv_whatif_admit(ctx, model, cand, t(q.p_new), t(q.c_new), t(q.phase_new), t(u), d(L), d(B), slo, A, T, S)
    assert ctx.status() == lv.LV_OK
    T, S, A = T.cpu().numpy(), S.cpu().numpy(), A.cpu().numpy()
    _check(c.offsets, c.p, c.c, c.phase, q.p_new, q.c_new, q.phase_new, q.coef, q.split, T, S)
    assert np.array_equal(A, oracle.admit(T, S, u, L, B, slo))
    Ao = oracle.admit(To, So, u, L, B, slo)
    margin = np.minimum(np.abs(L[u][:, None] + So - B[u][:, None]) / B[u][:, None], np.abs(To - slo) / slo)
    assert np.all((A == Ao) | (margin <= 4 * TOL))
    assert 0.05 < A.mean() < 0.95
    A2 = torch.full((npd, nc), 7, dtype=torch.uint8, device="cuda")
    lv.lv_whatif_admit(ctx, model, cand, t(q.p_new), t(q.c_new), t(q.phase_new), t(u), d(L), d(B), slo, A2)
    assert np.array_equal(A2.cpu().numpy(), A)


def test_whatif_admit_invalid_tenant_and_arguments(lv, ctx):
    import torch
    q = workloads.whatif_config(scale=0.05)
    c = q.cand
    u, L, B, slo, _, _ = _admit_inputs(q)
    u[3] = 8  # out of range: data error, that request's pairs inadmissible
    cand = lv.batches_to_device(c.p, c.c, c.phase, c.offsets)
    t = lambda a: torch.as_tensor(np.ascontiguousarray(a, dtype=np.int32), device="cuda")  # noqa: E731
    d = lambda a: torch.as_tensor(np.ascontiguousarray(a, dtype=np.float64), device="cuda")  # noqa: E731
    A = torch.full((q.n_pending, c.n_batch), 7, dtype=torch.uint8, device="cuda")
    model = lv.make_model(q.coef, q.split)
    lv.lv_whatif_admit(ctx, model, cand, t(q.p_new), t(q.c_new), t(q.phase_new), t(u), d(L), d(B), slo, A)
    assert ctx.status() == lv.LV_EDATA
    A = A.cpu().numpy()
    assert np.all(A[3] == 0) and np.all(A <= 1)
    with pytest.raises(lv.LVError) as ei:
        lv.lv_whatif_admit(ctx, model, cand, t(q.p_new), t(q.c_new), t(q.phase_new), t(u), d(L), d(B), slo, None)
    assert ei.value.status == lv.LV_EINVAL
