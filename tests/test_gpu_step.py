"""Single-step scheduler mode: one serving batch of 2048 requests through a CUDA
graph of lv_tenant_acc_reset + lv_attribute + lv_tenant_totals, or of the one
call lv_attribute_step, captured once and replayed.

Every replay must give the eager call's T, shares and tenant totals bit for
bit, and those the oracle's within the attribution tolerance (1e-12 relative).
Inputs of at most 4,096 requests in at most 16 batches take a one-cluster
kernel; its cases are checked against the oracle and against the general
kernels here as well.
"""

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


def _bits(t):
    return t.cpu().numpy().view(np.int64)


@pytest.mark.parametrize("n_req,n_prefill", [(2048, 4), (128, 0), (1, 1)])
def test_graph_replay_matches_eager_and_oracle(lv, n_req, n_prefill):
    import torch
    w = workloads.step_config(n_req=n_req, n_prefill=n_prefill)
    ctx = lv.Context()
    b = lv.batches_to_device(w.p, w.c, w.phase, w.offsets, w.tenant, w.n_tenants)
    model = lv.make_model(w.coef, w.split)
    acc = lv.TenantAcc(ctx, w.n_tenants)

    def bufs():
        nan = float("nan")
        return (torch.full((w.n_batch,), nan, dtype=torch.float64, device="cuda"),
                torch.full((w.n_req,), nan, dtype=torch.float64, device="cuda"),
                torch.full((w.n_tenants,), nan, dtype=torch.float64, device="cuda"))

    def run(st, T, S, L):
        acc.reset(stream=st)
        lv.lv_attribute(ctx, model, b, T, S, acc, stream=st)
        lv.lv_tenant_totals(ctx, acc, L, stream=st)

    T0, S0, L0 = bufs()
    run(torch.cuda.current_stream(), T0, S0, L0)
    torch.cuda.synchronize()

    T1, S1, L1 = bufs()
    cs = torch.cuda.Stream()
    cs.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(cs):
        for _ in range(2):
            run(cs, T1, S1, L1)
    torch.cuda.synchronize()
    for t in (T1, S1, L1):
        t.fill_(float("nan"))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=cs):
        run(cs, T1, S1, L1)
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    assert ctx.status() == lv.LV_OK
    for a, e in ((T1, T0), (S1, S0), (L1, L0)):
        assert np.array_equal(_bits(a), _bits(e))

    T_o, s_o = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
    T, S, L = T1.cpu().numpy(), S1.cpu().numpy(), L1.cpu().numpy()
    assert np.max(np.abs(T - T_o) / np.abs(T_o)) <= TOL
    assert np.max(np.abs(S - s_o) / np.abs(s_o)) <= TOL
    L_o = oracle.tenant_totals(s_o, w.tenant, w.n_tenants)
    m = L_o != 0
    assert np.all(L[~m] == 0)
    assert np.max(np.abs(L[m] - L_o[m]) / np.abs(L_o[m])) <= TOL


@pytest.mark.parametrize("sizes,nt,arith", [
    ([300, 0, 17, 2048, 1, 0, 900, 5], 256, 0),          # several batches, two empty
    ([2048, 2048], 3000, 0),                             # 4096 requests (the limit), tenants beyond the shared table
    ([7, 64, 1000, 3, 3, 3, 3, 3, 3, 3, 3, 3, 3, 3, 3, 3], 40, 1),  # 16 batches, the fp64 arithmetic mode
])
def test_small_inputs_against_oracle(lv, sizes, nt, arith):
    """lv_attribute on a serving step's worth of requests (at most 4,096 in at most 16 batches)
    runs the one-cluster kernel: T, shares and tenant totals against the oracle over two calls
    into one accumulator, each total equal to the exact sum of the returned shares."""
    import torch
    from fractions import Fraction
    rng = np.random.default_rng(sum(sizes) + nt)
    off = np.zeros(len(sizes) + 1, np.int64)
    np.cumsum(sizes, out=off[1:])
    n = int(off[-1])
    ph = (rng.random(n) < 0.05).astype(np.int32)
    p = np.where(ph == 1, rng.integers(1, 2000, n), 1).astype(np.int32)
    c = np.where(ph == 1, 0, rng.integers(1, 32768, n)).astype(np.int32)
    t = rng.integers(0, nt, n).astype(np.int32)
    coef, _ = workloads.draw_coefficients(np.random.default_rng(3), "qwen2.5-14b")
    split = np.array([256, 256], np.int64)
    ctx = lv.Context()
    ctx.set_arith(arith)
    b = lv.batches_to_device(p, c, ph, off, t, nt)
    model = lv.make_model(coef, split)
    acc = lv.TenantAcc(ctx, nt)
    T = torch.full((len(sizes),), float("nan"), dtype=torch.float64, device="cuda")
    S = torch.full((n,), float("nan"), dtype=torch.float64, device="cuda")
    for _ in range(2):
        lv.lv_attribute(ctx, model, b, T, S, acc)
    L = torch.empty(nt, dtype=torch.float64, device="cuda")
    lv.lv_tenant_totals(ctx, acc, L)
    assert ctx.status() == lv.LV_OK
    T_o, s_o = oracle.attribute(off, p, c, ph, split, coef)
    Tg, Sg, Lg = T.cpu().numpy(), S.cpu().numpy(), L.cpu().numpy()
    assert np.all(Tg[T_o == 0] == 0)
    assert np.max(np.abs(Tg[T_o != 0] - T_o[T_o != 0]) / np.abs(T_o[T_o != 0])) <= TOL
    assert np.max(np.abs(Sg - s_o) / np.abs(s_o)) <= TOL
    if arith == 1:
        assert np.array_equal(Tg, T_o) and np.array_equal(Sg, s_o)
    L_o = oracle.TenantSums(nt).add(s_o, t).add(s_o, t).totals()
    m = L_o != 0
    assert np.all(Lg[~m] == 0)
    assert np.max(np.abs(Lg[m] - L_o[m]) / np.abs(L_o[m])) <= TOL
    for u in list(np.unique(t)[:20]) + [int(t.max())]:
        tot = 2 * sum(round(Fraction(v) * 2**72) for v in Sg[t == u].tolist())
        assert Lg[u] == float(Fraction(tot, 2**72))


def test_small_input_data_error(lv):
    """A negative token count in a small input records LV_EDATA (clamped, no fault)."""
    import torch
    w = workloads.step_config(n_req=512, n_prefill=2)
    w.p[17] = -3
    ctx = lv.Context()
    b = lv.batches_to_device(w.p, w.c, w.phase, w.offsets, w.tenant, w.n_tenants)
    S = torch.empty(w.n_req, dtype=torch.float64, device="cuda")
    lv.lv_attribute(ctx, lv.make_model(w.coef, w.split), b, None, S, None)
    assert ctx.status() == lv.LV_EDATA
    assert ctx.status() == lv.LV_OK


def _step_case(kind):
    """Offsets, fields, tenants, tenant count and arithmetic mode of one lv_attribute_step case."""
    rng = np.random.default_rng({"serving": 1, "ragged": 2, "max": 3, "over": 4, "many": 5, "wide": 6, "one": 7,
                                 "decode": 8, "bad_offsets": 9, "bad_tenant": 10}[kind])
    if kind == "serving":
        w = workloads.step_config(n_req=2048, n_prefill=4)
        return w.offsets, w.p, w.c, w.phase, w.tenant, w.n_tenants, 0
    sizes, nt, arith = {"ragged": ([1, 2046], 512, 0), "max": ([4096], 300, 0), "over": ([4097], 256, 0),
                        "many": ([300, 0, 17, 900, 1, 0, 40, 5, 3, 3, 3, 3, 3, 3, 3, 600], 40, 1),
                        "wide": ([1500, 1500], 513, 0), "one": ([1], 1, 0), "decode": ([2048], 1, 0),
                        "bad_offsets": ([100, 200, 300], 64, 0), "bad_tenant": ([700], 64, 0)}[kind]
    off = np.zeros(len(sizes) + 1, np.int64)
    np.cumsum(sizes, out=off[1:])
    n = int(off[-1])
    ph = (rng.random(n) < (0 if kind == "decode" else 0.05)).astype(np.int32)
    p = np.where(ph == 1, rng.integers(1, 2000, n), 1).astype(np.int32)
    c = np.where(ph == 1, rng.integers(0, 30000, n), rng.integers(1, 32768, n)).astype(np.int32)
    t = rng.integers(0, nt, n).astype(np.int32)
    if kind == "bad_offsets":
        off[2] = 50  # below off[1]: clamped to a non-decreasing sequence, LV_EDATA
    if kind == "bad_tenant":
        t[123] = nt + 5
    return off, p, c, ph, t, nt, arith


STEP_CASES = ["serving", "ragged", "max", "over", "many", "wide", "one", "decode"]


@pytest.mark.parametrize("kind", STEP_CASES + ["bad_offsets", "bad_tenant"])
def test_attribute_step_matches_separate_calls(lv, kind):
    """lv_attribute_step (one launch for a serving step of at most 4,096 requests, 16 batches and 512
    tenants; the separate calls' kernels otherwise) gives lv_tenant_acc_reset + lv_attribute +
    lv_tenant_totals bit for bit, on a reset step and on a second step that accumulates; T and
    shares equal the general kernels' (the same batches inside an input too large for the step
    path) and the oracle's within 1e-12."""
    import torch
    off, p, c, ph, t, nt, arith = _step_case(kind)
    bad = kind.startswith("bad")
    coef, _ = workloads.draw_coefficients(np.random.default_rng(11), "qwen2.5-14b")
    split = np.array([256, 256], np.int64)
    nb, n = len(off) - 1, int(off[-1])
    ctx = lv.Context()
    ctx.set_arith(arith)
    b = lv.batches_to_device(p, c, ph, off, t, nt)
    model = lv.make_model(coef, split)
    acc_a, acc_b = lv.TenantAcc(ctx, nt), lv.TenantAcc(ctx, nt)

    def bufs():
        nan = float("nan")
        return (torch.full((nb,), nan, dtype=torch.float64, device="cuda"),
                torch.full((n,), nan, dtype=torch.float64, device="cuda"),
                torch.full((nt,), nan, dtype=torch.float64, device="cuda"))

    for reset in (True, False):
        Ta, Sa, La = bufs()
        Tb, Sb, Lb = bufs()
        if reset:
            acc_a.reset()
        lv.lv_attribute(ctx, model, b, Ta, Sa, acc_a)
        lv.lv_tenant_totals(ctx, acc_a, La)
        sa = ctx.status()
        lv.lv_attribute_step(ctx, model, b, Tb, Sb, acc_b, Lb, reset=reset)
        sb = ctx.status()
        assert sa == sb == (lv.LV_EDATA if bad else lv.LV_OK)
        for x, y in ((Ta, Tb), (Sa, Sb), (La, Lb)):
            assert np.array_equal(_bits(x), _bits(y))
        assert acc_a.export() == acc_b.export()
    if bad:
        return

    # the general kernels: the same batches followed by a filler batch that takes the input past 4,096 requests
    fill = 4097
    off_g = np.concatenate([off, [n + fill]]).astype(np.int64)
    p_g = np.concatenate([p, np.ones(fill, np.int32)])
    c_g = np.concatenate([c, np.full(fill, 100, np.int32)])
    ph_g = np.concatenate([ph, np.zeros(fill, np.int32)])
    bg = lv.batches_to_device(p_g, c_g, ph_g, off_g)
    Tg = torch.empty(nb + 1, dtype=torch.float64, device="cuda")
    Sg = torch.empty(n + fill, dtype=torch.float64, device="cuda")
    lv.lv_attribute(ctx, model, bg, Tg, Sg, None)
    assert ctx.status() == lv.LV_OK
    assert np.array_equal(_bits(Tg)[:nb], _bits(Tb)) and np.array_equal(_bits(Sg)[:n], _bits(Sb))

    T_o, s_o = oracle.attribute(off, p, c, ph, split, coef)
    T, S, L = Tb.cpu().numpy(), Sb.cpu().numpy(), Lb.cpu().numpy()
    assert np.all(T[T_o == 0] == 0)
    if np.any(T_o != 0):
        assert np.max(np.abs(T[T_o != 0] - T_o[T_o != 0]) / np.abs(T_o[T_o != 0])) <= TOL
    assert np.max(np.abs(S - s_o) / np.abs(s_o)) <= TOL
    L_o = oracle.TenantSums(nt).add(s_o, t).add(s_o, t).totals()
    m = L_o != 0
    assert np.all(L[~m] == 0)
    assert np.max(np.abs(L[m] - L_o[m]) / np.abs(L_o[m])) <= TOL


@pytest.mark.parametrize("kind", ["serving", "wide"])
def test_attribute_step_graph_replay(lv, kind):
    """lv_attribute_step with a reset, captured into a CUDA graph (one kernel node for a serving
    step): every replay gives the eager call's T, shares and totals bit for bit."""
    import torch
    off, p, c, ph, t, nt, arith = _step_case(kind)
    coef, _ = workloads.draw_coefficients(np.random.default_rng(11), "qwen2.5-14b")
    model = lv.make_model(coef, np.array([256, 256], np.int64))
    ctx = lv.Context()
    b = lv.batches_to_device(p, c, ph, off, t, nt)
    acc = lv.TenantAcc(ctx, nt)
    nb, n = len(off) - 1, int(off[-1])
    out = [torch.full((k,), float("nan"), dtype=torch.float64, device="cuda") for k in (nb, n, nt)]
    ref = [torch.empty_like(x) for x in out]
    lv.lv_attribute_step(ctx, model, b, *ref[:2], acc, ref[2], reset=True)
    torch.cuda.synchronize()
    cs = torch.cuda.Stream()
    cs.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(cs):
        for _ in range(2):
            lv.lv_attribute_step(ctx, model, b, *out[:2], acc, out[2], reset=True, stream=cs)
    torch.cuda.synchronize()
    for x in out:
        x.fill_(float("nan"))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=cs):
        lv.lv_attribute_step(ctx, model, b, *out[:2], acc, out[2], reset=True, stream=cs)
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize()
    assert ctx.status() == lv.LV_OK
    for x, y in zip(out, ref):
        assert np.array_equal(_bits(x), _bits(y))
