"""Single-step scheduler mode: one serving batch of 2048 requests through a CUDA
graph of lv_tenant_acc_reset + lv_attribute + lv_tenant_totals, captured once
and replayed.

Every replay must give the eager call's T, shares and tenant totals bit for
bit, and those the oracle's within the attribution tolerance (1e-12 relative;
shares relative to max(|oracle share|, T_b / n)).
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
