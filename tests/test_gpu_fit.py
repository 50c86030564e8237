"""GPU parity of lv_fit against the oracle's exact rational least squares.

The oracle solves each group's normal equations exactly and rounds once; the
device accumulates X^T X and X^T y exactly and solves in double-double, so for
the conditioning of these workloads the coefficients agree to a few units in
the last place.  The bar is the stated one, 1e-9 relative on fitted
predictions, also applied to every coefficient the oracle reports as non-zero.
Group sizes,
statuses and dropped columns are integers and must match exactly; SSR is
compared relative to y'y (the scale its cancellation works at) and r2 in
absolute terms.
"""

import numpy as np
import pytest

import oracle
import workloads

pytestmark = pytest.mark.gpu
COEF_TOL = 1e-9  # the stated bar for fitted predictions; coefficients are held to the same


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


def _gpu_fit(lv, ctx, off, p, c, ph, Y, split):
    import torch
    b = lv.batches_to_device(p, c, ph, off)
    Y = np.atleast_2d(np.asarray(Y, dtype=np.float64))
    yd = torch.as_tensor(np.ascontiguousarray(Y), device="cuda")
    models = [lv.make_model(np.full((4, 5), np.nan), split) for _ in range(Y.shape[0])]
    reps = lv.lv_fit(ctx, b, yd, models)
    return [lv.model_coef(m) for m in models], reps


def _compare(off, p, c, ph, Y, split, coefs, reps):
    feat, seg = oracle.batch_features(off, p, c, ph, split)
    for k, y in enumerate(np.atleast_2d(Y)):
        res = oracle.fit(feat, seg, y)
        for g in range(4):
            o, r = res[g], reps[k]
            assert r["n"][g] == o["n"]
            assert r["status"][g] == o["status"], (k, g)
            assert r["dropped"][g] == o["dropped"]
            if o["status"] != oracle.OK:
                assert np.all(np.isnan(coefs[k][g])), "coefficients of a failed group must stay untouched"
                continue
            cg, co = coefs[k][g], o["coef"]
            nz = co != 0
            assert np.all(cg[~nz] == 0)
            assert np.max(np.abs(cg[nz] - co[nz]) / np.abs(co[nz])) <= COEF_TOL, (k, g, cg, co)
            sel = (seg == g) & (feat[3] > 0)
            X = np.stack([np.ones(int(sel.sum())), feat[0, sel], feat[1, sel], feat[2, sel], feat[4, sel]], axis=1)
            pg, po = X @ cg, X @ co
            assert np.max(np.abs(pg - po) / np.abs(po)) <= COEF_TOL
            yy = float(np.dot(y[sel], y[sel]))
            assert abs(r["ssr"][g] - o["ssr"]) <= 1e-13 * yy
            if np.isnan(o["r2"]):
                assert np.isnan(r["r2"][g])
            else:
                assert abs(r["r2"][g] - o["r2"]) <= 1e-9
    return feat, seg


def _latencies(w):
    T, _ = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
    return T


def test_fit_noiseless_recovers_generating_coefficients(lv, ctx):
    w = workloads.config(2, scale=0.01)
    T = _latencies(w)
    coefs, reps = _gpu_fit(lv, ctx, w.offsets, w.p, w.c, w.phase, T, w.split)
    _compare(w.offsets, w.p, w.c, w.phase, T, w.split, coefs, reps)
    fitted = [g for g in range(4) if reps[0]["status"][g] == 0]
    assert len(fitted) >= 3  # decode batches never reach the compute regime at this split
    for g in fitted:
        truth = w.coef[g].copy()
        if reps[0]["dropped"][g] & 8:  # decode groups: a1 carries a1 + a3
            truth[1] += truth[3]
            truth[3] = 0.0
        nz = truth != 0
        assert np.max(np.abs(coefs[0][g][nz] - truth[nz]) / np.abs(truth[nz])) <= 1e-6


def test_fit_noisy_and_noiseless_in_one_pass(lv, ctx):
    w = workloads.config(2, scale=0.02)
    T = _latencies(w)
    Y = np.stack([T * w.noise, T, T * w.noise[::-1]])
    coefs, reps = _gpu_fit(lv, ctx, w.offsets, w.p, w.c, w.phase, Y, w.split)
    _compare(w.offsets, w.p, w.c, w.phase, Y, w.split, coefs, reps)
    assert all(0.9 < reps[0]["r2"][g] < 1.0 for g in range(4) if reps[0]["status"][g] == 0)


def test_fit_full_size_config2(lv, ctx):
    """2,000,000 profiled batches, noisy latencies: the workload the fit is sized for."""
    w = workloads.config(2)
    T = _latencies(w) * w.noise
    coefs, reps = _gpu_fit(lv, ctx, w.offsets, w.p, w.c, w.phase, T, w.split)
    _compare(w.offsets, w.p, w.c, w.phase, T, w.split, coefs, reps)
    assert sum(reps[0]["n"]) == w.n_batch


def test_fit_ragged_and_jumbo_batches(lv, ctx):
    """Empty batches, single requests, batches beyond one tile, splits hit exactly."""
    rng = np.random.default_rng(11)
    sizes = np.array([0, 1, 2, 1500, 0, 4096, 3, 1281, 1280, 1] + list(rng.integers(0, 300, 3000)))
    off = np.zeros(len(sizes) + 1, np.int64)
    np.cumsum(sizes, out=off[1:])
    n = int(off[-1])
    ph = (rng.random(n) < 0.05).astype(np.int32)
    p = np.where(ph == 1, rng.integers(1, 3000, n), 1).astype(np.int32)
    c = rng.integers(0, 100000, n).astype(np.int32)
    coef, _ = workloads.draw_coefficients(rng, "llama3.1-8b")
    split = np.array([128, 3000])
    T, _ = oracle.attribute(off, p, c, ph, split, coef)
    y = T * np.exp(0.05 * rng.standard_normal(len(sizes)))
    coefs, reps = _gpu_fit(lv, ctx, off, p, c, ph, y, split)
    _compare(off, p, c, ph, y, split, coefs, reps)


def test_fit_degenerate_groups(lv, ctx):
    """No batches at all; too few batches for a group; exactly singular groups."""
    # no batches: every group ENODATA with n = 0
    off = np.zeros(1, np.int64)
    e = np.zeros(0, np.int32)
    coefs, reps = _gpu_fit(lv, ctx, off, e, e, e, np.zeros(0), (4, 4))
    assert reps[0]["status"] == [oracle.ENODATA] * 4 and reps[0]["n"] == [0] * 4
    # decode batches of size 1 only (1 == S1 == n^2: singular) and three prefill batches (ENODATA)
    rng = np.random.default_rng(5)
    sizes = np.array([1] * 50 + [3, 4, 5])
    off = np.zeros(len(sizes) + 1, np.int64)
    np.cumsum(sizes, out=off[1:])
    n = int(off[-1])
    ph = np.zeros(n, np.int32)
    ph[off[50:53]] = 1
    p = np.where(ph == 1, 7, 1).astype(np.int32)
    c = rng.integers(0, 1000, n).astype(np.int32)
    y = rng.random(len(sizes)) + 0.5
    coefs, reps = _gpu_fit(lv, ctx, off, p, c, ph, y, (1 << 30, 1 << 30))
    _compare(off, p, c, ph, y, (1 << 30, 1 << 30), coefs, reps)
    assert reps[0]["status"][0] == oracle.ESINGULAR and reps[0]["status"][2] == oracle.ENODATA


def test_fit_deterministic(lv, ctx):
    w = workloads.config(2, scale=0.05)
    T = _latencies(w) * w.noise
    a = _gpu_fit(lv, ctx, w.offsets, w.p, w.c, w.phase, T, w.split)
    b = _gpu_fit(lv, ctx, w.offsets, w.p, w.c, w.phase, T, w.split)
    # bit-identical, NaN (untouched empty groups) included
    assert all(np.array_equal(x.view(np.int64), y.view(np.int64)) for x, y in zip(a[0], b[0]))
    assert repr(a[1]) == repr(b[1])


def test_fit_errors(lv, ctx):
    import torch
    w = workloads.config(0, scale=0.01)
    T = _latencies(w)
    b = lv.batches_to_device(w.p, w.c, w.phase, w.offsets)
    m = lambda sp: lv.make_model(np.zeros((4, 5)), sp)  # noqa: E731
    # non-finite latency: data error, models untouched
    bad = T.copy()
    bad[7] = np.nan
    models = [m(w.split)]
    with pytest.raises(lv.LVError) as ei:
        lv.lv_fit(ctx, b, torch.as_tensor(bad, device="cuda")[None], models)
    assert ei.value.status == lv.LV_EDATA
    assert np.all(lv.model_coef(models[0]) == 0)
    # splits must agree across the fitted models; at most four y vectors
    y2 = torch.as_tensor(np.stack([T, T]), device="cuda")
    with pytest.raises(lv.LVError) as ei:
        lv.lv_fit(ctx, b, y2, [m(w.split), m((w.split[0] + 1, w.split[1]))])
    assert ei.value.status == lv.LV_EINVAL
    y5 = torch.as_tensor(np.stack([T] * 5), device="cuda")
    with pytest.raises(lv.LVError) as ei:
        lv.lv_fit(ctx, b, y5, [m(w.split) for _ in range(5)])
    assert ei.value.status == lv.LV_EINVAL
    # batch sums beyond 2^48 (p^2 of a 2^30-token prefill): overflow, not a wrong fit
    off = np.array([0, 2], np.int64)
    big = lv.batches_to_device(np.array([1 << 30, 1], np.int32), np.array([0, 0], np.int32),
                               np.array([1, 0], np.int32), off)
    with pytest.raises(lv.LVError) as ei:
        lv.lv_fit(ctx, big, torch.ones((1, 1), dtype=torch.float64, device="cuda"), [m((1, 1))])
    assert ei.value.status == lv.LV_EOVERFLOW
    assert ctx.status() == lv.LV_OK  # the sticky status was consumed by lv_fit
