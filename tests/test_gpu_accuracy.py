"""GPU parity of the token-count baseline fit (lv_fit_vtc) and of the accuracy
metrics (lv_accuracy) against the oracle.

The VTC line is held to the fit's bar, 1e-9 relative on each coefficient
(the oracle solves exactly and rounds once).  Accuracy: the sample count and
the three percentiles are exact (each is one of the relative errors, computed
by the same correctly rounded subtraction and division on both sides; on
the GPU's exact path that division is done in integers); R^2 and the mean
relative error within 1e-12 (exact integer or fixed-order fp64 sums against
the oracle's correctly rounded fp64 ones).  Inputs cover both of the
library's paths: values on one 79-bit grid (the exact integer path) and
magnitudes too far apart, non-finite or extreme ones (the fp64 path).
"""

import numpy as np
import pytest

import oracle
import workloads

pytestmark = pytest.mark.gpu


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


def _dev(a):
    import torch
    return torch.as_tensor(np.ascontiguousarray(a, dtype=np.float64), device="cuda")


@pytest.mark.parametrize("scale", [0.01, 0.1])
def test_vtc_fit_matches_oracle(lv, ctx, scale):
    w = workloads.config(2, scale=scale)
    T, _ = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
    Y = np.stack([T * w.noise, T])
    b = lv.batches_to_device(w.p, w.c, w.phase, w.offsets)
    res = lv.lv_fit_vtc(ctx, b, _dev(Y))
    feat, _ = oracle.batch_features(w.offsets, w.p, w.c, w.phase, w.split)
    for k in range(2):
        beta, a, st, m = oracle.vtc_fit(feat[0], feat[3], Y[k])
        gb, ga, gst, gm = res[k]
        assert (gst, gm) == (st, m)
        assert abs(gb - beta) <= 1e-9 * abs(beta) and abs(ga - a) <= 1e-9 * abs(a)


def test_vtc_fit_degenerate(lv, ctx):
    # every batch with the same S1: singular; one batch: no data
    off = np.array([0, 2, 4, 6], np.int64)
    p = np.array([3, 4, 2, 5, 6, 1], np.int32)
    c = np.arange(6, dtype=np.int32)
    ph = np.ones(6, np.int32)
    b = lv.batches_to_device(p, c, ph, off)
    assert lv.lv_fit_vtc(ctx, b, _dev(np.array([[1.0, 2.0, 3.0]])))[0][2] == lv.LV_ESINGULAR
    b1 = lv.batches_to_device(p[:2], c[:2], ph[:2], off[:2])
    assert lv.lv_fit_vtc(ctx, b1, _dev(np.array([[1.0]])))[0][2] == lv.LV_ENODATA


def _check_accuracy(g, o):
    assert g["n"] == o["n"]
    for key in ("p50", "p90", "p99"):
        assert g[key] == o[key], key
    for key in ("r2_ssr", "r2_corr", "mean_rel"):
        if np.isnan(o[key]):
            assert np.isnan(g[key])
        else:
            assert abs(g[key] - o[key]) <= 1e-12 * max(1.0, abs(o[key])), key


def test_accuracy_models_vs_vtc_config2(lv, ctx):
    """The paper's comparison on synthetic profiles: the fitted piecewise model
    and the token-count line, each against the noisy latencies."""
    import torch
    w = workloads.config(2, scale=0.05)
    T, _ = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
    y = T * w.noise
    b = lv.batches_to_device(w.p, w.c, w.phase, w.offsets)
    models = [lv.make_model(np.zeros((4, 5)), w.split)]
    lv.lv_fit(ctx, b, _dev(y[None]), models)
    Tm = torch.empty(w.n_batch, dtype=torch.float64, device="cuda")
    lv.lv_attribute(ctx, models[0], b, Tm, None, None)
    beta, a, st, _ = lv.lv_fit_vtc(ctx, b, _dev(y[None]))[0]
    assert st == lv.LV_OK
    vtc = lv.make_model(np.tile([beta, a, 0.0, 0.0, 0.0], (4, 1)), w.split)
    Tv = torch.empty(w.n_batch, dtype=torch.float64, device="cuda")
    lv.lv_attribute(ctx, vtc, b, Tv, None, None)
    yd = _dev(y)
    gm, gv = lv.lv_accuracy(ctx, yd, Tm), lv.lv_accuracy(ctx, yd, Tv)
    _check_accuracy(gm, oracle.accuracy(y, Tm.cpu().numpy()))
    _check_accuracy(gv, oracle.accuracy(y, Tv.cpu().numpy()))
    assert gm["r2_ssr"] > gv["r2_ssr"] and gm["p90"] < gv["p90"]  # the roofline form fits better
    assert lv.lv_accuracy(ctx, yd, Tm) == gm  # fixed-order sums: bit-identical repeats


def test_accuracy_edge_cases(lv, ctx):
    rng = np.random.default_rng(9)
    for n in (1, 2, 3, 257, 100_003):
        y = rng.uniform(0.5, 2.0, n)
        y[rng.random(n) < 0.1] = 0.0  # not samples
        T = y * (1 + rng.normal(0, 0.1, n))
        _check_accuracy(lv.lv_accuracy(ctx, _dev(y), _dev(T)), oracle.accuracy(y, T))
    # ties everywhere: many equal relative errors
    y = np.ones(1000)
    T = 1.0 + np.repeat(np.arange(10) / 16.0, 100)
    _check_accuracy(lv.lv_accuracy(ctx, _dev(y), _dev(T)), oracle.accuracy(y, T))
    # no sample at all
    g = lv.lv_accuracy(ctx, _dev(np.zeros(5)), _dev(np.ones(5)))
    assert g["n"] == 0 and np.isnan(g["p50"]) and np.isnan(g["r2_ssr"])


def test_accuracy_division_single_samples(lv, ctx):
    """n = 1: every percentile and the mean are the one relative error, so each
    call checks one correctly rounded fl(fl(T - y) / y) bit for bit, over
    differences that need rounding (exponents up to 26 apart), tiny ones (T
    within a few ulps of y), negative and zero T, and power-of-two y."""
    rng = np.random.default_rng(21)
    cases = []
    for k in range(400):
        y = float(rng.uniform(0.5, 2.0)) * 2.0 ** int(rng.integers(-12, 12))
        kind = k % 8
        if kind == 0:
            T = y * (1 + rng.normal(0, 0.1))
        elif kind == 1:
            T = y + float(rng.integers(-6, 7)) * np.spacing(y)
        elif kind == 2:
            T = -y * float(rng.uniform(0, 3))
        elif kind == 3:
            T = float(rng.uniform(0.5, 2.0)) * 2.0 ** int(rng.integers(-14, 14))
        elif kind == 4:
            T = 0.0
        elif kind == 5:
            y = 2.0 ** int(rng.integers(-20, 20))
            T = y * float(rng.uniform(0, 4))
        elif kind == 6:
            T = y * (1 + float(rng.integers(1, 2 ** 20)) * 2.0 ** -52)
        else:
            T = y * 2.0 ** 25 * float(rng.uniform(1, 2))  # far apart: the difference is rounded
        cases.append((y, T))
    for y, T in cases:
        g = lv.lv_accuracy(ctx, _dev([y]), _dev([T]))
        o = oracle.accuracy(np.array([y]), np.array([T]))
        assert g["n"] == 1
        assert g["p50"] == o["p50"] and g["p99"] == o["p99"], (y, T)
        assert g["mean_rel"] == o["mean_rel"], (y, T)


_PATH_CASES = ["integers", "negative_T", "wide_range", "large", "huge", "tiny", "nonfinite_T", "few_values",
               "zero_T"]


@pytest.mark.parametrize("case", _PATH_CASES)
def test_accuracy_paths(lv, ctx, case):
    """Both paths against the oracle: values on one grid (integers with zero
    low bits, negative or zero predictions, magnitudes near 1e60 or 1e-40) take
    the exact integer path; magnitudes 2^60 apart, non-finite predictions and
    values near 1e100 take the fp64 path."""
    rng = np.random.default_rng(100 + _PATH_CASES.index(case))
    n = 200_003
    y = rng.uniform(0.5, 2.0, n) * 1e-3
    T = y * (1 + rng.normal(0, 0.2, n))
    if case == "integers":
        y = rng.integers(1, 2 ** 40, n).astype(np.float64)
        T = np.round(y * (1 + rng.normal(0, 0.1, n)))
    elif case == "negative_T":
        T = -T
    elif case == "wide_range":
        y = y * 2.0 ** rng.integers(-30, 30, n)
        T = y * (1 + rng.normal(0, 0.2, n))
    elif case == "large":
        y, T = y * 1e63, T * 1e63
    elif case == "huge":
        y, T = y * 1e63, T * 1e63
        y[:10], T[:10] = y[:10] * 1e40, T[:10] * 1e40
    elif case == "tiny":
        y, T = y * 1e-37, T * 1e-37
    elif case == "nonfinite_T":
        T[5] = np.inf
    elif case == "few_values":
        y = np.ones(n)
        T = 1.0 + rng.integers(0, 7, n) / 8.0
    elif case == "zero_T":
        T[rng.random(n) < 0.3] = 0.0
    y[rng.random(n) < 0.05] = 0.0
    if case == "nonfinite_T":
        y[5] = 1e-3  # a sample whose prediction is infinite
    g = lv.lv_accuracy(ctx, _dev(y), _dev(T))
    if case == "nonfinite_T":
        # the oracle's correctly rounded sums reject inf - inf; the order
        # statistics below the top are those of the same data with the
        # infinite prediction replaced by one larger than every other
        Tf = T.copy()
        Tf[5] = 1e300
        o = oracle.accuracy(y, Tf)
        assert g["n"] == o["n"] and g["p50"] == o["p50"] and g["p90"] == o["p90"]
        assert np.isinf(g["mean_rel"])
        return
    o = oracle.accuracy(y, T)
    _check_accuracy(g, o)
    again = lv.lv_accuracy(ctx, _dev(y), _dev(T))  # repeats bit for bit (NaN where NaN)
    assert all(again[k] == g[k] or (np.isnan(again[k]) and np.isnan(g[k])) for k in g)


@pytest.mark.parametrize("n", [4_000, 30_000, 200_000])
def test_accuracy_select_list_sizes(lv, ctx, n):
    """Relative errors in two clusters: 70% in [0.5, 0.5 + 2^-14), the rest in
    [0.52, 0.53).  Every sample shares the sign, exponent and top mantissa
    bits, so the first select digit puts the first cluster into four bins of
    about n / 6 each, and p50 (inside the first cluster) is settled from a
    candidate list that is short (n = 4k, ranked directly), mid-sized (30k,
    held in shared memory) or long (200k, read from global memory)."""
    rng = np.random.default_rng(n)
    y = rng.uniform(0.5, 2.0, n)
    first = rng.random(n) < 0.7
    rel = np.where(first, 0.5 + rng.uniform(0.0, 2.0 ** -14, n), rng.uniform(0.52, 0.53, n))
    T = y * (1.0 + rel)
    _check_accuracy(lv.lv_accuracy(ctx, _dev(y), _dev(T)), oracle.accuracy(y, T))


def test_accuracy_large_block_ranges(lv, ctx):
    """3.2 million batches: each block's share of the exact pass is then more
    than its shared-memory stage holds, so its relative errors go through
    device memory on their way to the block's first-digit sort."""
    rng = np.random.default_rng(77)
    n = 3_200_000
    T = rng.lognormal(-3.0, 0.6, n)
    y = T * rng.lognormal(0.0, 0.1, n)
    y[rng.random(n) < 0.02] = 0.0
    _check_accuracy(lv.lv_accuracy(ctx, _dev(y), _dev(T)), oracle.accuracy(y, T))


def test_barrier_wait_is_bounded(lv, ctx):
    """Failure detection without a fault: the accuracy kernel's grid barrier,
    run with one block that never arrives, gives up after a few seconds and
    reports LV_ETIMEOUT; the context stays usable."""
    import time
    t = time.perf_counter()
    assert ctx.selftest_barrier() == lv.LV_ETIMEOUT
    assert time.perf_counter() - t < 30.0
    y = np.array([1.0, 2.0, 4.0])
    T = np.array([1.5, 2.0, 3.0])
    _check_accuracy(lv.lv_accuracy(ctx, _dev(y), _dev(T)), oracle.accuracy(y, T))
