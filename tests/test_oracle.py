"""Pins for the CPU oracle (no GPU).

Each test ties the oracle to something other than itself: hand-computed golden
values, brute-force counts, invariants stated by the paper (additivity of the
shares, tenant roll-up), special cases that reduce to a library routine
(math.fsum, numpy.linalg.lstsq) and exact rational arithmetic.
"""

import json
import math
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle
import workloads


def _load(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as f:
        return json.load(f)


# ---------------------------------------------------------------- architecture constants

def test_arch_constants_hand_values(golden_dir):
    g = _load(golden_dir, "arch_constants.json")
    for case in g["cases"]:
        phi, W = oracle.arch_constants(case["arch"])
        assert phi.tolist() == case["phi"], case["name"]
        assert W == case["W"], case["name"]


def test_arch_constants_brute_force_counts():
    """Count parameters, KV bytes and causal attention FLOPs from explicit shapes and loops."""
    rng = np.random.default_rng(5)
    for _ in range(20):
        tp = int(rng.choice([1, 2, 4]))
        L = int(rng.integers(1, 5))
        d = int(rng.integers(1, 9)) * 8
        hkv = tp * int(rng.integers(1, 3))
        hq = hkv * int(rng.integers(1, 4))
        hd = int(rng.integers(1, 5)) * 4
        F = tp * int(rng.integers(1, 20))
        wb, kvb = int(rng.integers(1, 5)), int(rng.integers(1, 5))
        arch = (L, d, hq, hkv, hd, F, wb, kvb, tp)
        shapes = [(d, hq * hd), (d, hkv * hd), (d, hkv * hd), (hq * hd, d), (d, F), (d, F), (F, d)]
        params = sum(a * b for a, b in shapes)
        phi, W = oracle.arch_constants(arch)
        # weights: every layer's matrices, bytes, split over tp ranks
        assert W * tp == L * params * wb
        # dense GEMM FLOPs per token: 2 per multiply-accumulate per weight
        assert phi[0] * tp == 2 * L * params
        # KV bytes per context token: K and V rows of every kv head of every layer
        kv = sum(hd * kvb for _layer in range(L) for _kv in ("K", "V") for _h in range(hkv))
        assert phi[1] * tp == kv
        # causal attention: count (query, key) pairs with key <= query, 4*hd FLOPs each (QK^T and PV)
        for p in (1, 2, 3, 7):
            pairs = sum(1 for q in range(p) for k in range(q + 1))
            flops = 4 * hd * hq * L * pairs
            # pairs = (p^2 + p)/2, so the count is phi3*tp*(p^2 + p): the feature phi3*p^2
            # is its quadratic part, the linear remainder belongs with the a1*p term.
            assert flops == phi[2] * tp * (p * p + p)


def test_arch_constants_rejects():
    with pytest.raises(ValueError):
        oracle.arch_constants((32, 4096, 32, 8, 128, 14336, 2, 2, 3))  # tp does not divide heads
    with pytest.raises(ValueError):
        oracle.arch_constants((32, 4096, 32, 8, 128, 14336, 0, 2, 1))
    with pytest.raises(ValueError):
        oracle.arch_constants((2**30, 2**30, 2**20, 2**20, 2**20, 2**30, 2, 2, 1))  # int64 overflow


def test_request_features_hand():
    phi = np.array([68, 8, 4])
    out = oracle.request_features([1, 3], [5, 0], phi)
    assert out.tolist() == [[68, 204], [40, 0], [4, 36]]


# ---------------------------------------------------------------- Eq. 1, shares, tenants (hand values)

def test_hand_cases(golden_dir):
    g = _load(golden_dir, "eq1_hand_cases.json")
    coef = np.array(g["coef"], dtype=np.float64)
    feat, seg = oracle.batch_features(g["offsets"], g["p"], g["c"], g["phase"], g["split"])
    assert feat.T.tolist() == g["batch_feat_S1_S2_S3_n_n2"]
    assert seg.tolist() == g["batch_seg"]
    T, share = oracle.attribute(g["offsets"], g["p"], g["c"], g["phase"], g["split"], coef)
    assert T.tolist() == g["T"]
    assert share.tolist() == g["share"]
    assert oracle.batch_latency(feat, seg, coef).tolist() == g["T"]
    L = oracle.tenant_totals(share, g["tenant"], g["n_tenants"])
    assert L.tolist() == g["tenant_totals"]
    w = g["whatif"]
    Tn, Sn = oracle.whatif(w["cand_offsets"], w["cand_p"], w["cand_c"], w["cand_phase"], w["p_new"], w["c_new"],
                           w["phase_new"], g["split"], coef)
    assert Tn.tolist() == w["T_new"]
    assert Sn.tolist() == w["share_new"]


def _exact_T(k, S1, S2, S3, n):
    if n == 0:
        return Fraction(0)
    f = [Fraction(float(v)) for v in k]
    return f[0] + f[1] * S1 + f[2] * S2 + f[3] * S3 + f[4] * n * n


def _small_random(seed, n_batch=300, hi=40):
    rng = np.random.default_rng(seed)
    p, c, ph, t, off = workloads.random_batches(
        rng, n_batch, 0, hi, 0.3, lambda r, n: r.integers(1, 3000, size=n).astype(np.int32),
        lambda r, n: r.integers(0, 70000, size=n).astype(np.int32), n_tenants=7)
    coef, split = workloads.draw_coefficients(rng, "llama3.1-8b", split=(20, 900))
    return p, c, ph, t, off, coef, split


def test_eq1_and_shares_within_rounding_of_exact():
    """Oracle T and shares are within a few ulp of the exact rational values."""
    p, c, ph, t, off, coef, split = _small_random(1)
    T, share = oracle.attribute(off, p, c, ph, split, coef)
    for b in range(len(off) - 1):
        lo, hi = off[b], off[b + 1]
        n = int(hi - lo)
        pb = [int(v) for v in p[lo:hi]]
        cb = [int(v) for v in c[lo:hi]]
        S1, S2, S3 = sum(pb), sum(cb), sum(v * v for v in pb)
        pre = int(any(ph[lo:hi] == 1))
        seg = pre * 2 + (1 if (n and S1 >= split[pre]) else 0)
        k = coef[seg] if n else coef[0]
        ex = _exact_T(k, S1, S2, S3, n)
        assert abs(Fraction(float(T[b])) - ex) <= 8 * 2.0**-53 * abs(ex) + 0
        for i in range(n):
            f = [Fraction(float(v)) for v in k]
            exs = f[0] / n + f[1] * pb[i] + f[2] * cb[i] + f[3] * pb[i] ** 2 + f[4] * n
            assert abs(Fraction(float(share[lo + i])) - exs) <= 10 * 2.0**-53 * abs(exs)


def test_additivity_symmetry_vtc():
    """Shares sum to T (problem formulation); identical requests get identical
    shares; with beta = a2 = a3 = a4 = 0 shares are proportional to p (token count)."""
    p, c, ph, t, off, coef, split = _small_random(2)
    T, share = oracle.attribute(off, p, c, ph, split, coef)
    sizes = np.diff(off)
    for b in np.nonzero(sizes)[0]:
        s = math.fsum(share[off[b]:off[b + 1]])
        assert abs(s - T[b]) <= 4 * sizes[b] * 2.0**-52 * T[b]
    # symmetry: duplicate the first request of each batch over the whole batch
    p2, c2, ph2 = p.copy(), c.copy(), ph.copy()
    for b in np.nonzero(sizes)[0]:
        p2[off[b]:off[b + 1]] = p[off[b]]
        c2[off[b]:off[b + 1]] = c[off[b]]
        ph2[off[b]:off[b + 1]] = ph[off[b]]
    T2, s2 = oracle.attribute(off, p2, c2, ph2, split, coef)
    for b in np.nonzero(sizes)[0]:
        seg = s2[off[b]:off[b + 1]]
        assert np.all(seg == seg[0])
    # VTC special case
    vtc = np.zeros_like(coef)
    vtc[:, 1] = np.array([1.5, 2.5, 3.5, 4.5])
    T3, s3 = oracle.attribute(off, p, c, ph, split, vtc)
    nz = sizes > 0
    ratio = s3 / p
    rep = np.repeat(np.arange(len(sizes)), sizes)
    for b in np.nonzero(nz)[0][:50]:
        r = ratio[off[b]:off[b + 1]]
        assert np.all(r == r[0]) and r[0] in (1.5, 2.5, 3.5, 4.5)
    assert rep.shape[0] == p.shape[0]


def test_segment_rule_boundaries():
    """Tie S1 == split is compute-bound; one prefill request makes the batch prefill."""
    coef = np.array([[1, 0, 0, 0, 0], [2, 0, 0, 0, 0], [3, 0, 0, 0, 0], [4, 0, 0, 0, 0]], dtype=np.float64)
    split = [4, 6]
    cases = [  # (p list, phase list, expected T)
        ([1, 1, 1], [0, 0, 0], 1.0), ([1, 1, 1, 1], [0, 0, 0, 0], 2.0), ([2, 3], [1, 1], 3.0),
        ([3, 3], [1, 0], 4.0), ([5, 1], [0, 0], 2.0), ([5], [0], 2.0), ([5], [1], 3.0), ([1], [0], 1.0)]
    for pl, phl, exp in cases:
        T, _ = oracle.attribute([0, len(pl)], pl, [0] * len(pl), phl, split, coef)
        assert T[0] == exp, (pl, phl)


def test_tenant_totals_vs_fsum_and_decomposition():
    """Neumaier totals agree with math.fsum (exactly rounded sum), with the
    integer decomposition of the shares, and are insensitive to request order."""
    x = workloads.config(0, scale=0.05)
    T, share = oracle.attribute(x.offsets, x.p, x.c, x.phase, x.split, x.coef)
    L = oracle.tenant_totals(share, x.tenant, x.n_tenants)
    for u in range(x.n_tenants):
        exact = math.fsum(share[x.tenant == u])
        assert abs(L[u] - exact) <= 2.0**-52 * abs(exact)
    # decomposition: L_u = sum_s [beta_s * sum 1/n_b + a1 P + a2 C + a3 Q + a4 N], exact integer sums
    feat, seg = oracle.batch_features(x.offsets, x.p, x.c, x.phase, x.split)
    sizes = np.diff(x.offsets)
    rseg = np.repeat(seg, sizes)
    rn = np.repeat(sizes, sizes)
    for u in range(x.n_tenants):
        tot = Fraction(0)
        for s in range(4):
            m = (x.tenant == u) & (rseg == s)
            k = [Fraction(float(v)) for v in x.coef[s]]
            inv = sum((Fraction(1, int(n)) for n in rn[m]), Fraction(0))
            P = int(x.p[m].astype(np.int64).sum())
            C = int(x.c[m].astype(np.int64).sum())
            Q = int((x.p[m].astype(np.int64) ** 2).sum())
            N = int(rn[m].sum())
            tot += k[0] * inv + k[1] * P + k[2] * C + k[3] * Q + k[4] * N
        assert abs(Fraction(float(L[u])) - tot) <= 1e-13 * tot
    # order independence
    perm = np.random.default_rng(3).permutation(share.shape[0])
    L2 = oracle.tenant_totals(share[perm], x.tenant[perm], x.n_tenants)
    assert np.max(np.abs(L2 - L) / L) <= 1e-15


def test_tenant_totals_continue_across_calls():
    x = workloads.config(0, scale=0.02)
    _, share = oracle.attribute(x.offsets, x.p, x.c, x.phase, x.split, x.coef)
    acc = oracle.TenantSums(x.n_tenants)
    h = share.shape[0] // 3
    acc.add(share[:h], x.tenant[:h]).add(share[h:], x.tenant[h:])
    for u in range(x.n_tenants):
        assert abs(acc.totals()[u] - math.fsum(share[x.tenant == u])) <= 2.0**-52 * acc.totals()[u]


# ---------------------------------------------------------------- what-if

def test_whatif_brute_force():
    """Each (pending, candidate) pair equals Eq. 1 on the explicitly concatenated
    batch, evaluated here in exact rationals from the integer sums."""
    q = workloads.whatif_config(scale=0.02, n_pending=9)
    c = q.cand
    Tn, Sn = oracle.whatif(c.offsets, c.p, c.c, c.phase, q.p_new, q.c_new, q.phase_new, q.split, q.coef)
    for j in range(q.n_pending):
        for b in range(c.n_batch):
            lo, hi = c.offsets[b], c.offsets[b + 1]
            pb = [int(v) for v in c.p[lo:hi]] + [int(q.p_new[j])]
            cb = [int(v) for v in c.c[lo:hi]] + [int(q.c_new[j])]
            pre = int(any(c.phase[lo:hi] == 1) or q.phase_new[j] == 1)
            n = len(pb)
            S1, S2, S3 = sum(pb), sum(cb), sum(v * v for v in pb)
            seg = pre * 2 + int(S1 >= q.split[pre])
            f = [Fraction(float(v)) for v in q.coef[seg]]
            exT = f[0] + f[1] * S1 + f[2] * S2 + f[3] * S3 + f[4] * n * n
            exS = f[0] / n + f[1] * pb[-1] + f[2] * cb[-1] + f[3] * pb[-1] ** 2 + f[4] * n
            assert abs(Fraction(float(Tn[j, b])) - exT) <= 8 * 2.0**-53 * exT
            assert abs(Fraction(float(Sn[j, b])) - exS) <= 10 * 2.0**-53 * exS


def test_admit_hand_case(golden_dir):
    """The admission predicate on a hand-worked case: equality admits, the
    tenant is the pending request's, and both conditions are required."""
    g = _load(golden_dir, "admit_hand_case.json")
    m = oracle.admit(np.array(g["T_new"]), np.array(g["share_new"]), g["tenant_new"], g["L"], g["budget"], g["slo"])
    assert m.dtype == np.uint8 and m.shape == (2, 3)
    assert np.array_equal(m, np.array(g["expected"], dtype=np.uint8))


def test_admit_brute_force():
    """Against a per-pair restatement in exact rationals on random what-if outputs
    (dyadic values, so the single fp64 addition is exact)."""
    rng = np.random.default_rng(7)
    npd, nc, nt = 13, 17, 5
    T = rng.integers(0, 64, (npd, nc)) / 32.0
    S = rng.integers(0, 64, (npd, nc)) / 64.0
    u = rng.integers(0, nt, npd)
    L = rng.integers(0, 64, nt) / 64.0
    B = rng.integers(0, 128, nt) / 64.0
    m = oracle.admit(T, S, u, L, B, 1.0)
    for j in range(npd):
        for b in range(nc):
            want = Fraction(float(L[u[j]])) + Fraction(float(S[j, b])) <= Fraction(float(B[u[j]])) and T[j, b] <= 1.0
            assert m[j, b] == int(want)


# ---------------------------------------------------------------- fit

def test_accuracy_hand_case():
    """Worked by hand: y = [1, 2, 4, 8], T = [1, 2.2, 3, 8] plus a non-positive
    measurement that must be ignored; R^2 restated in exact rationals."""
    y = np.array([1.0, 2.0, 4.0, 0.0, 8.0])
    T = np.array([1.0, 2.2, 3.0, 5.0, 8.0])
    a = oracle.accuracy(y, T)
    assert a["n"] == 4
    rel = sorted([0.0, abs(2.2 - 2.0) / 2.0, 0.25, 0.0])
    assert a["p50"] == rel[1] and a["p90"] == rel[3] and a["p99"] == rel[3]
    assert abs(a["mean_rel"] - sum(rel) / 4) <= 1e-16
    ys = [Fraction(v) for v in (1.0, 2.0, 4.0, 8.0)]
    ts = [Fraction(v) for v in (1.0, 2.2, 3.0, 8.0)]
    my, mt = sum(ys) / 4, sum(ts) / 4
    sxx = sum((v - my) ** 2 for v in ys)
    syy = sum((v - mt) ** 2 for v in ts)
    sxy = sum((u - my) * (v - mt) for u, v in zip(ys, ts))
    ssr = sum((u - v) ** 2 for u, v in zip(ys, ts))
    assert abs(a["r2_ssr"] - float(1 - ssr / sxx)) <= 1e-15
    assert abs(a["r2_corr"] - float(sxy * sxy / (sxx * syy))) <= 1e-15


def test_accuracy_invariants_and_ranks():
    rng = np.random.default_rng(2)
    y = rng.uniform(0.5, 2.0, 1000)
    a = oracle.accuracy(y, y)
    assert a["r2_ssr"] == 1.0 and a["r2_corr"] == 1.0 and a["p99"] == 0.0 and a["mean_rel"] == 0.0
    assert oracle.accuracy(y, 2 * y)["r2_corr"] == 1.0  # an affine prediction is perfectly correlated
    assert oracle.accuracy(y, 2 * y)["p50"] == 1.0
    # nearest rank: with relative errors 1..100 (x 1/128) the q-th percentile is the q-th value
    e = np.arange(1, 101) / 128.0
    a = oracle.accuracy(np.ones(100), 1.0 + rng.permutation(e))
    assert (a["p50"], a["p90"], a["p99"]) == (e[49], e[89], e[98])
    a = oracle.accuracy(np.ones(1), np.array([1.5]))
    assert a["p50"] == a["p99"] == 0.5
    assert math.isnan(oracle.accuracy(np.zeros(3), np.ones(3))["r2_ssr"])


def test_vtc_fit_pins():
    """Exact recovery of a noiseless line, the line through two points, empty
    batches skipped, degenerate cases, and agreement with numpy's least squares."""
    S1 = np.array([3, 7, 1, 12, 5], dtype=np.int64)
    n = np.array([1, 2, 1, 3, 0])
    y = 0.25 + 0.0625 * S1.astype(np.float64)
    assert oracle.vtc_fit(S1, n, y) == (0.25, 0.0625, oracle.OK, 4)
    b, a, st, m = oracle.vtc_fit(np.array([2, 6]), np.array([1, 1]), np.array([1.0, 3.0]))
    assert (b, a, st, m) == (0.0, 0.5, oracle.OK, 2)
    assert oracle.vtc_fit(np.array([4, 4, 4]), np.ones(3), np.array([1.0, 2.0, 3.0]))[2] == oracle.ESINGULAR
    assert oracle.vtc_fit(np.array([4]), np.ones(1), np.array([1.0]))[2] == oracle.ENODATA
    rng = np.random.default_rng(4)
    S1 = rng.integers(1, 4000, 300)
    y = 1e-3 + 2e-6 * S1 * np.exp(0.05 * rng.standard_normal(300))
    b, a, st, m = oracle.vtc_fit(S1, np.ones(300), y)
    ref = np.linalg.lstsq(np.stack([np.ones(300), S1.astype(np.float64)], 1), y, rcond=None)[0]
    assert st == oracle.OK and abs(b - ref[0]) <= 1e-9 * abs(ref[0]) and abs(a - ref[1]) <= 1e-9 * abs(ref[1])


def _fit_data(scale=0.004, seed_noise=True):
    x = workloads.config(2, scale=scale)
    feat, seg = oracle.batch_features(x.offsets, x.p, x.c, x.phase, x.split)
    y0 = oracle.batch_latency(feat, seg, x.coef)
    return x, feat, seg, y0


def test_fit_noiseless_recovery():
    x, feat, seg, y0 = _fit_data()
    res = oracle.fit(feat, seg, y0)
    assert [r["status"] for r in res] == [0, oracle.ENODATA, 0, 0]
    for g in (0, 2, 3):
        truth = x.coef[g].copy()
        if res[g]["dropped"] & 8:
            truth[1] += truth[3]
            truth[3] = 0.0
        nz = truth != 0
        assert np.all(np.abs(res[g]["coef"][nz] - truth[nz]) <= 1e-9 * np.abs(truth[nz]))
        assert res[g]["coef"][~nz].tolist() == [0.0] * int((~nz).sum())
    assert res[0]["dropped"] == 8 and res[2]["dropped"] == 0


def test_fit_exact_interpolation_small():
    """Integer coefficients and integer-valued y: the exact solution is recovered exactly."""
    X = np.array([[1, 3, 5, 9, 4], [1, 7, 1, 29, 9], [1, 2, 8, 4, 1], [1, 9, 0, 41, 16], [1, 4, 4, 8, 4],
                  [1, 6, 3, 20, 9]], dtype=np.int64)
    a = np.array([5.0, -2.0, 3.0, 0.5, 0.25])
    y = X.astype(np.float64) @ a
    r = oracle.fit_group(X, y)
    assert r["status"] == 0 and r["coef"].tolist() == a.tolist()
    assert r["ssr"] == 0.0 and r["r2"] == 1.0


def test_fit_matches_lstsq():
    """Against LAPACK least squares (numpy.linalg.lstsq) on column-equilibrated data."""
    x, feat, seg, y0 = _fit_data(scale=0.002)
    y = y0 * x.noise
    res = oracle.fit(feat, seg, y)
    nonempty = feat[3] > 0
    for g in (0, 2, 3):
        sel = (seg == g) & nonempty
        X = np.stack([np.ones(sel.sum()), feat[0, sel], feat[1, sel], feat[2, sel], feat[4, sel]], 1).astype(float)
        cols = [0, 1, 2, 4] if res[g]["dropped"] & 8 else [0, 1, 2, 3, 4]
        Xs = X[:, cols]
        sc = np.abs(Xs).max(axis=0)
        sol, *_ = np.linalg.lstsq(Xs / sc, y[sel], rcond=None)
        pred_l = (Xs / sc) @ sol
        pred_o = X @ res[g]["coef"]
        assert np.max(np.abs(pred_l - pred_o) / np.abs(pred_o)) < 1e-9
        assert res[g]["r2"] > 0.9 and 0 < res[g]["ssr"]


def test_fit_column_scaling_invariance():
    """Physical units (features times phi) give the same fitted predictions."""
    x, feat, seg, y0 = _fit_data(scale=0.002)
    y = y0 * x.noise
    phi, W = oracle.arch_constants(x.arch)
    res = oracle.fit(feat, seg, y)
    for g in (2, 3):
        sel = (seg == g) & (feat[3] > 0)
        X = np.stack([np.ones(sel.sum(), dtype=np.int64), feat[0, sel], feat[1, sel], feat[2, sel], feat[4, sel]], 1)
        Xp = X.copy()
        Xp[:, 1] *= phi[0]
        Xp[:, 2] *= phi[1]
        Xp[:, 3] *= phi[2]
        Xp[:, 0] *= W
        rp = oracle.fit_group(Xp, y[sel])
        pred = X.astype(float) @ res[g]["coef"]
        predp = np.array([sum(Fraction(int(v)) * Fraction(float(cf)) for v, cf in zip(row, rp["coef"]))
                          for row in Xp[:200]], dtype=object).astype(float)
        assert np.max(np.abs(predp - pred[:200]) / pred[:200]) < 1e-12


def test_fit_degenerate_groups():
    # fewer samples than columns
    X = np.array([[1, 3, 5, 9, 4], [1, 7, 1, 29, 9]], dtype=np.int64)
    assert oracle.fit_group(X, np.array([1.0, 2.0]))["status"] == oracle.ENODATA
    # constant n: the n^2 column is a multiple of the intercept -> singular
    X = np.array([[1, s1, s2, s3, 16] for s1, s2, s3 in [(3, 5, 9), (7, 1, 29), (2, 8, 4), (9, 0, 41), (4, 4, 8),
                                                          (6, 3, 20)]], dtype=np.int64)
    assert oracle.fit_group(X, np.arange(6, dtype=float) + 1)["status"] == oracle.ESINGULAR
    # decode-like group: S1 == S3 everywhere -> a3 dropped, a1 carries a1 + a3
    n = np.array([1, 2, 3, 5, 8, 13, 21])
    S2 = np.array([10, 40, 7, 80, 90, 300, 11])
    X = np.stack([np.ones(7, dtype=np.int64), n, S2, n, n * n], 1)
    a = np.array([2.0, 3.0, 0.5, 1.0, 0.125])
    y = X.astype(float) @ a
    r = oracle.fit_group(X, y)
    assert r["status"] == 0 and r["dropped"] == 8
    assert r["coef"].tolist() == [2.0, 4.0, 0.5, 0.0, 0.125]


def test_plausible_mistakes_are_caught(golden_dir):
    """A planted mistake (swapped a2/a3 columns in the coefficient layout)
    breaks the hand-computed values even though additivity still holds."""
    g = _load(golden_dir, "eq1_hand_cases.json")
    coef = np.array(g["coef"], dtype=np.float64)
    bad = coef[:, [0, 1, 3, 2, 4]]
    T, share = oracle.attribute(g["offsets"], g["p"], g["c"], g["phase"], g["split"], bad)
    assert T.tolist() != g["T"]
    sizes = np.diff(g["offsets"])
    for b in np.nonzero(sizes)[0]:
        assert math.isclose(math.fsum(share[g["offsets"][b]:g["offsets"][b + 1]]), T[b], rel_tol=1e-15)


# ---------------------------------------------------------------- the pins catch planted mistakes

_MUTANTS = [
    ("wrong feature index in Eq. 1", "T = T + k[2] * (double)f[1];", "T = T + k[2] * (double)f[2];"),
    ("dropped a4 term in the share", "t = t + k[4] * (double)n;", "t = t + 0.0 * (double)n;"),
    ("beta not split", "double t = k[0] / (double)n;", "double t = k[0];"),
    ("regime tie goes memory-bound", "S1 >= split[prefill]", "S1 > split[prefill]"),
    ("batch phase from decode requests", "if (phase[i] == 1) prefill = 1;", "if (phase[i] == 0) prefill = 1;"),
    ("linear |B| instead of sum_i |B|", "feat[4] = n * n;", "feat[4] = n;"),
    ("p*c instead of p^2", "S3 += (int64_t)p[i] * (int64_t)p[i];", "S3 += (int64_t)p[i] * (int64_t)c[i];"),
    ("Neumaier compensation sign", "comp[u] += (s - t) + x;", "comp[u] += (t - s) + x;"),
    ("what-if appends the wrong field", "bp[n0] = p_new[j];", "bp[n0] = c_new[j];"),
    ("one KV projection only", "ovf |= mul64(2 * d, kv, &t2);", "ovf |= mul64(d, kv, &t2);"),
    ("attention phi without the factor 2", "ovf |= mul64(2 * L, q, &a);", "ovf |= mul64(L, q, &a);"),
]


def _pins_pass(golden_dir):
    """Run the golden pins against whichever oracle build is active; True if all hold."""
    g = _load(golden_dir, "eq1_hand_cases.json")
    coef = np.array(g["coef"], dtype=np.float64)
    ok = True
    feat, seg = oracle.batch_features(g["offsets"], g["p"], g["c"], g["phase"], g["split"])
    ok &= feat.T.tolist() == g["batch_feat_S1_S2_S3_n_n2"] and seg.tolist() == g["batch_seg"]
    T, share = oracle.attribute(g["offsets"], g["p"], g["c"], g["phase"], g["split"], coef)
    ok &= T.tolist() == g["T"] and share.tolist() == g["share"]
    ok &= oracle.tenant_totals(share, g["tenant"], g["n_tenants"]).tolist() == g["tenant_totals"]
    w = g["whatif"]
    Tn, Sn = oracle.whatif(w["cand_offsets"], w["cand_p"], w["cand_c"], w["cand_phase"], w["p_new"], w["c_new"],
                           w["phase_new"], g["split"], coef)
    ok &= Tn.tolist() == w["T_new"] and Sn.tolist() == w["share_new"]
    a = _load(golden_dir, "arch_constants.json")
    for case in a["cases"]:
        phi, W = oracle.arch_constants(case["arch"])
        ok &= phi.tolist() == case["phi"] and W == case["W"]
    return bool(ok)


@pytest.mark.parametrize("name,old,new", _MUTANTS, ids=[m[0] for m in _MUTANTS])
def test_pins_catch_mutant(golden_dir, tmp_path, name, old, new):
    import subprocess
    src = open(os.path.join(os.path.dirname(oracle.__file__), "lvo.c")).read()
    assert src.count(old) == 1, name
    mut = tmp_path / "lvo_mut.c"
    mut.write_text(src.replace(old, new))
    so = tmp_path / "liblvo_mut.so"
    subprocess.run(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fPIC", "-shared", "-o", str(so), str(mut),
                    "-lm"], check=True)
    assert _pins_pass(golden_dir)
    with oracle.using(str(so)):
        assert not _pins_pass(golden_dir), f"mutant not caught: {name}"
