"""Exact least-squares fit of Eq. 1's coefficients -- TEST INFRASTRUCTURE ONLY.

Section 2.1 fits the coefficient sets (beta, a1, a2, a3, a4) "via ordinary
least squares on profiling data", one set per phase and regime, four in all.
For each segment g the design matrix has one row per profiled batch of that
segment, ``x_b = [1, S1, S2, S3, n^2]`` (the Eq. 1 sums), and the target is the
measured latency ``y_b``.  The oracle solves the normal equations
``(X^T X) a = X^T y`` EXACTLY, in rational arithmetic: the Gram matrix is a sum
of integer products (Python ints), ``X^T y`` an exact dyadic rational (every
float is one), and Gaussian elimination runs on ``fractions.Fraction``.  The
exact solution is rounded once to double.  Being exact, the result does not
depend on conditioning or summation order.

Readings taken where the paper is silent:
  * Decode steps have p_i = 1, so S1 == S3 in every decode batch and a1, a3
    cannot be told apart.  When every batch of a group has S1 == S3 the a3
    column is dropped; a1 then carries a1 + a3 and a3 is reported as 0.
  * Empty batches (n = 0) are not profiling samples and are skipped.
  * Fewer samples than kept columns -> status ENODATA; an exactly singular Gram
    matrix -> ESINGULAR.  Either way that group's coefficients are NaN here.

Only tests/, __graft_entry__.smoke() and bench.py's CPU baseline may use this.
"""

from __future__ import annotations

from fractions import Fraction

import numpy as np

OK, ENODATA, ESINGULAR = 0, -3, -4


def _exact_targets(y: np.ndarray):
    """Return (Y ints as object array, E) with y_b == Y_b * 2**E exactly."""
    y = np.asarray(y, dtype=np.float64)
    if y.size == 0:
        return np.zeros(0, dtype=object), 0
    if not np.all(np.isfinite(y)):
        raise ValueError("non-finite latency")
    mant, ex = np.frexp(y)                      # y = mant * 2**ex, 0.5 <= |mant| < 1
    M = np.ldexp(mant, 53).astype(np.int64)     # exact 53-bit integer mantissas
    sh = ex.astype(np.int64) - 53
    E = int(sh.min())
    Y = np.empty(y.size, dtype=object)
    shifts = (sh - E).tolist()
    ms = M.tolist()
    for i, (m, s) in enumerate(zip(ms, shifts)):
        Y[i] = m << s
    return Y, E


def _solve_exact(G, r):
    """Gaussian elimination over the rationals.  Returns None when singular."""
    k = len(r)
    A = [[Fraction(G[i][j]) for j in range(k)] + [r[i]] for i in range(k)]
    for col in range(k):
        piv = next((i for i in range(col, k) if A[i][col] != 0), None)
        if piv is None:
            return None
        A[col], A[piv] = A[piv], A[col]
        for i in range(k):
            if i != col and A[i][col] != 0:
                f = A[i][col] / A[col][col]
                A[i] = [a - f * b for a, b in zip(A[i], A[col])]
    return [A[i][k] / A[i][i] for i in range(k)]


def fit_group(X: np.ndarray, y: np.ndarray):
    """Exact OLS for one group.  X int64[m, 5] columns [1, S1, S2, S3, n^2].

    Returns dict(status, coef float64[5], dropped bitmask, n, ssr, r2, exact).
    """
    m = X.shape[0]
    res = dict(status=OK, coef=np.full(5, np.nan), dropped=0, n=m, ssr=np.nan, r2=np.nan, exact=None)
    cols = [0, 1, 2, 3, 4]
    if m > 0 and np.array_equal(X[:, 1], X[:, 3]):
        cols.remove(3)
        res["dropped"] = 1 << 3
    k = len(cols)
    if m < k:
        res["status"] = ENODATA
        return res
    Xo = X[:, cols].astype(object)
    Y, E = _exact_targets(y)
    G = [[int(np.dot(Xo[:, a], Xo[:, b])) for b in range(k)] for a in range(k)]
    rY = [int(np.dot(Xo[:, a], Y)) for a in range(k)]
    scale = Fraction(2) ** E
    r = [Fraction(v) * scale for v in rY]
    sol = _solve_exact(G, r)
    if sol is None:
        res["status"] = ESINGULAR
        return res
    coef = np.zeros(5)
    for j, cidx in enumerate(cols):
        coef[cidx] = float(sol[j])           # correctly rounded
    res["coef"] = coef
    res["exact"] = {cidx: sol[j] for j, cidx in enumerate(cols)}
    # Residuals of the ROUNDED coefficients, exactly: SSR = y'y - 2 c'X'y + c'Gc.
    cr = [Fraction(float(coef[cidx])) for cidx in cols]
    yy = Fraction(int(np.dot(Y, Y))) * scale * scale
    cXy = sum(ci * ri for ci, ri in zip(cr, r))
    cGc = sum(cr[a] * G[a][b] * cr[b] for a in range(k) for b in range(k))
    ssr = yy - 2 * cXy + cGc
    sy = Fraction(int(Y.sum())) * scale
    sst = yy - sy * sy / m
    res["ssr"] = float(ssr)
    res["r2"] = float(1 - ssr / sst) if sst != 0 else np.nan
    return res


def fit(feat: np.ndarray, seg: np.ndarray, y: np.ndarray):
    """Per-segment exact OLS.

    feat: int64[5, n_batch] rows (S1, S2, S3, n, n^2) as produced by the oracle's
    batch reduction; seg: uint8[n_batch] segment codes phase*2 + regime;
    y: float64[n_batch] latencies.  Returns a list of four fit_group results.
    """
    feat = np.asarray(feat, dtype=np.int64)
    seg = np.asarray(seg)
    y = np.asarray(y, dtype=np.float64)
    nonempty = feat[3] > 0
    out = []
    for g in range(4):
        sel = (seg == g) & nonempty
        X = np.stack([np.ones(int(sel.sum()), dtype=np.int64), feat[0, sel], feat[1, sel], feat[2, sel],
                      feat[4, sel]], axis=1)
        out.append(fit_group(X, y[sel]))
    return out


def vtc_fit(S1: np.ndarray, n: np.ndarray, y: np.ndarray):
    """The token-count baseline the paper compares against (VTC, Tables 1-2): one
    least-squares line T = beta + a * S1 over every profiled batch, whatever its
    phase and regime, S1 being the batch's total new tokens.  Exact normal
    equations in rationals, rounded once; empty batches (n = 0) are skipped.
    Returns (beta, a, status, count); beta and a are NaN unless status is OK."""
    S1 = np.asarray(S1, dtype=np.int64)
    sel = np.asarray(n) > 0
    S = [int(v) for v in S1[sel].tolist()]
    Y, E = _exact_targets(np.asarray(y, dtype=np.float64)[sel])
    m = len(S)
    if m < 2:
        return float("nan"), float("nan"), ENODATA, m
    G = [[m, sum(S)], [sum(S), sum(v * v for v in S)]]
    scale = Fraction(2) ** E
    r = [Fraction(sum(Y.tolist())) * scale, Fraction(sum(s * yv for s, yv in zip(S, Y.tolist()))) * scale]
    sol = _solve_exact(G, r)
    if sol is None:
        return float("nan"), float("nan"), ESINGULAR, m
    return float(sol[0]), float(sol[1]), OK, m


def accuracy(y: np.ndarray, T: np.ndarray):
    """Accuracy of predicted batch latencies T against measured y, as the paper
    reports it (Section 3.2, Tables 1-2): R^2 in both of its usual forms and
    percentiles of the relative error, over the batches with y > 0 (m of them).
      r2_ssr   = 1 - sum (y - T)^2 / sum (y - mean y)^2
      r2_corr  = (sum (y - mean y)(T - mean T))^2 / (sum (y - mean y)^2 sum (T - mean T)^2)
      rel_b    = |T_b - y_b| / y_b; mean_rel is its mean, and p50, p90, p99 are
                 nearest-rank percentiles: the ceil(q m)-th smallest of the m.
    Sums are correctly rounded (math.fsum); an R^2 whose denominator is 0 is
    NaN; with m = 0 every value is NaN."""
    import math
    y = np.asarray(y, dtype=np.float64)
    T = np.asarray(T, dtype=np.float64)
    sel = y > 0
    y, T = y[sel], T[sel]
    m = int(y.size)
    nan = float("nan")
    out = {"n": m, "r2_ssr": nan, "r2_corr": nan, "mean_rel": nan, "p50": nan, "p90": nan, "p99": nan}
    if m == 0:
        return out
    my, mT = math.fsum(y.tolist()) / m, math.fsum(T.tolist()) / m
    dy, dT = y - my, T - mT
    sxx = math.fsum((dy * dy).tolist())
    syy = math.fsum((dT * dT).tolist())
    sxy = math.fsum((dy * dT).tolist())
    ssr = math.fsum(((y - T) ** 2).tolist())
    out["r2_ssr"] = 1.0 - ssr / sxx if sxx != 0 else nan
    out["r2_corr"] = sxy * sxy / (sxx * syy) if sxx != 0 and syy != 0 else nan
    rel = np.abs(T - y) / y
    out["mean_rel"] = math.fsum(rel.tolist()) / m
    srt = np.sort(rel)
    for name, q in (("p50", 50), ("p90", 90), ("p99", 99)):
        k = -(-q * m // 100)  # ceil(q m / 100), exact in integers
        out[name] = float(srt[k - 1])
    return out
