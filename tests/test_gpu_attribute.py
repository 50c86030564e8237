"""GPU parity of features, Eq. 1, shares and tenant totals against the CPU oracle.

Tolerances: integer features, aggregates and segment codes bit-exact; fp64 T,
shares and tenant totals within 1e-12 relative.  Shares are compared by plain
relative error |s - s_o| / |s_o|; only the case built to cancel (a negative
coefficient, where the oracle's own left-to-right rounding error is relative to
its largest term rather than to the result) measures it against
max(|s_o|, T_b/n).  The FP64 arithmetic mode evaluates in the oracle's order
and must be bit-identical.
"""

import math
from fractions import Fraction

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


def _dev(lv, w, tenant=True):
    return lv.batches_to_device(w.p, w.c, w.phase, w.offsets, w.tenant if tenant else None, w.n_tenants)


def _run(lv, ctx, w, acc=True, arith=0):
    import torch
    ctx.set_arith(arith)
    b = _dev(lv, w, tenant=acc)
    model = lv.make_model(w.coef, w.split)
    T = torch.full((w.n_batch,), float("nan"), dtype=torch.float64, device="cuda")
    share = torch.full((w.n_req,), float("nan"), dtype=torch.float64, device="cuda")
    L = None
    if acc:
        a = lv.TenantAcc(ctx, w.n_tenants)
        lv.lv_attribute(ctx, model, b, T, share, a)
        L = torch.empty(w.n_tenants, dtype=torch.float64, device="cuda")
        lv.lv_tenant_totals(ctx, a, L)
        L = L.cpu().numpy()
    else:
        lv.lv_attribute(ctx, model, b, T, share, None)
    st = ctx.status()
    ctx.set_arith(0)
    return T.cpu().numpy(), share.cpu().numpy(), L, st


def exact_tenant_total(shares):
    """Correctly rounded sum of shares each rounded (half to even) to a multiple of 2^-72."""
    tot = 0
    for v in shares.tolist():
        tot += round(Fraction(v) * 2**72)
    return float(Fraction(tot, 2**72))


def _share_den(T_o, off, s_o):
    sizes = np.diff(off)
    return np.maximum(np.abs(s_o), np.repeat(np.abs(T_o) / np.maximum(sizes, 1), sizes))


def _share_err(share, s_o, T_o, off, guarded=False):
    """Largest relative share error: plain |s - s_o| / |s_o| (zero oracle shares must be
    zero), or against max(|s_o|, T_b/n) where `guarded` (a case built to cancel)."""
    if guarded:
        return float(np.max(np.abs(share - s_o) / _share_den(T_o, off, s_o)))
    z = s_o == 0
    assert np.all(share[z] == 0)
    return float(np.max(np.abs(share[~z] - s_o[~z]) / np.abs(s_o[~z]))) if (~z).any() else 0.0


def _check_parity(w, T, share, L, guarded=False):
    T_o, s_o = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
    nz = T_o != 0
    assert np.all(T[~nz] == 0)
    errT = np.max(np.abs(T[nz] - T_o[nz]) / np.abs(T_o[nz])) if nz.any() else 0.0
    assert errT <= TOL, errT
    if w.n_req:
        errS = _share_err(share, s_o, T_o, w.offsets, guarded)
        assert errS <= TOL, errS
    if L is not None:
        L_o = oracle.tenant_totals(s_o, w.tenant, w.n_tenants)
        m = L_o != 0
        assert np.all(L[~m] == 0)
        if m.any():
            errL = np.max(np.abs(L[m] - L_o[m]) / np.abs(L_o[m]))
            assert errL <= TOL, errL
        # exactness: each GPU total is the correctly rounded exact sum of the GPU's own
        # shares, every share first rounded to a multiple of 2^-72 s
        for u in (np.unique(w.tenant)[:64] if w.n_req <= 3_000_000 else []):
            assert L[u] == exact_tenant_total(share[w.tenant == u])
    return T_o, s_o


def _wl(p, c, ph, off, tenant, nt, coef=None, split=(256, 256), name="case"):
    if coef is None:
        coef, _ = workloads.draw_coefficients(np.random.default_rng(7), "llama3.1-8b")
    return workloads.Workload(name=name, arch=np.asarray(workloads.ARCHS["llama3.1-8b"], np.int32),
                              p=np.asarray(p, np.int32), c=np.asarray(c, np.int32), phase=np.asarray(ph, np.int32),
                              tenant=np.asarray(tenant, np.int32), offsets=np.asarray(off, np.int64),
                              n_tenants=int(nt), coef=np.asarray(coef, np.float64),
                              split=np.asarray(split, np.int64))


def _from_sizes(rng, sizes, nt=5, pmax=20000, cmax=131072, pre=0.3, split=(256, 256)):
    off = np.zeros(len(sizes) + 1, np.int64)
    np.cumsum(sizes, out=off[1:])
    n = int(off[-1])
    ph = (rng.random(n) < pre).astype(np.int32)
    p = np.where(ph == 1, rng.integers(1, pmax + 1, n), 1).astype(np.int32)
    c = np.where(ph == 1, 0, rng.integers(0, cmax + 1, n)).astype(np.int32)
    t = rng.integers(0, nt, n).astype(np.int32)
    return _wl(p, c, ph, off, t, nt, split=split)


# ------------------------------------------------------------------ hand cases

def test_hand_cases_exact(lv, ctx, golden_dir):
    import json
    import os
    g = json.load(open(os.path.join(golden_dir, "eq1_hand_cases.json")))
    w = _wl(g["p"], g["c"], g["phase"], g["offsets"], g["tenant"], g["n_tenants"], coef=g["coef"], split=g["split"])
    for arith in (0, 1):
        T, share, L, st = _run(lv, ctx, w, arith=arith)
        assert st == lv.LV_OK
        assert T.tolist() == g["T"] and share.tolist() == g["share"] and L.tolist() == g["tenant_totals"]


# ------------------------------------------------------------------ parity

@pytest.mark.parametrize("arith", [0, 1])
def test_config0_parity(lv, ctx, arith):
    w = workloads.config(0)
    T, share, L, st = _run(lv, ctx, w, arith=arith)
    assert st == lv.LV_OK
    T_o, s_o = _check_parity(w, T, share, L)
    if arith == 1:  # fp64 mode follows the oracle's rounding sequence
        assert np.array_equal(T, T_o) and np.array_equal(share, s_o)


def test_shapes_adversarial(lv, ctx):
    """Empty batches, size-1 batches, batches far larger than a tile (block-wide
    path), batches straddling every tile boundary, n_req not a multiple of 4."""
    rng = np.random.default_rng(11)
    cases = [
        [0, 0, 3, 0, 1, 0, 0, 0, 5],
        [1] * 5000,
        [4096, 1, 4095, 2, 0, 9000, 3],
        list(rng.integers(0, 3, 3000)) + [2047, 2048, 2049, 1023, 1024, 1025],
        [0] * 2500 + [7] + [0] * 2500,
        [100000] + [1] * 7,
        list(rng.integers(1, 4097, 300)),
        [3],
        [0],
    ]
    for sizes in cases:
        w = _from_sizes(rng, np.asarray(sizes))
        T, share, L, st = _run(lv, ctx, w)
        assert st == lv.LV_OK, sizes[:8]
        _check_parity(w, T, share, L)


def test_all_one_tenant_and_last_tenant(lv, ctx):
    rng = np.random.default_rng(3)
    w = _from_sizes(rng, rng.integers(1, 300, 2000), nt=1)
    T, share, L, st = _run(lv, ctx, w)
    _check_parity(w, T, share, L)
    w2 = _from_sizes(rng, rng.integers(1, 300, 2000), nt=70000)
    w2.tenant[:] = 69999
    T, share, L, st = _run(lv, ctx, w2)
    assert st == lv.LV_OK
    _check_parity(w2, T, share, L)


def test_segment_boundaries_and_ties(lv, ctx):
    """S1 == split exactly in both phases; decode batch of exactly 256."""
    rng = np.random.default_rng(5)
    sizes = [256, 255, 257, 1, 2]
    w = _from_sizes(rng, np.asarray(sizes), pre=0.0)
    w.split[:] = (256, 300)
    T, share, L, st = _run(lv, ctx, w)
    T_o, _ = _check_parity(w, T, share, L)
    feat, seg = oracle.batch_features(w.offsets, w.p, w.c, w.phase, w.split)
    assert seg.tolist() == [1, 0, 1, 0, 0]


def test_wide_coefficients_use_fp64_path(lv, ctx):
    """Coefficients too far apart for the integer path fall back to fp64, still in tolerance."""
    rng = np.random.default_rng(9)
    w = _from_sizes(rng, rng.integers(1, 200, 3000))
    w.coef[:, 3] = 1e-290
    T, share, L, st = _run(lv, ctx, w)
    _check_parity(w, T, share, L)


@pytest.mark.parametrize("scale", ["low", "high"])
def test_fixed_point_value_ranges(lv, ctx, scale):
    """Shares whose exact fixed-point value lies below 2^64 or at or above 2^96 (outside the
    decode fast path's window) are attributed exactly all the same, with and without tenants."""
    rng = np.random.default_rng(11)
    w = _from_sizes(rng, rng.integers(1, 300, 3000), pre=0.05)
    if scale == "low":
        # power-of-two coefficients: the scale is set by beta (2^-10 - 66), values near 2^59
        w.coef[:] = [2.0 ** -10, 2.0 ** -20, 2.0 ** -27, 2.0 ** -33, 2.0 ** -27]
    else:
        # an odd multiple of 2^-130 in a4 puts the scale at 2^-130, values near 2^115
        w.coef[:, 4] = 3.0 * 2.0 ** -130
    for acc in (True, False):
        T, share, L, st = _run(lv, ctx, w, acc=acc)
        assert st == lv.LV_OK
        _check_parity(w, T, share, L)


def test_negative_coefficient_cancellation(lv, ctx):
    rng = np.random.default_rng(10)
    w = _from_sizes(rng, rng.integers(1, 200, 3000))
    w.coef[:, 4] = -1e-9
    T, share, L, st = _run(lv, ctx, w)
    _check_parity(w, T, share, L, guarded=True)


def test_outputs_only_8_byte_aligned(lv, ctx):
    """Share and T arrays need only 8-byte alignment: an output offset by one double gives the
    same bits as an aligned one (the kernel falls back from its 16-byte stores)."""
    import torch
    w = workloads.config(0, scale=0.1)
    b = _dev(lv, w)
    model = lv.make_model(w.coef, w.split)
    outs = []
    for off in (0, 1):
        T = torch.full((w.n_batch + off,), float("nan"), dtype=torch.float64, device="cuda")[off:]
        S = torch.full((w.n_req + off,), float("nan"), dtype=torch.float64, device="cuda")[off:]
        a = lv.TenantAcc(ctx, w.n_tenants)
        lv.lv_attribute(ctx, model, b, T, S, a)
        L = torch.empty(w.n_tenants, dtype=torch.float64, device="cuda")
        lv.lv_tenant_totals(ctx, a, L)
        assert ctx.status() == lv.LV_OK
        outs.append((T.cpu().numpy(), S.cpu().numpy(), L.cpu().numpy()))
    for x, y in zip(*outs):
        assert np.array_equal(x.view(np.int64), y.view(np.int64))
    _check_parity(w, *outs[1])


def test_determinism(lv, ctx):
    w = workloads.config(4, scale=0.02)
    a = _run(lv, ctx, w)
    b = _run(lv, ctx, w)
    assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1]) and np.array_equal(a[2], b[2])
    _check_parity(w, *a[:3])


# ------------------------------------------------------------------ features / Eq. 1 alone

def test_features_and_batch_latency(lv, ctx):
    import torch
    w = workloads.config(0, scale=0.3)
    b = _dev(lv, w)
    model = lv.make_model(w.coef, w.split)
    rf = torch.empty((3, w.n_req), dtype=torch.int64, device="cuda")
    bf = torch.empty((5, w.n_batch), dtype=torch.int64, device="cuda")
    bs = torch.empty(w.n_batch, dtype=torch.uint8, device="cuda")
    lv.lv_features(ctx, b, arch=w.arch, model=model, req_feat=rf, batch_feat=bf, batch_seg=bs)
    T = torch.empty(w.n_batch, dtype=torch.float64, device="cuda")
    lv.lv_batch_latency(ctx, model, bf, bs, T)
    assert ctx.status() == lv.LV_OK
    phi, W = oracle.arch_constants(w.arch)
    assert np.array_equal(rf.cpu().numpy(), oracle.request_features(w.p, w.c, phi))
    feat, seg = oracle.batch_features(w.offsets, w.p, w.c, w.phase, w.split)
    assert np.array_equal(bf.cpu().numpy(), feat) and np.array_equal(bs.cpu().numpy(), seg)
    T_o = oracle.batch_latency(feat, seg, w.coef)
    assert np.max(np.abs(T.cpu().numpy() - T_o) / T_o) <= TOL


def test_features_skew_workload(lv, ctx):
    """lv_features on the skew workload (Pareto batch sizes up to 4096): batches above the
    warp kernel's size limit take the block-wide kernel, whose S1..n^2 and segment codes are
    compared bit for bit here, as are the per-request physical features."""
    import torch
    w = workloads.config(4, scale=0.1)
    assert np.diff(w.offsets).max() > 512
    b = _dev(lv, w, tenant=False)
    model = lv.make_model(w.coef, w.split)
    rf = torch.empty((3, w.n_req), dtype=torch.int64, device="cuda")
    bf = torch.empty((5, w.n_batch), dtype=torch.int64, device="cuda")
    bs = torch.empty(w.n_batch, dtype=torch.uint8, device="cuda")
    lv.lv_features(ctx, b, arch=w.arch, model=model, req_feat=rf, batch_feat=bf, batch_seg=bs)
    assert ctx.status() == lv.LV_OK
    phi, _ = oracle.arch_constants(w.arch)
    assert np.array_equal(rf.cpu().numpy(), oracle.request_features(w.p, w.c, phi))
    feat, seg = oracle.batch_features(w.offsets, w.p, w.c, w.phase, w.split)
    assert np.array_equal(bf.cpu().numpy(), feat)
    assert np.array_equal(bs.cpu().numpy(), seg)


def test_request_feature_overflow_saturates(lv, ctx):
    """A physical feature beyond int64 is stored as INT64_MAX and records LV_EDATA; every
    other element stays exact (products checked in Python integers)."""
    import torch
    rng = np.random.default_rng(21)
    w = _from_sizes(rng, rng.integers(1, 40, 200))
    big = [3, 77, w.n_req - 1]
    w.p[big] = 2**31 - 1          # p * phi0 and p^2 * phi2 exceed int64 for the 8B model
    w.c[5] = 2**31 - 1            # c * phi1 = 2^31 * 2^17 stays below 2^63: exact
    b = _dev(lv, w, tenant=False)
    rf = torch.empty((3, w.n_req), dtype=torch.int64, device="cuda")
    lv.lv_features(ctx, b, arch=w.arch, req_feat=rf)
    assert ctx.status() == lv.LV_EDATA
    phi, _ = oracle.arch_constants(w.arch)
    got = rf.cpu().numpy()
    imax = np.iinfo(np.int64).max
    for i in range(w.n_req):
        p, c = int(w.p[i]), int(w.c[i])
        for k, v in enumerate((p * int(phi[0]), c * int(phi[1]), p * p * int(phi[2]))):
            assert int(got[k, i]) == (v if v <= imax else imax), (i, k)
    assert ctx.status() == lv.LV_OK


# ------------------------------------------------------------------ tenant accumulator

def test_tenant_accumulate_continue_export_import(lv, ctx):
    import torch
    w = workloads.config(0, scale=0.2)
    T_o, s_o = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
    sh = torch.as_tensor(s_o, device="cuda")
    tn = torch.as_tensor(w.tenant, device="cuda")
    acc = lv.TenantAcc(ctx, w.n_tenants)
    h = w.n_req // 3
    lv.lv_tenant_accumulate(ctx, acc, sh[:h], tn[:h])
    state = acc.export()
    acc2 = lv.TenantAcc(ctx, w.n_tenants)
    acc2.import_(state)
    for a in (acc, acc2):
        lv.lv_tenant_accumulate(ctx, a, sh[h:], tn[h:])
    L1 = torch.empty(w.n_tenants, dtype=torch.float64, device="cuda")
    L2 = torch.empty_like(L1)
    lv.lv_tenant_totals(ctx, acc, L1)
    lv.lv_tenant_totals(ctx, acc2, L2)
    assert ctx.status() == lv.LV_OK
    l1, l2 = L1.cpu().numpy(), L2.cpu().numpy()
    assert np.array_equal(l1, l2)
    for u in range(w.n_tenants):
        assert l1[u] == exact_tenant_total(s_o[w.tenant == u])
        assert abs(l1[u] - math.fsum(s_o[w.tenant == u])) <= 1e-15 * l1[u]
    acc.reset()
    lv.lv_tenant_totals(ctx, acc, L1)
    assert float(L1.abs().max()) == 0.0


def test_tenant_accumulate_cold_tenants(lv, ctx):
    """3,000 tenants: ids from 512 up do not fit the per-CTA shared-memory table and go
    through the global 64-bit limb counters; totals within 1e-12 of the oracle and equal
    to the exact sums (each share on the 2^-72 s grid), across two calls."""
    import torch
    rng = np.random.default_rng(31)
    w = workloads.config(0, scale=0.2)
    nt = 3000
    ten = rng.integers(0, nt, w.n_req).astype(np.int32)
    ten[:4000] = rng.integers(2990, nt, 4000)      # a few tenants hot among the cold ids
    _, s_o = oracle.attribute(w.offsets, w.p, w.c, w.phase, w.split, w.coef)
    sh = torch.as_tensor(s_o, device="cuda")
    tn = torch.as_tensor(ten, device="cuda")
    acc = lv.TenantAcc(ctx, nt)
    h = w.n_req // 2
    lv.lv_tenant_accumulate(ctx, acc, sh[:h], tn[:h])
    lv.lv_tenant_accumulate(ctx, acc, sh[h:], tn[h:])
    L = torch.empty(nt, dtype=torch.float64, device="cuda")
    lv.lv_tenant_totals(ctx, acc, L)
    assert ctx.status() == lv.LV_OK
    Lg = L.cpu().numpy()
    L_o = oracle.tenant_totals(s_o, ten, nt)
    m = L_o != 0
    assert np.all(Lg[~m] == 0)
    assert np.max(np.abs(Lg[m] - L_o[m]) / np.abs(L_o[m])) <= TOL
    order = np.argsort(ten, kind="stable")
    bounds = np.searchsorted(ten[order], np.arange(nt + 1))
    for u in list(range(0, 8)) + list(range(500, 530)) + list(range(2980, nt)):
        assert Lg[u] == exact_tenant_total(s_o[order[bounds[u]:bounds[u + 1]]]), u


# ------------------------------------------------------------------ errors

def test_data_errors_flagged_not_faulting(lv, ctx):
    import torch
    rng = np.random.default_rng(2)
    w = _from_sizes(rng, rng.integers(1, 50, 500), nt=4)
    w.tenant[5] = 17          # out of range
    T, share, L, st = _run(lv, ctx, w)
    assert st == lv.LV_EDATA
    w = _from_sizes(rng, rng.integers(1, 50, 500), nt=4)
    w.p[3] = -5
    _, _, _, st = _run(lv, ctx, w)
    assert st == lv.LV_EDATA
    w = _from_sizes(rng, rng.integers(1, 50, 500), nt=4)
    w.offsets[100] = w.offsets[102] + 3   # non-monotone
    _, _, _, st = _run(lv, ctx, w)
    assert st == lv.LV_EDATA
    assert ctx.status() == lv.LV_OK     # status is cleared once read


def test_misaligned_and_bad_arguments(lv, ctx):
    import torch
    w = workloads.config(0, scale=0.01)
    b = _dev(lv, w)
    model = lv.make_model(w.coef, w.split)
    share = torch.empty(w.n_req + 1, dtype=torch.float64, device="cuda")
    bad = lv.Batches(p=b.p[1:], c=b.c[1:], phase=b.phase[1:], offsets=b.offsets, tenant=None)
    with pytest.raises(lv.LVError) as e:
        lv.lv_attribute(ctx, model, bad, None, share, None)
    assert e.value.status == lv.LV_EINVAL
    nanm = lv.make_model(np.full((4, 5), np.nan), w.split)
    with pytest.raises(lv.LVError):
        lv.lv_attribute(ctx, nanm, b, None, share, None)


# ------------------------------------------------------------------ full-size workloads

@pytest.mark.parametrize("k", [1, 4])
def test_full_size_parity(lv, ctx, k):
    """The benchmark workloads at full size, every output element against the oracle."""
    w = workloads.config(k)
    T, share, L, st = _run(lv, ctx, w)
    assert st == lv.LV_OK
    _check_parity(w, T, share, L)


def test_chunked_calls_equal_one_call(lv, ctx):
    """Batch ranges submitted one call at a time (rebased offsets, views into the same arrays,
    one tenant accumulator) give the one-call T, shares and tenant totals bit for bit: every
    sum is exact, so the split cannot change a result."""
    import torch
    w = workloads.config(1, scale=0.005)
    b = _dev(lv, w)
    model = lv.make_model(w.coef, w.split)
    outs = []
    for k in (1, 5):
        T = torch.full((w.n_batch,), float("nan"), dtype=torch.float64, device="cuda")
        S = torch.full((w.n_req,), float("nan"), dtype=torch.float64, device="cuda")
        acc = lv.TenantAcc(ctx, w.n_tenants)
        cuts = [0]
        for j in range(1, k):
            c = w.n_batch * j // k
            while w.offsets[c] % 4:
                c += 1
            cuts.append(c)
        cuts.append(w.n_batch)
        for b0, b1 in zip(cuts[:-1], cuts[1:]):
            lo, hi = int(w.offsets[b0]), int(w.offsets[b1])
            off = torch.as_tensor(w.offsets[b0:b1 + 1] - w.offsets[b0], device="cuda")
            bj = lv.Batches(p=b.p[lo:hi], c=b.c[lo:hi], phase=b.phase[lo:hi], offsets=off, tenant=b.tenant[lo:hi],
                            n_tenants=w.n_tenants)
            lv.lv_attribute(ctx, model, bj, T[b0:b1], S[lo:hi], acc)
        L = torch.empty(w.n_tenants, dtype=torch.float64, device="cuda")
        lv.lv_tenant_totals(ctx, acc, L)
        assert ctx.status() == lv.LV_OK
        outs.append((T.cpu().numpy(), S.cpu().numpy(), L.cpu().numpy()))
    for x, y in zip(*outs):
        assert np.array_equal(x.view(np.int64), y.view(np.int64))
    _check_parity(w, *outs[1])
