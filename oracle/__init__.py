"""CPU oracle for the LLMVisor attribution path -- TEST INFRASTRUCTURE ONLY.

Plain C loops (``lvo.c``) for features, Eq. 1, shares, tenant roll-up and
what-if, plus an exact rational least-squares fit (``fit.py``).  Only tests/,
``__graft_entry__.smoke()`` and bench.py's CPU-baseline leg may import this
package; the product library never does, and this package never imports the
product.
"""

from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

from . import fit as _fit  # noqa: F401  (re-exported)
from .fit import fit, fit_group, vtc_fit, accuracy, OK, ENODATA, ESINGULAR  # noqa: F401

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "lvo.c")
_BUILD = os.path.join(_HERE, "_build")
_SO = os.path.join(_BUILD, "liblvo.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile lvo.c into oracle/_build/liblvo.so (gcc, -O2, no FP contraction)."""
    os.makedirs(_BUILD, exist_ok=True)
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + f".tmp{os.getpid()}"
        subprocess.run(["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC", "-shared",
                        "-o", tmp, _SRC, "-lm"], check=True)
        os.replace(tmp, _SO)
    return _SO


def load(path: str):
    """Load an oracle shared library built from lvo.c (or a test's mutant of it)."""
    L = ctypes.CDLL(path)
    P = ctypes.c_void_p
    I64 = ctypes.c_int64
    L.lvo_arch_constants.argtypes = [P, P, P]
    L.lvo_request_features.argtypes = [I64, P, P, P, P]
    L.lvo_batch_features.argtypes = [I64, P, P, P, P, P, P, P]
    L.lvo_batch_latency.argtypes = [I64, P, P, P, P]
    L.lvo_attribute.argtypes = [I64, P, P, P, P, P, P, P, P]
    L.lvo_tenant_accumulate.argtypes = [I64, P, P, P, P]
    L.lvo_tenant_totals.argtypes = [ctypes.c_int32, P, P, P]
    L.lvo_whatif.argtypes = [I64, P, P, P, P, I64, P, P, P, P, P, P, P]
    for f in (L.lvo_arch_constants, L.lvo_request_features):
        f.restype = ctypes.c_int
    return L


def lib():
    global _lib
    if _lib is None:
        build()
        _lib = load(_SO)
    return _lib


class using:
    """Context manager: route this module's wrappers through another build of lvo.c."""

    def __init__(self, path: str):
        self._new = load(path)

    def __enter__(self):
        global _lib
        self._old, _lib = lib(), self._new
        return self

    def __exit__(self, *exc):
        global _lib
        _lib = self._old
        return False


def _ptr(a):
    return a.ctypes.data_as(ctypes.c_void_p) if a is not None else None


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


def arch_constants(arch):
    """(phi int64[3], W) for arch = (L, d, hq, hkv, hd, F, wb, kvb, tp); raises on error."""
    a = _c(arch, np.int32)
    phi = np.zeros(3, dtype=np.int64)
    w = np.zeros(1, dtype=np.int64)
    rc = lib().lvo_arch_constants(_ptr(a), _ptr(phi), _ptr(w))
    if rc != 0:
        raise ValueError(f"lvo_arch_constants status {rc}")
    return phi, int(w[0])


def request_features(p, c, phi):
    p, c, phi = _c(p, np.int32), _c(c, np.int32), _c(phi, np.int64)
    out = np.zeros((3, p.shape[0]), dtype=np.int64)
    rc = lib().lvo_request_features(p.shape[0], _ptr(p), _ptr(c), _ptr(phi), _ptr(out))
    if rc != 0:
        raise OverflowError("request feature overflow")
    return out


def batch_features(offsets, p, c, phase, split):
    off = _c(offsets, np.int64)
    p, c, ph, sp = _c(p, np.int32), _c(c, np.int32), _c(phase, np.int32), _c(split, np.int64)
    nb = off.shape[0] - 1
    feat = np.zeros((5, nb), dtype=np.int64)
    seg = np.zeros(nb, dtype=np.uint8)
    lib().lvo_batch_features(nb, _ptr(off), _ptr(p), _ptr(c), _ptr(ph), _ptr(sp), _ptr(feat), _ptr(seg))
    return feat, seg


def batch_latency(feat, seg, coef):
    feat, seg, coef = _c(feat, np.int64), _c(seg, np.uint8), _c(coef, np.float64)
    nb = seg.shape[0]
    T = np.zeros(nb, dtype=np.float64)
    lib().lvo_batch_latency(nb, _ptr(feat), _ptr(seg), _ptr(coef), _ptr(T))
    return T


def attribute(offsets, p, c, phase, split, coef):
    """Returns (T float64[n_batch], share float64[n_req])."""
    off = _c(offsets, np.int64)
    p, c, ph = _c(p, np.int32), _c(c, np.int32), _c(phase, np.int32)
    sp, coef = _c(split, np.int64), _c(coef, np.float64)
    nb = off.shape[0] - 1
    T = np.zeros(nb, dtype=np.float64)
    share = np.zeros(p.shape[0], dtype=np.float64)
    lib().lvo_attribute(nb, _ptr(off), _ptr(p), _ptr(c), _ptr(ph), _ptr(sp), _ptr(coef), _ptr(T), _ptr(share))
    return T, share


class TenantSums:
    """Running per-tenant Neumaier sums; ``add`` continues across calls."""

    def __init__(self, n_tenants: int):
        self.n_tenants = int(n_tenants)
        self.sum = np.zeros(self.n_tenants, dtype=np.float64)
        self.comp = np.zeros(self.n_tenants, dtype=np.float64)

    def add(self, share, tenant):
        share, tenant = _c(share, np.float64), _c(tenant, np.int32)
        lib().lvo_tenant_accumulate(share.shape[0], _ptr(share), _ptr(tenant), _ptr(self.sum), _ptr(self.comp))
        return self

    def totals(self):
        L = np.zeros(self.n_tenants, dtype=np.float64)
        lib().lvo_tenant_totals(self.n_tenants, _ptr(self.sum), _ptr(self.comp), _ptr(L))
        return L


def tenant_totals(share, tenant, n_tenants):
    return TenantSums(n_tenants).add(share, tenant).totals()


def admit(T_new, share_new, tenant_new, L, budget, slo):
    """Admission over what-if pairs (Section 1: what-if planning for admission
    control).  Pending request j may join candidate batch b when its tenant's
    running total plus its share in the merged batch stays within the tenant's
    budget, L[u_j] + share_new[j, b] <= budget[u_j] (one fp64 addition), and
    the merged batch meets the latency objective, T_new[j, b] <= slo.
    Returns uint8[n_pending, n_cand] (1 = admissible)."""
    T_new = np.asarray(T_new, dtype=np.float64)
    share_new = np.asarray(share_new, dtype=np.float64)
    u = np.asarray(tenant_new, dtype=np.int64)
    Lu = np.asarray(L, dtype=np.float64)[u][:, None]
    Bu = np.asarray(budget, dtype=np.float64)[u][:, None]
    ok = ((Lu + share_new) <= Bu) & (T_new <= float(slo))
    return ok.astype(np.uint8)


def whatif(offsets, p, c, phase, p_new, c_new, phase_new, split, coef):
    """Returns (T_new, share_new), each float64[n_pending, n_cand]."""
    off = _c(offsets, np.int64)
    p, c, ph = _c(p, np.int32), _c(c, np.int32), _c(phase, np.int32)
    pn, cn, phn = _c(p_new, np.int32), _c(c_new, np.int32), _c(phase_new, np.int32)
    sp, coef = _c(split, np.int64), _c(coef, np.float64)
    nc, npd = off.shape[0] - 1, pn.shape[0]
    T = np.zeros((npd, nc), dtype=np.float64)
    S = np.zeros((npd, nc), dtype=np.float64)
    lib().lvo_whatif(nc, _ptr(off), _ptr(p), _ptr(c), _ptr(ph), npd, _ptr(pn), _ptr(cn), _ptr(phn), _ptr(sp),
                     _ptr(coef), _ptr(T), _ptr(S))
    return T, S
