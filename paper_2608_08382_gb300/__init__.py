"""Python binding of the LLMVisor GB300 attribution library (``include/llmvisor.h``).

Argument marshalling only: every computation runs in the CUDA kernels of
``csrc/``.  Functions keep the C names (``lv_attribute``, ``lv_fit``, ...) and take
``torch`` CUDA tensors, passing their device pointers and the current CUDA stream.
There is no CPU fallback: importing this module fails loudly when the shared
library has not been built (``__graft_entry__.build()`` or
``python paper_2608_08382_gb300/build.py``).
"""

from __future__ import annotations

import ctypes
import dataclasses
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "_build", "libllmvisor.so")

LV_OK, LV_EINVAL, LV_EOVERFLOW, LV_ENODATA, LV_ESINGULAR, LV_ECUDA, LV_EDATA, LV_ENOMEM, LV_ETIMEOUT = (
    0, -1, -2, -3, -4, -5, -6, -7, -8)
LV_ARITH_AUTO, LV_ARITH_FP64 = 0, 1
LV_TIME_TILES, LV_TIME_PAIRS = 1, 2
LV_STEP_RESET = 1

EXPORTED = [
    "lv_status_string", "lv_arch_constants", "lv_ctx_create", "lv_ctx_destroy", "lv_ctx_set_arith", "lv_ctx_status",
    "lv_ctx_set_timing", "lv_ctx_kernel_time", "lv_ctx_selftest_barrier",
    "lv_features", "lv_batch_latency", "lv_attribute", "lv_attribute_f32", "lv_attribute_step",
    "lv_tenant_acc_create", "lv_tenant_acc_destroy",
    "lv_tenant_acc_reset", "lv_tenant_accumulate", "lv_tenant_totals", "lv_tenant_acc_state_bytes",
    "lv_tenant_acc_export", "lv_tenant_acc_import", "lv_fit", "lv_fit_vtc", "lv_accuracy", "lv_whatif",
    "lv_whatif_admit", "lv_attribute_noalloc",
]


class LVError(RuntimeError):
    def __init__(self, status: int, where: str = ""):
        self.status = int(status)
        super().__init__(f"{where}: {lv_status_string(status)} ({status})")


class lv_arch(ctypes.Structure):
    _fields_ = [(n, ctypes.c_int32) for n in ("n_layers", "d_model", "n_q_heads", "n_kv_heads", "head_dim",
                                              "ffn_dim", "weight_bytes", "kv_bytes", "tp")]


class lv_coef(ctypes.Structure):
    _fields_ = [(n, ctypes.c_double) for n in ("beta", "a1", "a2", "a3", "a4")]


class lv_model(ctypes.Structure):
    _fields_ = [("seg", (lv_coef * 2) * 2), ("split", ctypes.c_int64 * 2)]


class lv_batches(ctypes.Structure):
    _fields_ = [("p", ctypes.c_void_p), ("c", ctypes.c_void_p), ("phase", ctypes.c_void_p),
                ("tenant", ctypes.c_void_p), ("offsets", ctypes.c_void_p), ("n_req", ctypes.c_int64),
                ("n_batch", ctypes.c_int64), ("n_tenants", ctypes.c_int32), ("reserved", ctypes.c_int32)]


class lv_fit_report(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int64 * 4), ("status", ctypes.c_int32 * 4), ("dropped", ctypes.c_int32 * 4),
                ("ssr", ctypes.c_double * 4), ("r2", ctypes.c_double * 4)]


class lv_accuracy_report(ctypes.Structure):
    _fields_ = [("n", ctypes.c_int64), ("r2_ssr", ctypes.c_double), ("r2_corr", ctypes.c_double),
                ("mean_rel", ctypes.c_double), ("p50", ctypes.c_double), ("p90", ctypes.c_double),
                ("p99", ctypes.c_double)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError(f"LLMVisor CUDA library not built: {LIB_PATH} is missing "
                          "(run __graft_entry__.build() or python paper_2608_08382_gb300/build.py)")
    L = ctypes.CDLL(LIB_PATH)
    P, I32, I64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
    sig = {
        "lv_status_string": ([I32], ctypes.c_char_p),
        "lv_arch_constants": ([P, P, P], I32),
        "lv_ctx_create": ([P], I32),
        "lv_ctx_destroy": ([P], None),
        "lv_ctx_set_arith": ([P, I32], I32),
        "lv_ctx_status": ([P, P], I32),
        "lv_ctx_set_timing": ([P, I32], I32),
        "lv_ctx_kernel_time": ([P, P, P], I32),
        "lv_ctx_selftest_barrier": ([P, P], I32),
        "lv_features": ([P, P, P, P, P, P, P, P], I32),
        "lv_batch_latency": ([P, P, P, P, I64, P, P], I32),
        "lv_attribute": ([P, P, P, P, P, P, P], I32),
        "lv_attribute_f32": ([P, P, P, P, P, P, P], I32),
        "lv_attribute_step": ([P, P, P, P, P, P, P, I32, P], I32),
        "lv_tenant_acc_create": ([P, I32, P], I32),
        "lv_tenant_acc_destroy": ([P], None),
        "lv_tenant_acc_reset": ([P, P], I32),
        "lv_tenant_accumulate": ([P, P, P, P, I64, P], I32),
        "lv_tenant_totals": ([P, P, P, P], I32),
        "lv_tenant_acc_state_bytes": ([P], I64),
        "lv_tenant_acc_export": ([P, P, I64, P], I32),
        "lv_tenant_acc_import": ([P, P, I64, P], I32),
        "lv_fit": ([P, P, P, I32, P, P, P], I32),
        "lv_fit_vtc": ([P, P, P, I32, P, P, P, P], I32),
        "lv_accuracy": ([P, P, P, I64, P, P], I32),
        "lv_whatif": ([P, P, P, P, P, P, I64, P, P, P], I32),
        "lv_whatif_admit": ([P, P, P, P, P, P, P, I64, P, P, I32, ctypes.c_double, P, P, P, P], I32),
        "lv_attribute_noalloc": ([P, P, P, P, P, P], I32),
    }
    for name, (args, res) in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = res
    return L


_lib = _load()


def lib():
    return _lib


def lv_status_string(status: int) -> str:
    return _lib.lv_status_string(int(status)).decode()


def _check(status, where):
    if status != LV_OK:
        raise LVError(status, where)


def _ptr(t):
    if t is None:
        return None
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream))


# ------------------------------------------------------------------ structs

def make_arch(arch) -> lv_arch:
    a = [int(v) for v in arch]
    return lv_arch(*a)


def make_model(coef, split) -> lv_model:
    """coef: (4, 5) array [phase*2 + regime][beta, a1, a2, a3, a4]; split: (2,) ints."""
    coef = np.asarray(coef, dtype=np.float64).reshape(4, 5)
    m = lv_model()
    for s in range(4):
        k = m.seg[s >> 1][s & 1]
        k.beta, k.a1, k.a2, k.a3, k.a4 = (float(v) for v in coef[s])
    m.split[0], m.split[1] = int(split[0]), int(split[1])
    return m


def model_coef(m: lv_model) -> np.ndarray:
    out = np.zeros((4, 5))
    for s in range(4):
        k = m.seg[s >> 1][s & 1]
        out[s] = (k.beta, k.a1, k.a2, k.a3, k.a4)
    return out


@dataclasses.dataclass
class Batches:
    """Device tensors of a batch set: int32 p, c, phase, tenant (or None), int64 offsets."""
    p: object
    c: object
    phase: object
    offsets: object
    tenant: object = None
    n_tenants: int = 0

    def struct(self) -> lv_batches:
        b = lv_batches()
        b.p, b.c, b.phase = _ptr(self.p), _ptr(self.c), _ptr(self.phase)
        b.tenant = _ptr(self.tenant)
        b.offsets = _ptr(self.offsets)
        b.n_req = int(self.p.numel())
        b.n_batch = int(self.offsets.numel()) - 1
        b.n_tenants = int(self.n_tenants)
        return b

    @property
    def n_req(self):
        return int(self.p.numel())

    @property
    def n_batch(self):
        return int(self.offsets.numel()) - 1


def batches_to_device(p, c, phase, offsets, tenant=None, n_tenants=0, device="cuda"):
    import torch
    def t(a, dt):
        return torch.as_tensor(np.ascontiguousarray(a), dtype=dt).to(device)
    return Batches(p=t(p, torch.int32), c=t(c, torch.int32), phase=t(phase, torch.int32),
                   offsets=t(offsets, torch.int64), tenant=None if tenant is None else t(tenant, torch.int32),
                   n_tenants=int(n_tenants))


# ------------------------------------------------------------------ context

class Context:
    def __init__(self):
        h = ctypes.c_void_p()
        _check(_lib.lv_ctx_create(ctypes.byref(h)), "lv_ctx_create")
        self.h = h

    def set_arith(self, mode: int):
        _check(_lib.lv_ctx_set_arith(self.h, int(mode)), "lv_ctx_set_arith")

    def set_timing(self, mask):
        """mask: LV_TIME_TILES | LV_TIME_PAIRS, or 0 (True selects LV_TIME_TILES)."""
        _check(_lib.lv_ctx_set_timing(self.h, int(mask)), "lv_ctx_set_timing")

    def kernel_time(self):
        """(milliseconds, launches) of the timed kernels since the previous query."""
        ms, n = ctypes.c_double(), ctypes.c_int64()
        _check(_lib.lv_ctx_kernel_time(self.h, ctypes.byref(ms), ctypes.byref(n)), "lv_ctx_kernel_time")
        return float(ms.value), int(n.value)

    def selftest_barrier(self, stream=None) -> int:
        """Status of the grid-barrier self-test: LV_ETIMEOUT when the bounded wait works."""
        return int(_lib.lv_ctx_selftest_barrier(self.h, _stream(stream)))

    def status(self, stream=None) -> int:
        return int(_lib.lv_ctx_status(self.h, _stream(stream)))

    def close(self):
        if self.h:
            _lib.lv_ctx_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def lv_arch_constants(arch):
    a = make_arch(arch)
    phi = (ctypes.c_int64 * 3)()
    w = ctypes.c_int64()
    _check(_lib.lv_arch_constants(ctypes.byref(a), phi, ctypes.byref(w)), "lv_arch_constants")
    return np.array(list(phi), dtype=np.int64), int(w.value)


def lv_features(ctx: Context, b: Batches, arch=None, model: lv_model | None = None, req_feat=None, batch_feat=None,
                batch_seg=None, stream=None):
    a = make_arch(arch) if arch is not None else None
    bs = b.struct()
    _check(_lib.lv_features(ctx.h, ctypes.byref(a) if a is not None else None,
                            ctypes.byref(model) if model is not None else None, ctypes.byref(bs), _ptr(req_feat),
                            _ptr(batch_feat), _ptr(batch_seg), _stream(stream)), "lv_features")


def lv_batch_latency(ctx: Context, model: lv_model, batch_feat, batch_seg, T, stream=None):
    n = int(T.numel())
    _check(_lib.lv_batch_latency(ctx.h, ctypes.byref(model), _ptr(batch_feat), _ptr(batch_seg), n, _ptr(T),
                                 _stream(stream)), "lv_batch_latency")


def lv_attribute(ctx: Context, model: lv_model, b: Batches, T=None, share=None, acc: "TenantAcc | None" = None,
                 stream=None):
    bs = b.struct()
    _check(_lib.lv_attribute(ctx.h, ctypes.byref(model), ctypes.byref(bs), _ptr(T), _ptr(share),
                             acc.h if acc is not None else None, _stream(stream)), "lv_attribute")


def lv_attribute_step(ctx: Context, model: lv_model, b: Batches, T=None, share=None, acc: "TenantAcc | None" = None,
                      L=None, reset: bool = False, stream=None):
    """One serving step: lv_attribute, then (with acc) the tenant totals into L; reset starts acc from zero."""
    bs = b.struct()
    _check(_lib.lv_attribute_step(ctx.h, ctypes.byref(model), ctypes.byref(bs), _ptr(T), _ptr(share),
                                  acc.h if acc is not None else None, _ptr(L), LV_STEP_RESET if reset else 0,
                                  _stream(stream)), "lv_attribute_step")


def lv_attribute_f32(ctx: Context, model: lv_model, b: "Batches", T=None, share=None, acc: "TenantAcc | None" = None,
                     stream=None):
    bs = b.struct()
    _check(_lib.lv_attribute_f32(ctx.h, ctypes.byref(model), ctypes.byref(bs), _ptr(T), _ptr(share),
                                 acc.h if acc is not None else None, _stream(stream)), "lv_attribute_f32")


class TenantAcc:
    def __init__(self, ctx: Context, n_tenants: int):
        h = ctypes.c_void_p()
        _check(_lib.lv_tenant_acc_create(ctx.h, int(n_tenants), ctypes.byref(h)), "lv_tenant_acc_create")
        self.h, self.ctx, self.n_tenants = h, ctx, int(n_tenants)

    def reset(self, stream=None):
        _check(_lib.lv_tenant_acc_reset(self.h, _stream(stream)), "lv_tenant_acc_reset")

    def state_bytes(self) -> int:
        return int(_lib.lv_tenant_acc_state_bytes(self.h))

    def export(self, stream=None) -> bytes:
        n = self.state_bytes()
        buf = ctypes.create_string_buffer(n)
        _check(_lib.lv_tenant_acc_export(self.h, buf, n, _stream(stream)), "lv_tenant_acc_export")
        return buf.raw

    def import_(self, state: bytes, stream=None):
        buf = ctypes.create_string_buffer(bytes(state), len(state))
        _check(_lib.lv_tenant_acc_import(self.h, buf, len(state), _stream(stream)), "lv_tenant_acc_import")

    def close(self):
        if self.h:
            _lib.lv_tenant_acc_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def lv_tenant_accumulate(ctx: Context, acc: TenantAcc, share, tenant, stream=None):
    _check(_lib.lv_tenant_accumulate(ctx.h, acc.h, _ptr(share), _ptr(tenant), int(share.numel()), _stream(stream)),
           "lv_tenant_accumulate")


def lv_tenant_totals(ctx: Context, acc: TenantAcc, L, stream=None):
    _check(_lib.lv_tenant_totals(ctx.h, acc.h, _ptr(L), _stream(stream)), "lv_tenant_totals")


def lv_fit(ctx: Context, b: Batches, y, models: list, stream=None):
    """y: device float64 tensor [n_y, n_batch]; models: list of lv_model (split read, coefficients written).
    Returns a list of report dicts."""
    n_y = len(models)
    arr = (lv_model * n_y)(*models)
    reps = (lv_fit_report * n_y)()
    bs = b.struct()
    _check(_lib.lv_fit(ctx.h, ctypes.byref(bs), _ptr(y), n_y, arr, reps, _stream(stream)), "lv_fit")
    out = []
    for k in range(n_y):
        models[k] = arr[k]
        r = reps[k]
        out.append(dict(n=list(r.n), status=list(r.status), dropped=list(r.dropped), ssr=list(r.ssr),
                        r2=list(r.r2)))
    return out


def lv_fit_vtc(ctx: Context, b: Batches, y, stream=None):
    """y: device float64 tensor [n_y, n_batch].  Returns a list of (beta, a, status, count), one per y vector."""
    n_y = int(y.shape[0])
    coef = (ctypes.c_double * (2 * n_y))()
    st = (ctypes.c_int32 * n_y)()
    cnt = (ctypes.c_int64 * n_y)()
    bs = b.struct()
    _check(_lib.lv_fit_vtc(ctx.h, ctypes.byref(bs), _ptr(y), n_y, coef, st, cnt, _stream(stream)), "lv_fit_vtc")
    nan = float("nan")
    return [(coef[2 * k] if st[k] == 0 else nan, coef[2 * k + 1] if st[k] == 0 else nan, st[k], cnt[k])
            for k in range(n_y)]


def lv_accuracy(ctx: Context, y, T, stream=None) -> dict:
    """Accuracy of predictions T against measurements y (device float64 tensors of one length)."""
    r = lv_accuracy_report()
    _check(_lib.lv_accuracy(ctx.h, _ptr(y), _ptr(T), int(y.numel()), ctypes.byref(r), _stream(stream)),
           "lv_accuracy")
    return dict(n=r.n, r2_ssr=r.r2_ssr, r2_corr=r.r2_corr, mean_rel=r.mean_rel, p50=r.p50, p90=r.p90, p99=r.p99)


def lv_whatif(ctx: Context, model: lv_model, cand: Batches, p_new, c_new, phase_new, T_new=None, share_new=None,
              stream=None):
    bs = cand.struct()
    _check(_lib.lv_whatif(ctx.h, ctypes.byref(model), ctypes.byref(bs), _ptr(p_new), _ptr(c_new), _ptr(phase_new),
                          int(p_new.numel()), _ptr(T_new), _ptr(share_new), _stream(stream)), "lv_whatif")


def lv_whatif_admit(ctx: Context, model: lv_model, cand: Batches, p_new, c_new, phase_new, tenant_new, L, budget,
                    slo: float, admit, T_new=None, share_new=None, stream=None):
    bs = cand.struct()
    _check(_lib.lv_whatif_admit(ctx.h, ctypes.byref(model), ctypes.byref(bs), _ptr(p_new), _ptr(c_new),
                                _ptr(phase_new), _ptr(tenant_new), int(p_new.numel()), _ptr(L), _ptr(budget),
                                int(L.numel()), float(slo), _ptr(T_new), _ptr(share_new), _ptr(admit),
                                _stream(stream)), "lv_whatif_admit")
