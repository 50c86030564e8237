"""The C ABI library loads and exports every symbol of include/llmvisor.h, and
host-side argument checks answer before anything touches a GPU (no GPU needed)."""

import ctypes
import os
import re

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lv():
    import importlib.util
    spec = importlib.util.spec_from_file_location("_lv_build", os.path.join(ROOT, "paper_2608_08382_gb300",
                                                                          "build.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    mod.build()
    import paper_2608_08382_gb300
    return paper_2608_08382_gb300


def _declared():
    src = open(os.path.join(ROOT, "include", "llmvisor.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(lv_[a-z_0-9]+)\s*\(", src)))


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("lv_features", "lv_batch_latency", "lv_attribute", "lv_tenant_accumulate", "lv_fit", "lv_whatif"):
        assert n in names


def test_library_exports_every_declared_symbol(lv):
    L = ctypes.CDLL(lv.LIB_PATH)
    missing = [n for n in _declared() if not hasattr(L, n)]
    assert missing == []
    assert sorted(lv.EXPORTED) == _declared()


def test_struct_layouts(lv):
    assert ctypes.sizeof(lv.lv_arch) == 36
    assert ctypes.sizeof(lv.lv_model) == 4 * 5 * 8 + 16
    assert ctypes.sizeof(lv.lv_batches) == 5 * 8 + 2 * 8 + 8
    assert ctypes.sizeof(lv.lv_fit_report) == 32 + 16 + 16 + 32 + 32
    assert ctypes.sizeof(lv.lv_accuracy_report) == 8 + 6 * 8


def test_arch_constants_host(lv, golden_dir):
    import json
    g = json.load(open(os.path.join(golden_dir, "arch_constants.json")))
    for case in g["cases"]:
        phi, W = lv.lv_arch_constants(case["arch"])
        assert phi.tolist() == case["phi"] and W == case["W"]
    with pytest.raises(lv.LVError) as e:
        lv.lv_arch_constants((32, 4096, 32, 8, 128, 14336, 2, 2, 3))
    assert e.value.status == lv.LV_EINVAL
    with pytest.raises(lv.LVError) as e:
        lv.lv_arch_constants((2**30, 2**30, 2**20, 2**20, 2**20, 2**30, 2, 2, 1))
    assert e.value.status == lv.LV_EOVERFLOW


def test_invalid_arguments_rejected_before_launch(lv):
    L = lv.lib()
    m = lv.make_model(np.ones((4, 5)), (1, 1))
    b = lv.lv_batches()
    assert L.lv_attribute(None, ctypes.byref(m), ctypes.byref(b), None, None, None, None) == lv.LV_EINVAL
    assert L.lv_ctx_set_arith(None, 0) == lv.LV_EINVAL
    assert L.lv_ctx_status(None, None) == lv.LV_EINVAL
    assert L.lv_tenant_acc_create(None, 4, ctypes.byref(ctypes.c_void_p())) == lv.LV_EINVAL
    assert L.lv_arch_constants(None, None, None) == lv.LV_EINVAL
    assert L.lv_accuracy(None, None, None, 0, None, None) == lv.LV_EINVAL
    assert L.lv_fit_vtc(None, None, None, 1, None, None, None, None) == lv.LV_EINVAL
    assert lv.lv_status_string(lv.LV_EDATA) == "invalid input data"
    assert L.lv_tenant_acc_state_bytes(None) == 0
    # lv_attribute_step: unknown flags, totals or a reset without an accumulator, a misaligned L, no context
    fake = ctypes.c_void_p(1 << 20)
    step = L.lv_attribute_step
    assert step(None, ctypes.byref(m), ctypes.byref(b), None, None, None, None, 2, None) == lv.LV_EINVAL
    assert step(None, ctypes.byref(m), ctypes.byref(b), None, None, None, fake, 0, None) == lv.LV_EINVAL
    assert step(None, ctypes.byref(m), ctypes.byref(b), None, None, None, None, lv.LV_STEP_RESET, None) == lv.LV_EINVAL
    assert step(None, ctypes.byref(m), ctypes.byref(b), None, None, fake, ctypes.c_void_p((1 << 20) + 4), 0,
                None) == lv.LV_EINVAL
    assert step(None, ctypes.byref(m), ctypes.byref(b), None, None, None, None, 0, None) == lv.LV_EINVAL
    assert L.lv_ctx_selftest_barrier(None, None) == lv.LV_EINVAL


def test_import_fails_loudly_without_library(tmp_path):
    """The binding refuses to load when the CUDA library is absent (no CPU fallback)."""
    import shutil
    import subprocess
    import sys
    pkg = tmp_path / "paper_2608_08382_gb300"
    pkg.mkdir()
    shutil.copy(os.path.join(ROOT, "paper_2608_08382_gb300", "__init__.py"), pkg / "__init__.py")
    r = subprocess.run([sys.executable, "-c", "import paper_2608_08382_gb300"], cwd=tmp_path, capture_output=True,
                       text=True)
    assert r.returncode != 0 and "not built" in r.stderr


def test_binding_constants_match_header(lv):
    src = open(os.path.join(ROOT, "include", "llmvisor.h")).read()
    defs = dict(re.findall(r"#define\s+(LV_[A-Z_0-9]+)\s+\(?(-?\d+)\)?", src))
    assert len(defs) >= 13
    for name, value in defs.items():
        assert getattr(lv, name) == int(value), name
