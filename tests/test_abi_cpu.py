"""The C-ABI library builds, loads, exports every declared symbol, and rejects
bad arguments on the host before touching CUDA. CPU only (no GPU calls)."""
import ctypes
import os
import re

import numpy as np
import pytest

from paper_2609_10018_gb300 import binding, synth
from paper_2609_10018_gb300 import build as builder

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    srcs = builder.sources() + [os.path.join(ROOT, "include", f) for f in os.listdir(os.path.join(ROOT, "include"))]
    stale = (not os.path.exists(binding.LIB_PATH) or
             os.path.getmtime(binding.LIB_PATH) < max(os.path.getmtime(s) for s in srcs))
    if stale:
        builder.build()
    return binding.lib()


def _declared_functions():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            text = open(os.path.join(ROOT, "include", f)).read()
            names |= set(re.findall(r"^\s*(?:elasto_status|const char\*)\s+(elasto_\w+)\s*\(", text, re.M))
    return names


def test_exports_every_declared_symbol(lib):
    names = _declared_functions()
    assert {"elasto_create", "elasto_set_mode", "elasto_forward", "elasto_destroy", "elasto_last_error",
            "elasto_debug_export_packed", "elasto_op_gemm", "elasto_op_attention"} <= names
    for n in names:
        assert hasattr(lib, n), n


def test_null_handle_calls_fail_cleanly(lib):
    assert lib.elasto_set_mode(None, 0) == binding.ERR_INVALID_ARG
    assert "null handle" in binding.elasto_last_error()
    assert lib.elasto_forward(None, None, None, 1, None) == binding.ERR_INVALID_ARG
    assert lib.elasto_destroy(None) == binding.ERR_INVALID_ARG
    v = ctypes.c_int64()
    assert lib.elasto_query(None, 0, 0, ctypes.byref(v)) == binding.ERR_INVALID_ARG


def _tiny_args(tables=None, **desc_kw):
    cfg = synth.TINY
    keep = binding._Keep()
    w = synth.make_vit_weights(cfg)
    desc = binding.vit_desc(cfg, 8)
    for k, v in desc_kw.items():
        setattr(desc, k, v)
    tables = tables if tables is not None else synth.make_vit_tables(cfg)
    mt = binding.vit_mode_tables(keep, tables)
    ws = binding.weights_struct(keep, [w[k] for k in synth.vit_weight_names(cfg)])
    return keep, desc, ws, mt, len(tables)


def _create(lib, desc, ws, mt, n):
    h = ctypes.c_void_p()
    return lib.elasto_create(ctypes.byref(desc), ctypes.byref(ws), mt, n, ctypes.byref(h))


@pytest.mark.parametrize("mutate, code", [
    (lambda t: t[1]["heads"].__setitem__(0, np.array([1, 0], np.int32)), binding.ERR_BAD_TABLE),     # unsorted
    (lambda t: t[1]["heads"].__setitem__(0, np.array([1, 1], np.int32)), binding.ERR_BAD_TABLE),     # duplicate
    (lambda t: t[1]["heads"].__setitem__(0, np.array([0, 3], np.int32)), binding.ERR_BAD_TABLE),     # out of range
    (lambda t: t[1]["mlp"].__setitem__(2, np.array([-1, 5], np.int32)), binding.ERR_BAD_TABLE),      # negative
    (lambda t: t[1]["heads"].__setitem__(0, np.arange(4, dtype=np.int32)), binding.ERR_BAD_TABLE),   # too many
])
def test_bad_tables_rejected_before_cuda(lib, mutate, code):
    tables = synth.make_vit_tables(synth.TINY)
    mutate(tables)
    keep, desc, ws, mt, n = _tiny_args(tables)
    assert _create(lib, desc, ws, mt, n) == code
    assert "mode 1" in binding.elasto_last_error()


@pytest.mark.parametrize("field, value", [("dim", 200), ("heads", 4), ("patch", 5), ("max_batch", 0),
                                          ("weight_dtype", 7), ("arch", 9), ("img_w", 16)])
def test_bad_descriptor_rejected(lib, field, value):
    keep, desc, ws, mt, n = _tiny_args(**{field: value})
    assert _create(lib, desc, ws, mt, n) in (binding.ERR_INVALID_ARG, binding.ERR_UNSUPPORTED)
    assert binding.elasto_last_error() != ""


def test_wrong_tensor_count_rejected(lib):
    keep, desc, ws, mt, n = _tiny_args()
    ws.n_tensors -= 1
    assert _create(lib, desc, ws, mt, n) == binding.ERR_INVALID_ARG
    assert "weight tensors" in binding.elasto_last_error()


def test_build_flags_target_sm103a_only():
    assert builder.ARCH == ["-gencode", "arch=compute_103a,code=sm_103a"]
