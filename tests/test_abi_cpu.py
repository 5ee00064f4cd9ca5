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
    assert lib.elasto_check_guards(None, None, None) == binding.ERR_INVALID_ARG
    assert lib.elasto_debug_damage_guard(None, 0) == binding.ERR_INVALID_ARG
    assert lib.elasto_set_one_launch(None, 1) == binding.ERR_INVALID_ARG
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
    (lambda t: t[1].__setitem__("embed", np.array([3, 2, 9], np.int32)), binding.ERR_BAD_TABLE),     # embed unsorted
    (lambda t: t[1].__setitem__("embed", np.array([0, 192], np.int32)), binding.ERR_BAD_TABLE),      # embed >= dim
    (lambda t: t[1].__setitem__("embed", np.arange(193, dtype=np.int32) % 192), binding.ERR_BAD_TABLE),  # > dim
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


def _resnet_args(tables=None, **desc_kw):
    import dataclasses
    cfg = dataclasses.replace(synth.RESNET50, img=32, classes=10)
    keep = binding._Keep()
    w = synth.make_resnet_weights(cfg)
    desc = binding.resnet_desc(cfg, 4)
    for k, v in desc_kw.items():
        setattr(desc, k, v)
    tables = tables if tables is not None else synth.make_resnet_tables(cfg)
    mt = binding.resnet_mode_tables(keep, tables)
    ws = binding.weights_struct(keep, [w[k] for k in synth.resnet_weight_names(cfg)])
    return keep, desc, ws, mt, len(tables)


@pytest.mark.parametrize("mutate", [
    lambda t: t[2]["a"].__setitem__(0, np.array([3, 1], np.int32)),            # unsorted
    lambda t: t[2]["b"].__setitem__(5, np.array([0, 0], np.int32)),            # duplicate
    lambda t: t[2]["a"].__setitem__(15, np.array([0, 512], np.int32)),         # out of range (width 512)
    lambda t: t[2]["b"].__setitem__(1, np.zeros(0, np.int32)),                 # empty kept set
    lambda t: t[2]["a"].__setitem__(0, np.arange(65, dtype=np.int32)),         # more than the width
])
def test_resnet_bad_tables_rejected_before_cuda(lib, mutate):
    import dataclasses
    tables = synth.make_resnet_tables(dataclasses.replace(synth.RESNET50, img=32, classes=10))
    mutate(tables)
    keep, desc, ws, mt, n = _resnet_args(tables)
    assert _create(lib, desc, ws, mt, n) == binding.ERR_BAD_TABLE
    assert "mode 2" in binding.elasto_last_error()


@pytest.mark.parametrize("field, value", [("img_c", 4), ("img_h", 16), ("classes", 0)])
def test_resnet_bad_descriptor_rejected(lib, field, value):
    keep, desc, ws, mt, n = _resnet_args(**{field: value})
    assert _create(lib, desc, ws, mt, n) == binding.ERR_INVALID_ARG


def test_resnet_tensor_count_is_267(lib):
    keep, desc, ws, mt, n = _resnet_args()
    assert ws.n_tensors == 267
    ws.n_tensors = 266
    assert _create(lib, desc, ws, mt, n) == binding.ERR_INVALID_ARG
    assert "267" in binding.elasto_last_error()


def test_oracle_pool_matches_direct_call():
    """The spawn pool used by the ResNet parity tests returns the oracle's own
    logits (two 32x32 images, one per worker)."""
    import dataclasses
    from oracle import resnet as orr
    from oracle.vit import widen_all
    from oracle_pool import resnet_logits
    cfg = dataclasses.replace(synth.RESNET50, img=32, classes=10)
    tables = synth.make_resnet_tables(cfg)
    img = synth.make_images(cfg, 2)
    got = resnet_logits(cfg, tables, 1, img, chunk=1)
    ref = orr.resnet_forward_sliced(widen_all(synth.make_resnet_weights(cfg)), cfg, tables[1]["a"], tables[1]["b"], img)
    # equal up to the BLAS summation order (one thread per worker here)
    assert np.max(np.abs(got - ref)) <= 1e-12 * np.max(np.abs(ref))
