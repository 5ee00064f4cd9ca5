"""The FC1 epilogue's GELU (csrc/act.cuh, used by csrc/gemm.cu and
csrc/persistent.cu) against the exact x * Phi(x) of the oracle, on the CPU:
the three constants are read from the kernel source and the same formula is
evaluated in fp64, so a wrong sign, a dropped term or a mistyped digit in the
kernel shows up here without a GPU."""
import math
import pathlib
import re

import numpy as np

from oracle import vit as ov
from paper_2609_10018_gb300 import gelu_fit

SRC = pathlib.Path(__file__).resolve().parents[1] / "paper_2609_10018_gb300" / "csrc" / "act.cuh"


def _kernel_constants():
    text = SRC.read_text()
    body = text[text.index("float gelu(float x)"):]
    body = body[:body.index("\n}\n")]
    vals = dict(re.findall(r"constexpr float (kB\d) = (-?[0-9.eE+-]+)f;", body))
    assert sorted(vals) == ["kB0", "kB1", "kB2"], vals
    clamp = re.search(r"fminf\(x \* x, ([0-9.]+)f\)", body)
    assert clamp, "clamp of x^2 not found"
    return [np.float32(float(vals[k])) for k in ("kB0", "kB1", "kB2")], float(clamp.group(1))


def _kernel_gelu_f64(x):
    (b0, b1, b2), clamp = _kernel_constants()
    s = np.minimum(x * x, clamp)
    v = x * ((float(b2) * s + float(b1)) * s + float(b0))
    with np.errstate(over="ignore"):
        return x / (1.0 + np.exp2(v))


def test_constants_are_the_fitted_ones():
    (b0, b1, b2), clamp = _kernel_constants()
    k = -2.0 * math.log2(math.e)
    for b, a in zip((b0, b1, b2), (gelu_fit.A0, gelu_fit.A1, gelu_fit.A2)):
        assert b == np.float32(k * a)
    assert clamp == gelu_fit.S_CLAMP


def test_error_bound_over_the_real_line():
    x = np.concatenate([np.linspace(-12.0, 12.0, 480001), [-1e4, -300.0, -88.0, 88.0, 300.0, 1e4]])
    err = np.abs(_kernel_gelu_f64(x) - ov.gelu(x))
    assert float(err.max()) <= gelu_fit.MAX_ABS_ERR * 1.01, float(err.max())
    # the bound is tight (a refit that loosened it would show here)
    assert float(err.max()) >= gelu_fit.MAX_ABS_ERR * 0.9


def test_special_values():
    assert _kernel_gelu_f64(np.zeros(1))[0] == 0.0
    x = np.linspace(0.0, 10.0, 1001)
    # g(x) - g(-x) = x holds for the logistic form exactly, as for the exact GELU
    assert np.allclose(_kernel_gelu_f64(x) - _kernel_gelu_f64(-x), x, atol=1e-12)
    # saturation: GELU(x) -> x for large x, -> 0 for large -x
    assert abs(_kernel_gelu_f64(np.array([60.0]))[0] - 60.0) < 1e-12
    assert abs(_kernel_gelu_f64(np.array([-60.0]))[0]) < 1e-12


def test_fit_script_reproduces_constants():
    coeffs, err = gelu_fit.fit(points=20001, iters=60)
    assert err <= gelu_fit.MAX_ABS_ERR * 1.05
    assert np.allclose(coeffs, [gelu_fit.A0, gelu_fit.A1, gelu_fit.A2], rtol=2e-3)
