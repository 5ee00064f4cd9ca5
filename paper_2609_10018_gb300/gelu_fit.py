"""Coefficients of the GELU used by the fused FC1 epilogue (csrc/gemm.cu).

The MLP activation of the ViT is the exact GELU, x * Phi(x) (Section 3.1's
MLP block, as in the base ViT). The epilogue evaluates it in the logistic form

    GELU(x) ~= x * sigma(2 u(x)),   u(x) = x (a0 + a1 s + a2 s^2),  s = min(x^2, 36)

which is the tanh approximation of Hendrycks & Gimpel (2016),
x * (1 + tanh(u)) / 2 with u = sqrt(2/pi) (x + 0.044715 x^3), rewritten through
(1 + tanh u) / 2 = sigma(2u) and with one more odd term. The coefficients below
are refitted here to minimise the maximum absolute error on [0, 8]
(Lawson's iteratively reweighted least squares followed by a Nelder-Mead
polish). The error is an even function of x because both the exact and the
approximate GELU satisfy g(-x) = g(x) - x, so [0, 8] covers [-8, 8]; beyond,
the clamp of s keeps u increasing and the logistic saturates. Maximum absolute
error 2.52e-5 (the Hendrycks-Gimpel coefficients give 4.7e-4).

Run as a script to refit and print the coefficients; nothing imports this
module at run time.
"""
import numpy as np

A0, A1, A2 = 0.7975078842851289, 0.0370056460225075, -0.00035151678856300587
S_CLAMP = 36.0
MAX_ABS_ERR = 2.52e-5


def gelu_logistic(x, a=(A0, A1, A2)):
    """The approximation above, in fp64."""
    x = np.asarray(x, dtype=np.float64)
    s = np.minimum(x * x, S_CLAMP)
    u = x * ((a[2] * s + a[1]) * s + a[0])
    return x / (1.0 + np.exp(-2.0 * u))


def fit(lo=0.0, hi=8.0, points=160001, iters=200):
    from scipy.optimize import minimize
    from scipy.special import erf

    x = np.linspace(lo, hi, points)
    g = 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))
    c0 = np.sqrt(2.0 / np.pi)
    p = np.array([c0, c0 * 0.044715, 0.0])
    w = np.full_like(x, 1.0 / x.size)
    for _ in range(iters):  # Lawson: weights grow where the error is largest
        e = gelu_logistic(x, p) - g
        jac = np.stack([(gelu_logistic(x, p + d) - gelu_logistic(x, p - d)) / 2e-7 for d in np.eye(3) * 1e-7], 1)
        sw = np.sqrt(w)
        step, *_ = np.linalg.lstsq(jac * sw[:, None], -e * sw, rcond=None)
        p = p + step
        w = np.maximum(w * np.abs(gelu_logistic(x, p) - g), 1e-300)
        w /= w.sum()
    res = minimize(lambda q: np.abs(gelu_logistic(x, q) - g).max(), p, method="Nelder-Mead",
                   options={"xatol": 1e-14, "fatol": 1e-14, "maxiter": 40000})
    return res.x, float(np.abs(gelu_logistic(x, res.x) - g).max())


if __name__ == "__main__":
    coeffs, err = fit()
    print("a0, a1, a2 =", ", ".join(repr(float(c)) for c in coeffs), " max |error| =", err)
