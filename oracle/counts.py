"""Multiply-accumulate accounting for the oracle's matrix products.

Test infrastructure only (see the package docstring).

Every matrix product the oracle's forward passes perform goes through `mm`,
which adds m*k*n to the counter named by its tag. Counting the products the
forward actually executes (rather than a separate formula) ties the paper's
cost figures (Table 1 caption: 16.86 G for ViT-B; Table 2: 4.12 G for
ResNet-50) to the shapes the oracle really uses.
"""
from __future__ import annotations

import contextlib
from collections import defaultdict

import numpy as np

_active: list = []


def mm(a: np.ndarray, b: np.ndarray, tag: str) -> np.ndarray:
    """a @ b over the last two axes; counts prod(batch) * m * k * n MACs."""
    out = a @ b
    if _active:
        k = a.shape[-1]
        macs = int(np.prod(out.shape, dtype=np.int64)) * int(k)
        for c in _active:
            c[tag] += macs
    return out


@contextlib.contextmanager
def counting():
    """Collect MACs by tag for the products executed inside the block."""
    c = defaultdict(int)
    _active.append(c)
    try:
        yield c
    finally:
        _active.remove(c)
