"""Runtime DN selection (Section 4.4, Eq. 10): the oracle restatement pinned by
hand-checked cases and invariants, then the C-ABI's elasto_select_dn (host
only, no GPU) against the oracle on random look-up tables."""
import math

import numpy as np
import pytest

from oracle.select import select_dn
from paper_2609_10018_gb300 import binding

NAN = float("nan")

# A look-up table shaped like the paper's: bigger DNs cost more FLOPs, take
# longer, need more memory and are more accurate.
LUT = [
    {"latency_ms": 5.1, "memory_bytes": 330e6, "gflops": 35.1, "accuracy": 81.0},   # full
    {"latency_ms": 3.9, "memory_bytes": 250e6, "gflops": 26.4, "accuracy": 79.5},
    {"latency_ms": 2.8, "memory_bytes": 170e6, "gflops": 17.7, "accuracy": 76.0},
    {"latency_ms": 2.0, "memory_bytes": 115e6, "gflops": 11.9, "accuracy": 70.2},
    {"latency_ms": 1.7, "memory_bytes": 88e6, "gflops": 9.0, "accuracy": 64.0},     # core network
]


def test_oracle_hand_checked_cases():
    assert select_dn(LUT, NAN, NAN, NAN) == 4                 # no constraint: the cheapest DN
    assert select_dn(LUT, NAN, NAN, 75.0) == 2                # accuracy floor: cheapest DN above it
    assert select_dn(LUT, NAN, NAN, 80.0) == 0
    assert select_dn(LUT, 3.0, NAN, 75.0) == 2                # latency allows 2, 3, 4; accuracy 0, 1, 2
    assert select_dn(LUT, 2.5, NAN, 75.0) is None              # nothing is both fast and accurate enough
    assert select_dn(LUT, NAN, 200e6, 70.0) == 3
    assert select_dn(LUT, NAN, 80e6, NAN) is None              # even the core network does not fit
    assert select_dn(LUT, 1.7, 88e6, 64.0) == 4                # bounds are inclusive


def test_oracle_tie_rules_and_unknown_accuracy():
    tied = [{"latency_ms": 2.0, "memory_bytes": 1.0, "gflops": 5.0, "accuracy": 1.0},
            {"latency_ms": 1.0, "memory_bytes": 1.0, "gflops": 5.0, "accuracy": 1.0},
            {"latency_ms": 1.0, "memory_bytes": 1.0, "gflops": 5.0, "accuracy": 1.0}]
    assert select_dn(tied, NAN, NAN, NAN) == 1                 # equal FLOPs: lower latency, then lower index
    unknown = [dict(e, accuracy=NAN) for e in LUT]
    assert select_dn(unknown, NAN, NAN, NAN) == 4              # no floor given: accuracy not needed
    assert select_dn(unknown, NAN, NAN, 0.0) is None           # a floor cannot be met by an unknown


def test_oracle_relaxing_a_budget_never_raises_the_cost():
    rng = np.random.default_rng(0)
    for _ in range(200):
        lut = _random_lut(rng, 6)
        lat = float(rng.uniform(0, 10))
        a = select_dn(lut, lat, NAN, NAN)
        b = select_dn(lut, lat + float(rng.uniform(0, 5)), NAN, NAN)
        if a is not None:
            assert b is not None and lut[b]["gflops"] <= lut[a]["gflops"]


def _random_lut(rng, n):
    lut = []
    for _ in range(n):
        acc = float(rng.uniform(50, 90)) if rng.random() > 0.2 else NAN
        lut.append({"latency_ms": float(rng.integers(1, 8)), "memory_bytes": float(rng.integers(1, 6)) * 1e8,
                    "gflops": float(rng.integers(1, 6)), "accuracy": acc})
    return lut


def test_c_abi_matches_oracle_on_random_tables():
    rng = np.random.default_rng(1)
    for _ in range(500):
        n = int(rng.integers(1, 8))
        lut = _random_lut(rng, n)
        bounds = [NAN if rng.random() < 0.3 else float(rng.uniform(0, 9)),
                  NAN if rng.random() < 0.3 else float(rng.uniform(0, 6e8)),
                  NAN if rng.random() < 0.3 else float(rng.uniform(40, 95))]
        # the C-ABI compares in float for latency / accuracy; keep the bounds exactly representable
        bounds = [b if math.isnan(b) else float(np.float32(b)) for b in bounds]
        assert binding.elasto_select_dn(lut, *bounds) == select_dn(lut, *bounds)


def test_c_abi_rejects_empty_table():
    with pytest.raises(binding.ElastoError):
        binding.elasto_select_dn([], NAN, NAN, NAN)
