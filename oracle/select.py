"""fp64 oracle: runtime descendant-network selection (Section 4.4, Eq. 10).

Test infrastructure only (see the package docstring).

Eq. 10: among the DNs of the profiled look-up table, choose the one with the
lowest computational cost (FLOPs) that satisfies every operational
constraint: Latency(DN) <= L_d, Memory(DN) <= M_d, Accuracy(DN) >= A_min.

Readings where the paper is silent:
  - ties in FLOPs go to the lower latency, then to the lower table index;
  - a constraint whose bound is NaN is not applied (no budget given);
  - an entry whose accuracy is unknown (NaN) does not satisfy a given A_min;
  - no feasible DN -> None.
"""
from __future__ import annotations

import math
from typing import Optional, Sequence


def select_dn(lut: Sequence[dict], max_latency_ms: float, max_memory_bytes: float,
              min_accuracy: float) -> Optional[int]:
    """lut: entries with keys latency_ms, memory_bytes, gflops, accuracy."""
    feasible = []
    for i, e in enumerate(lut):
        if not math.isnan(max_latency_ms) and not e["latency_ms"] <= max_latency_ms:
            continue
        if not math.isnan(max_memory_bytes) and not e["memory_bytes"] <= max_memory_bytes:
            continue
        if not math.isnan(min_accuracy) and not e["accuracy"] >= min_accuracy:
            continue
        feasible.append(i)
    if not feasible:
        return None
    return min(feasible, key=lambda i: (lut[i]["gflops"], lut[i]["latency_ms"], i))
