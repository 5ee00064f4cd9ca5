"""fp64 CPU oracle for the Elastoformer descendant-network (DN) forward pass.

TEST INFRASTRUCTURE ONLY. Only the tests, the package's smoke check and the
benchmark's CPU-baseline leg may import this package. The CUDA library never
calls it, and it shares no code with the CUDA path: it reads the same seeded
input arrays (weights, kept-index tables, images) and nothing else.

Everything here is a plain, slow, readable definition in float64:
- `vit`    : patch embedding, pre-norm transformer blocks with multi-head
             attention restricted to the kept heads (Eq. 2-4) and the MLP
             restricted to the kept hidden channels (Eq. 5-6), the class-token
             head; plus the dense base model, the zero-masked model, naive
             attention, and the per-mode index gather ("packing") that defines
             the packed weight layout.
- `resnet` : ResNet-50 v1.5 bottleneck network with per-block kept inner
             channels (Eq. 7), explicit (unfolded) batch norm, its masked and
             dense companions, and the BN-folded packed weights.
- `counts` : multiply-accumulate counting of what the forward passes compute.
- `select` : runtime DN selection over a profiled look-up table (Eq. 10).
- `saliency`: the Compress stage's L1-norm saliency (Section 4.1) and the
             kept tables it induces.

Inputs in bf16 are uint16 bit patterns and are widened exactly to float64;
the oracle never rounds after that.

Pinning: see the tests under `tests/test_oracle_*.py` and `tests/test_select_dn.py`, `tests/test_saliency.py` (paper figures from
Tables 1-3, library special cases via torch float64, closed forms, identities
of the method). Parity of the DN outputs against trained weights is unpinned:
no trained weights or datasets exist here.
"""
