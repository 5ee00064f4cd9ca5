"""Pins for the fp64 ResNet-50 oracle: paper figures (Tables 2-3), torch
float64 library routines, and the Eq. 7 identities. CPU only."""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as Fnn

from oracle import resnet as orn
from oracle.counts import counting
from oracle.vit import widen, widen_all
from paper_2609_10018_gb300 import synth

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_figures.json")))
CFG = synth.RESNET50
SMALL_IMG = 64   # spatial size for the fast identity tests (7x7 stem still has room)


def _rel(a, b):
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300))


@pytest.fixture(scope="module")
def weights():
    return synth.make_resnet_weights(CFG)


@pytest.fixture(scope="module")
def wide(weights):
    return widen_all(weights)


def _small_images(n, seed=3):
    cfg = synth.dataclasses.replace(CFG, img=SMALL_IMG)
    return synth.make_images(cfg, n, seed=seed)


def test_resnet50_cost_matches_table2(wide):
    """MACs the oracle executes for one 224x224 image of the full network,
    convolutions plus classifier: 4.089 G vs the paper's 4.12 G (Table 2)."""
    img = synth.make_images(CFG, 1)
    t = synth.make_resnet_tables(CFG)[0]
    with counting() as c:
        orn.resnet_forward_sliced(wide, CFG, t["a"], t["b"], img)
    total = c["conv"] + c["fc"]
    assert total == 4_089_184_256
    assert abs(total / 1e9 - GOLDEN["resnet50_gflops"]["value"]) / GOLDEN["resnet50_gflops"]["value"] < 0.01


def test_resnet50_params_match_table3():
    shapes = synth.resnet_weight_shapes(CFG)
    n = sum(int(np.prod(s)) for s in shapes.values())
    learnable = sum(int(np.prod(s)) for k, s in shapes.items() if not k.endswith((".mean", ".var")))
    assert learnable == 25_557_032           # conv + BN affine + fc
    mib = n * 4 / 2**20
    assert abs(mib - GOLDEN["resnet50_params_mb"]["value"]) / GOLDEN["resnet50_params_mb"]["value"] < 5e-3


def _torch_resnet_dense(w, cfg, images):
    T = {k: torch.from_numpy(np.ascontiguousarray(v)) for k, v in w.items()}

    def bn(x, name):
        return Fnn.batch_norm(x, T[name + ".mean"], T[name + ".var"], T[name + ".g"], T[name + ".b"],
                              training=False, eps=1e-5)

    x = torch.from_numpy(widen(images)).permute(0, 3, 1, 2)
    x = Fnn.max_pool2d(Fnn.relu(bn(Fnn.conv2d(x, T["stem_w"], stride=2, padding=3), "stem_bn")), 3, 2, 1)
    for i, (_, _, s, proj) in enumerate(orn.block_list(cfg)):
        p = f"b{i}."
        y = Fnn.relu(bn(Fnn.conv2d(x, T[p + "conv1_w"]), p + "bn1"))
        y = Fnn.relu(bn(Fnn.conv2d(y, T[p + "conv2_w"], stride=s, padding=1), p + "bn2"))
        y = bn(Fnn.conv2d(y, T[p + "conv3_w"]), p + "bn3")
        sc = bn(Fnn.conv2d(x, T[p + "down_w"], stride=s), p + "down_bn") if proj else x
        x = Fnn.relu(y + sc)
    return Fnn.linear(Fnn.adaptive_avg_pool2d(x, 1).flatten(1), T["fc_w"], T["fc_b"]).numpy()


def test_dense_matches_torch_library(wide):
    img = _small_images(2)
    assert _rel(orn.resnet_forward_dense(wide, CFG, img), _torch_resnet_dense(wide, CFG, img)) < 1e-10


def test_full_mode_equals_base_model(wide):
    img = _small_images(2)
    t = synth.make_resnet_tables(CFG)[0]
    assert _rel(orn.resnet_forward_sliced(wide, CFG, t["a"], t["b"], img),
                orn.resnet_forward_dense(wide, CFG, img)) < 1e-12


def test_zero_masking_equals_slicing(wide):
    """Eq. 7 (channel masks multiplied into full conv kernels) == slicing."""
    img = _small_images(2)
    base = orn.resnet_forward_dense(wide, CFG, img)
    for t in synth.make_resnet_tables(CFG)[1:]:
        sliced = orn.resnet_forward_sliced(wide, CFG, t["a"], t["b"], img)
        masked = orn.resnet_forward_dense(orn.resnet_masked_weights(wide, CFG, t["a"], t["b"]), CFG, img)
        assert _rel(sliced, masked) < 1e-12
        assert _rel(sliced, base) > 1e-3


def test_folded_bn_equals_explicit_bn(wide):
    img = _small_images(2)
    t = synth.make_resnet_tables(CFG)[2]
    assert _rel(orn.resnet_forward_folded(wide, CFG, t["a"], t["b"], img),
                orn.resnet_forward_sliced(wide, CFG, t["a"], t["b"], img)) < 1e-12


def test_conv_and_pool_against_torch():
    rng = np.random.default_rng(9)
    x = rng.standard_normal((2, 11, 13, 5))
    W = rng.standard_normal((7, 5, 3, 3))
    for stride, pad in ((1, 1), (2, 1), (2, 0)):
        ref = Fnn.conv2d(torch.from_numpy(x).permute(0, 3, 1, 2), torch.from_numpy(W), stride=stride,
                         padding=pad).permute(0, 2, 3, 1).numpy()
        assert _rel(orn.conv2d(x, W, stride, pad), ref) < 1e-13
    ref = Fnn.max_pool2d(torch.from_numpy(x).permute(0, 3, 1, 2), 3, 2, 1).permute(0, 2, 3, 1).numpy()
    assert np.array_equal(orn.max_pool_3x3_s2(x), ref)


def test_tables_nested():
    modes = synth.make_resnet_tables(CFG)
    blocks = orn.block_list(CFG)
    for m, t in enumerate(modes):
        for i, (_, wdt, _, _) in enumerate(blocks):
            for key in ("a", "b"):
                s = t[key][i]
                assert len(s) == int(round(wdt * CFG.mode_frac[m])) and np.all(np.diff(s) > 0)
                if m > 0:
                    assert set(s) <= set(modes[m - 1][key][i])
