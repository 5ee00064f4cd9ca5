"""Pins for embedding-width pruning in the fp64 oracle (Section 4.1: the
compress stage also shrinks the hidden size of the LayerNorm and patch
embedding layers). CPU only.

The oracle deletes the pruned channels (`slice_embedding`); the pins check it
against an independent masked formulation, the identity case, permutation
equivariance of the channel axis, an exact MAC scaling law and the paper's
Level-1 costs (Table 1)."""
import json
import os

import numpy as np

from oracle import vit as ov
from oracle.counts import counting
from paper_2609_10018_gb300 import synth

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_figures.json")))

SMALL = synth.vit_small_variant(synth.TINY, name="small_e", img=32, patch=8, dim=256, heads=4,
                                mlp=1024, layers=3, classes=16, dtype=synth.BF16,
                                mode_heads=(4, 3, 1), mode_mlp=(1024, 512, 128))


def _rel(a, b):
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300))


def _setup(seed=0):
    cfg = SMALL
    w = ov.widen_all(synth.make_vit_weights(cfg, seed=seed))
    t = synth.make_vit_tables(cfg)[1]
    img = synth.make_images(cfg, 3, seed=seed + 1)
    rng = np.random.default_rng(seed + 2)
    E = np.sort(rng.choice(cfg.dim, size=157, replace=False))
    return cfg, w, t, img, E


def _masked_ln(x, g, b, m):
    cnt = m.sum()
    mu = (x * m).sum(-1, keepdims=True) / cnt
    var = (((x - mu) * m) ** 2).sum(-1, keepdims=True) / cnt
    return ((x - mu) / np.sqrt(var + ov.LN_EPS) * g + b) * m


def _forward_masked(w, cfg, heads, mlp, E, images):
    """The DN as masks on the full-width model: the residual stream keeps all
    d channels with the pruned ones held at zero (embedding mask M_E on the
    patch embedding, W^O and W2 outputs), and every LayerNorm takes its
    statistics over the kept channels only."""
    d, h = cfg.dim, cfg.heads
    di = d // h
    m = np.zeros(d)
    m[E] = 1.0
    P = cfg.patch
    B, H, W, C = images.shape
    x = ov.widen(images).reshape(B, H // P, P, W // P, P, C).transpose(0, 1, 3, 5, 2, 4)
    x = x.reshape(B, -1, C * P * P)
    t = x @ w["patch_w"].reshape(d, -1).T + w["patch_b"]
    X = np.concatenate([np.broadcast_to(w["cls"], (B, 1, d)), t], axis=1) + w["pos"]
    X = X * m
    for l in range(cfg.layers):
        p = f"l{l}."
        Y = _masked_ln(X, w[p + "ln1_w"], w[p + "ln1_b"], m)
        outs = []
        for j in heads[l]:
            r = slice(j * di, (j + 1) * di)
            q = Y @ w[p + "qkv_w"][r].T + w[p + "qkv_b"][r]
            k = Y @ w[p + "qkv_w"][d:][r].T + w[p + "qkv_b"][d:][r]
            v = Y @ w[p + "qkv_w"][2 * d:][r].T + w[p + "qkv_b"][2 * d:][r]
            s = q @ k.transpose(0, 2, 1) / np.sqrt(di)
            s = np.exp(s - s.max(-1, keepdims=True))
            outs.append((s / s.sum(-1, keepdims=True)) @ v)
        cols = np.concatenate([np.arange(j * di, (j + 1) * di) for j in heads[l]])
        X = X + (np.concatenate(outs, -1) @ w[p + "proj_w"][:, cols].T + w[p + "proj_b"]) * m
        Y2 = _masked_ln(X, w[p + "ln2_w"], w[p + "ln2_b"], m)
        F = np.asarray(mlp[l])
        Hd = ov.gelu(Y2 @ w[p + "fc1_w"][F].T + w[p + "fc1_b"][F])
        X = X + (Hd @ w[p + "fc2_w"][:, F].T + w[p + "fc2_b"]) * m
    c = _masked_ln(X[:, 0], w["norm_w"], w["norm_b"], m)
    return c @ w["head_w"].T + w["head_b"]


def test_all_channels_kept_is_the_unpruned_dn_bit_for_bit():
    cfg, w, t, img, _ = _setup()
    a = ov.vit_forward_sliced(w, cfg, t["heads"], t["mlp"], img)
    b = ov.vit_forward_sliced(w, cfg, t["heads"], t["mlp"], img, embed_kept=np.arange(cfg.dim))
    assert np.array_equal(a, b)


def test_deletion_equals_masked_full_width_model():
    cfg, w, t, img, E = _setup()
    got = ov.vit_forward_sliced(w, cfg, t["heads"], t["mlp"], img, embed_kept=E)
    ref = _forward_masked(w, cfg, t["heads"], t["mlp"], E, img)
    assert _rel(got, ref) < 1e-12
    # and pruning changes the result (the pin is not vacuous)
    assert _rel(ov.vit_forward_sliced(w, cfg, t["heads"], t["mlp"], img), ref) > 1e-3


def test_permuting_the_embedding_channels_leaves_the_logits_unchanged():
    """Relabel the d channels by a permutation in every weight that carries
    them; the DN keeping the relabelled set computes the same function."""
    cfg, w, t, img, E = _setup(seed=3)
    perm = np.random.default_rng(9).permutation(cfg.dim)   # old channel c -> new index perm[c]
    inv = np.argsort(perm)
    wp = dict(w)
    wp["patch_w"] = w["patch_w"][inv]
    for k in ("patch_b", "cls", "norm_w", "norm_b"):
        wp[k] = w[k][inv]
    wp["pos"] = w["pos"][:, inv]
    wp["head_w"] = w["head_w"][:, inv]
    for l in range(cfg.layers):
        p = f"l{l}."
        for k in ("ln1_w", "ln1_b", "ln2_w", "ln2_b", "proj_b", "fc2_b"):
            wp[p + k] = w[p + k][inv]
        wp[p + "qkv_w"] = w[p + "qkv_w"][:, inv]
        wp[p + "fc1_w"] = w[p + "fc1_w"][:, inv]
        wp[p + "proj_w"] = w[p + "proj_w"][inv]
        wp[p + "fc2_w"] = w[p + "fc2_w"][inv]
    a = ov.vit_forward_sliced(w, cfg, t["heads"], t["mlp"], img, embed_kept=E)
    b = ov.vit_forward_sliced(wp, cfg, t["heads"], t["mlp"], img, embed_kept=np.sort(perm[E]))
    assert _rel(b, a) < 1e-12


def _uniform_tables(cfg, r):
    dm, hm, fm = round(r * cfg.dim), round(r * cfg.heads), round(r * cfg.mlp)
    heads = [np.arange(hm, dtype=np.int32)] * cfg.layers
    mlp = [np.arange(fm, dtype=np.int32)] * cfg.layers
    return heads, mlp, np.arange(dm, dtype=np.int32)


def test_linear_macs_scale_with_the_square_of_the_width():
    """Halving d, the heads and the MLP width in every layer divides the
    MACs of the qkv, proj, fc1 and fc2 products by exactly four (both of their
    dimensions shrink); patch and head products shrink by two (one does)."""
    cfg = synth.VIT_S
    w = ov.widen_all(synth.make_vit_weights(cfg))
    img = synth.make_images(cfg, 1)
    counts = []
    for r in (1.0, 0.5):
        heads, mlp, E = _uniform_tables(cfg, r)
        with counting() as c:
            ov.vit_forward_sliced(w, cfg, heads, mlp, img, embed_kept=E)
        counts.append(c)
    full, half = counts
    for tag in ("qkv", "proj", "fc1", "fc2"):
        assert 4 * half[tag] == full[tag], tag
    for tag in ("patch", "head"):
        assert 2 * half[tag] == full[tag], tag
    assert 2 * half["attn"] == full["attn"]


def test_level1_costs_near_table1():
    """A uniform DN keeping the fraction 1 - CR of d, of the heads and of the
    MLP channels costs about what Table 1 prints for its Level-1 network
    (the paper does not give its exact widths: within 12 %)."""
    cfg = synth.VIT_B
    w = ov.widen_all(synth.make_vit_weights(cfg))
    img = synth.make_images(cfg, 1)
    g = GOLDEN["vit_b_level1_gflops"]
    for cr, ref in zip(g["cr"], g["value"]):
        heads, mlp, E = _uniform_tables(cfg, 1.0 - cr)
        with counting() as c:
            ov.vit_forward_sliced(w, cfg, heads, mlp, img, embed_kept=E)
        linear = sum(v for k, v in c.items() if k != "attn") / 1e9
        assert abs(linear - ref) / ref < 0.12, (cr, linear, ref)
