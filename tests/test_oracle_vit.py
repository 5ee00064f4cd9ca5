"""Pins for the fp64 ViT oracle: paper figures, a library special case, closed
forms and the method's identities. CPU only."""
import json
import os

import numpy as np
import pytest
import torch
import torch.nn.functional as Fnn

from oracle import vit as ov
from oracle.counts import counting
from paper_2609_10018_gb300 import synth

GOLDEN = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_figures.json")))

# A small ViT with the structure of the paper's models (d_i = 64) that the
# oracle finishes in well under a second.
SMALL = synth.vit_small_variant(synth.TINY, name="small", img=32, patch=8, dim=256, heads=4,
                                mlp=1024, layers=3, classes=16, dtype=synth.BF16,
                                mode_heads=(4, 3, 1), mode_mlp=(1024, 512, 128))


def _rel(a, b):
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-300))


# ---------------------------------------------------------------- paper figures

def test_vit_b_cost_matches_table1():
    """MACs the oracle executes for one image of the full ViT-B model: the
    linear layers (patch, qkv, proj, fc1, fc2, head) give the paper's base
    cost (Table 1 caption, 16.86 G) within 0.1 %; attention is counted apart."""
    cfg = synth.VIT_B
    w = ov.widen_all(synth.make_vit_weights(cfg))
    tables = synth.make_vit_tables(cfg)[0]
    img = synth.make_images(cfg, 1)
    with counting() as c:
        ov.vit_forward_sliced(w, cfg, tables["heads"], tables["mlp"], img)
    linear = sum(v for k, v in c.items() if k != "attn")
    assert linear == 12 * 197 * 768 * (3 * 768 + 768 + 2 * 3072) + 196 * 768 * 768 + 768 * 1000
    assert abs(linear / 1e9 - GOLDEN["vit_b_base_gflops"]["value"]) / GOLDEN["vit_b_base_gflops"]["value"] < 1e-3
    assert c["attn"] == 12 * 12 * 2 * 197 * 197 * 64


def test_vit_b_params_match_table3():
    shapes = synth.vit_weight_shapes(synth.VIT_B)
    n = sum(int(np.prod(s)) for s in shapes.values())
    assert n == 86_567_656
    mib = n * 4 / 2**20
    assert abs(mib - GOLDEN["vit_b_params_mb"]["value"]) / GOLDEN["vit_b_params_mb"]["value"] < 1e-3


def test_dims_match_section_5_2():
    g = GOLDEN["vit_b_dims"]
    assert (synth.VIT_B.layers, synth.VIT_B.dim, synth.VIT_B.patch) == (g["layers"], g["dim"], g["patch"])
    for cfg in synth.VIT_CONFIGS.values():
        assert cfg.mlp == GOLDEN["mlp_ratio"]["value"] * cfg.dim
        assert cfg.dim // cfg.heads == 64


# ------------------------------------------------- library special case (torch)

def _torch_vit_dense(w, cfg, images):
    """The base ViT assembled from torch's own float64 modules: conv2d patch
    embedding, nn.TransformerEncoderLayer (pre-norm, GELU), layer_norm, linear."""
    d = cfg.dim
    T = {k: torch.from_numpy(np.ascontiguousarray(v)) for k, v in w.items()}
    x = torch.from_numpy(ov.widen(images)).permute(0, 3, 1, 2)
    t = Fnn.conv2d(x, T["patch_w"], T["patch_b"], stride=cfg.patch).flatten(2).transpose(1, 2)
    B = t.shape[0]
    X = torch.cat([T["cls"].expand(B, 1, d), t], dim=1) + T["pos"]
    for l in range(cfg.layers):
        p = f"l{l}."
        layer = torch.nn.TransformerEncoderLayer(d, cfg.heads, cfg.mlp, dropout=0.0, activation="gelu",
                                                 layer_norm_eps=1e-6, batch_first=True, norm_first=True,
                                                 dtype=torch.float64)
        with torch.no_grad():
            layer.self_attn.in_proj_weight.copy_(T[p + "qkv_w"])
            layer.self_attn.in_proj_bias.copy_(T[p + "qkv_b"])
            layer.self_attn.out_proj.weight.copy_(T[p + "proj_w"])
            layer.self_attn.out_proj.bias.copy_(T[p + "proj_b"])
            layer.linear1.weight.copy_(T[p + "fc1_w"])
            layer.linear1.bias.copy_(T[p + "fc1_b"])
            layer.linear2.weight.copy_(T[p + "fc2_w"])
            layer.linear2.bias.copy_(T[p + "fc2_b"])
            layer.norm1.weight.copy_(T[p + "ln1_w"])
            layer.norm1.bias.copy_(T[p + "ln1_b"])
            layer.norm2.weight.copy_(T[p + "ln2_w"])
            layer.norm2.bias.copy_(T[p + "ln2_b"])
        layer.train()  # dropout is 0; training mode keeps torch off its fused inference path
        with torch.no_grad():
            X = layer(X)
    c = Fnn.layer_norm(X[:, 0], (d,), T["norm_w"], T["norm_b"], eps=1e-6)
    return Fnn.linear(c, T["head_w"], T["head_b"]).numpy()


@pytest.mark.parametrize("cfg", [synth.TINY, SMALL], ids=["tiny", "small"])
def test_dense_matches_torch_library(cfg):
    w = ov.widen_all(synth.make_vit_weights(cfg))
    img = synth.make_images(cfg, 3)
    ref = _torch_vit_dense(w, cfg, img)
    got = ov.vit_forward_dense(w, cfg, img)
    assert _rel(got, ref) < 1e-10


# ------------------------------------------------------------ method identities

@pytest.mark.parametrize("cfg", [synth.TINY, SMALL], ids=["tiny", "small"])
def test_full_mode_equals_base_model(cfg):
    w = ov.widen_all(synth.make_vit_weights(cfg))
    t0 = synth.make_vit_tables(cfg)[0]
    assert all(len(h) == cfg.heads for h in t0["heads"]) and all(len(f) == cfg.mlp for f in t0["mlp"])
    img = synth.make_images(cfg, 4)
    assert _rel(ov.vit_forward_sliced(w, cfg, t0["heads"], t0["mlp"], img),
                ov.vit_forward_dense(w, cfg, img)) < 1e-12


@pytest.mark.parametrize("cfg", [synth.TINY, SMALL], ids=["tiny", "small"])
def test_zero_masking_equals_slicing(cfg):
    """Eq. 4/6 (masks multiplied into full weights) == deleting the rows/cols."""
    w = ov.widen_all(synth.make_vit_weights(cfg))
    img = synth.make_images(cfg, 4)
    for t in synth.make_vit_tables(cfg)[1:]:
        masked = ov.vit_masked_weights(w, cfg, t["heads"], t["mlp"])
        a = ov.vit_forward_dense(masked, cfg, img)
        b = ov.vit_forward_sliced(w, cfg, t["heads"], t["mlp"], img)
        assert _rel(b, a) < 1e-12
        # and the mode is a genuinely different network
        assert _rel(b, ov.vit_forward_dense(w, cfg, img)) > 1e-3


def test_degenerate_layer_without_heads_or_channels():
    """A layer that keeps no head and no MLP channel adds only b^O and b2."""
    cfg = SMALL
    w = ov.widen_all(synth.make_vit_weights(cfg))
    t = synth.make_vit_tables(cfg)[1]
    heads = [h.copy() for h in t["heads"]]
    mlp = [f.copy() for f in t["mlp"]]
    heads[1] = np.zeros(0, np.int32)
    mlp[1] = np.zeros(0, np.int32)
    img = synth.make_images(cfg, 2)
    masked = ov.vit_masked_weights(w, cfg, heads, mlp)
    assert _rel(ov.vit_forward_sliced(w, cfg, heads, mlp, img), ov.vit_forward_dense(masked, cfg, img)) < 1e-12


@pytest.mark.parametrize("cfg", [synth.TINY, synth.VIT_S, synth.VIT_B], ids=lambda c: c.name)
def test_tables_nested_sorted_unique(cfg):
    """Eq. 8: the larger DN contains the smaller one (weights are only added)."""
    modes = synth.make_vit_tables(cfg)
    for m, t in enumerate(modes):
        for l in range(cfg.layers):
            h, f = t["heads"][l], t["mlp"][l]
            assert len(h) == cfg.mode_heads[m] and len(f) == cfg.mode_mlp[m]
            assert np.all(np.diff(h) > 0) and np.all(np.diff(f) > 0)
            assert h.min() >= 0 and h.max() < cfg.heads and f.min() >= 0 and f.max() < cfg.mlp
            if m > 0:
                assert set(h) <= set(modes[m - 1]["heads"][l]) and set(f) <= set(modes[m - 1]["mlp"][l])
    # kept sets vary by layer
    assert len({tuple(h) for h in modes[-1]["heads"]}) > 1


# ----------------------------------------------------------------- closed forms

def test_attention_matrix_form_equals_naive_loops():
    rng = np.random.default_rng(5)
    q, k, v = rng.standard_normal((7, 4)), rng.standard_normal((5, 4)), rng.standard_normal((5, 3))
    assert _rel(ov.attention(q, k, v, 4), ov.attention_naive(q, k, v, 4)) < 1e-13


def test_attention_special_cases():
    rng = np.random.default_rng(6)
    q = rng.standard_normal((6, 8))
    v1 = rng.standard_normal((1, 8))
    # one key: every query returns that key's value
    assert np.allclose(ov.attention(q, rng.standard_normal((1, 8)), v1, 8), np.repeat(v1, 6, 0), rtol=0, atol=1e-15)
    # identical keys: uniform weights, the mean of the values
    kk = np.repeat(rng.standard_normal((1, 8)), 5, 0)
    vv = rng.standard_normal((5, 8))
    assert np.allclose(ov.attention(q, kk, vv, 8), np.repeat(vv.mean(0, keepdims=True), 6, 0), atol=1e-14)
    # huge equal scores stay finite (max-shifted softmax)
    big = np.full((2, 8), 1e3)
    out = ov.attention(big, big, vv[:2], 8)
    assert np.all(np.isfinite(out)) and np.allclose(out, vv[:2].mean(0), atol=1e-12)


def test_attention_against_torch_sdpa():
    rng = np.random.default_rng(7)
    q, k, v = (rng.standard_normal((2, 3, 9, 64)) for _ in range(3))
    ref = Fnn.scaled_dot_product_attention(*(torch.from_numpy(a) for a in (q, k, v))).numpy()
    assert _rel(ov.attention(q, k, v, 64), ref) < 1e-13


def test_layer_norm_closed_form():
    rng = np.random.default_rng(8)
    x = rng.standard_normal((5, 384)) * 3.0 + 1.5
    y = ov.layer_norm(x, np.ones(384), np.zeros(384))
    var = x.var(axis=-1)
    assert np.allclose(y.mean(-1), 0, atol=1e-14)
    assert np.allclose(y.var(-1), var / (var + ov.LN_EPS), rtol=1e-13)


def test_gelu_closed_forms():
    x = np.linspace(-6, 6, 97)
    assert ov.gelu(np.zeros(1))[0] == 0.0
    assert np.allclose(ov.gelu(x) - ov.gelu(-x), x, atol=1e-14)
    # GELU(1) = Phi(1) = 0.841344746068542948... (standard normal CDF at 1)
    assert abs(ov.gelu(np.array([1.0]))[0] - 0.8413447460685429) < 1e-15
    assert np.allclose(ov.gelu(x), Fnn.gelu(torch.from_numpy(x)).numpy(), rtol=1e-14, atol=1e-15)


# ------------------------------------------------------------- packed layout

def test_packed_layout_runs_as_a_small_dense_vit():
    """The per-mode packed buffers, read with torch library routines as the
    weights of a narrower ViT layer (q|k|v blocks, head-major), reproduce the
    oracle's sliced layer."""
    cfg = SMALL
    stored = synth.make_vit_weights(cfg)
    w = ov.widen_all(stored)
    t = synth.make_vit_tables(cfg)[1]
    img = synth.make_images(cfg, 2)
    one = synth.vit_small_variant(cfg, layers=1)
    ref = ov.vit_forward_sliced(w, one, t["heads"][:1], t["mlp"][:1], img)

    pk = ov.vit_pack_layer(stored, cfg, 0, t["heads"][0], t["mlp"][0])
    wide = {k: torch.from_numpy(ov.widen(v)) for k, v in pk.items()}
    T = {k: torch.from_numpy(v) for k, v in w.items()}
    X = torch.from_numpy(ov.embed(w, cfg, img))
    B, n, d = X.shape
    hm = len(t["heads"][0])
    Y = Fnn.layer_norm(X, (d,), T["l0.ln1_w"], T["l0.ln1_b"], eps=1e-6)
    qkv = Fnn.linear(Y, wide["qkv_w"], wide["qkv_b"]).reshape(B, n, 3, hm, 64).permute(2, 0, 3, 1, 4)
    O = Fnn.scaled_dot_product_attention(qkv[0], qkv[1], qkv[2]).permute(0, 2, 1, 3).reshape(B, n, hm * 64)
    X = X + Fnn.linear(O, wide["proj_w"], T["l0.proj_b"])
    Y2 = Fnn.layer_norm(X, (d,), T["l0.ln2_w"], T["l0.ln2_b"], eps=1e-6)
    X = X + Fnn.linear(Fnn.gelu(Fnn.linear(Y2, wide["fc1_w"], wide["fc1_b"])), wide["fc2_w"], T["l0.fc2_b"])
    c = Fnn.layer_norm(X[:, 0], (d,), T["norm_w"], T["norm_b"], eps=1e-6)
    got = Fnn.linear(c, T["head_w"], T["head_b"]).numpy()
    assert _rel(got, ref) < 1e-12


def test_pack_rounds_fp32_to_nearest_even():
    """The packed bf16 of an fp32-stored model is the round-to-nearest-even of
    each weight: check against values whose bf16 neighbours are known."""
    vals = np.array([1.0, 1.0 + 2**-8, 1.0 + 2**-8 + 2**-20, 1.0 + 3 * 2**-8, -2.5, 1.0 + 2**-9],
                    dtype=np.float32)
    bits = ov._bf16_bits_rne(vals)
    back = (bits.astype(np.uint32) << 16).view(np.float32)
    # 1+2^-8 is a tie between 1 and 1+2^-7 -> even (1.0); slightly above rounds up;
    # 1+3*2^-8 is a tie between 1+2^-7 and 1+2^-6 -> even (1+2^-6)
    assert back.tolist() == [1.0, 1.0, 1.0 + 2**-7, 1.0 + 2**-6, -2.5, 1.0]
    assert np.array_equal(bits, torch.from_numpy(vals).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16))


# ---------------------------------------------------------------- input widening

def _bf16_by_definition(bits: int) -> float:
    """Value of a bf16 bit pattern from the format's fields: 1 sign bit, 8
    exponent bits (bias 127), 7 fraction bits; exponent 0 is subnormal
    (2^-126 * f / 128), exponent 255 is infinity (f = 0) or NaN."""
    import math
    s, e, f = bits >> 15, (bits >> 7) & 0xFF, bits & 0x7F
    sign = -1.0 if s else 1.0
    if e == 0xFF:
        return sign * math.inf if f == 0 else math.nan
    if e == 0:
        return sign * math.ldexp(f, -126 - 7)
    return sign * math.ldexp(128 + f, e - 127 - 7)


def test_widen_decodes_every_bf16_pattern():
    """oracle.vit.widen on all 65,536 bf16 bit patterns against (a) the format's
    field definition and (b) torch's own bfloat16 -> float64 conversion; NaNs
    compare as NaN, and the sign of zero is kept. A wrong shift, byte order or
    sign handling fails here."""
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    got = ov.widen(bits)
    assert got.dtype == np.float64 and got.shape == (65536,)
    by_def = np.array([_bf16_by_definition(int(b)) for b in range(65536)])
    lib = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).to(torch.float64).numpy()
    for ref in (by_def, lib):
        nan = np.isnan(ref)
        assert np.array_equal(np.isnan(got), nan)
        assert np.array_equal(got[~nan], ref[~nan])
        assert np.array_equal(np.signbit(got[~nan]), np.signbit(ref[~nan]))
    # a few patterns worked out by hand
    hand = {0x3F80: 1.0, 0x4000: 2.0, 0xC040: -3.0, 0x3F81: 1.0 + 2.0**-7, 0x0001: 2.0**-133,
            0x0080: 2.0**-126, 0x7F7F: (2.0 - 2.0**-7) * 2.0**127, 0x7F80: np.inf, 0xFF80: -np.inf,
            0x3E80: 0.25, 0xBF00: -0.5}
    for b, v in hand.items():
        assert got[b] == v, hex(b)
    assert np.isnan(got[0x7FC0]) and got[0x8000] == 0.0 and np.signbit(got[0x8000])


def test_widen_keeps_fp32_and_multidimensional_arrays_exact():
    """fp32 inputs widen to the same real number, and bf16 arrays keep their
    shape and element order (a transposed or flattened decode fails)."""
    rng = np.random.default_rng(5)
    f = rng.standard_normal((3, 5)).astype(np.float32)
    assert np.array_equal(ov.widen(f), f.astype(np.float64)) and ov.widen(f).dtype == np.float64
    b = rng.integers(0, 0x7F80, size=(4, 3, 2)).astype(np.uint16)  # finite positives
    got = ov.widen(b)
    assert got.shape == b.shape
    for idx in np.ndindex(b.shape):
        assert got[idx] == _bf16_by_definition(int(b[idx]))
