"""Seeded synthetic workloads: model dimensions, weights, kept-index tables, images.

This module only draws numbers. It holds none of the method's arithmetic (no
forward pass, no gather, no folding); both the fp64 oracle and the CUDA path
consume what it returns, so a mistake here cannot make the two agree by
accident.

Workloads stand in for the paper's ImageNet-1K (224x224, 1000 classes) and
CIFAR-10 (32x32, 10 classes) inputs (Section 5.1): only their shapes are used.
Weights are random, not trained, so no accuracy claim follows from them.

Conventions shared with the C-ABI (canonical tensor order, PyTorch layouts):

ViT (pre-norm, class token, learned position embedding, Section 4.1 / 5.2):
    patch_w [d, C, P, P], patch_b [d], cls [d], pos [n, d],
    per layer: ln1_w, ln1_b, qkv_w [3d, d], qkv_b [3d], proj_w [d, d], proj_b [d],
               ln2_w, ln2_b, fc1_w [f, d], fc1_b [f], fc2_w [d, f], fc2_b [d],
    norm_w, norm_b, head_w [C, d], head_b [C].
    qkv_w rows are three blocks (q | k | v), each ordered head-major (row j*64+r
    of a block is channel r of head j).

ResNet-50 v1.5 (bottlenecks [3,4,6,3], stride on the 3x3 conv):
    stem_w [64, 3, 7, 7], stem BN (gamma, beta, mean, var),
    per block: conv1_w [w, cin, 1, 1], bn1 x4, conv2_w [w, w, 3, 3], bn2 x4,
               conv3_w [4w, w, 1, 1], bn3 x4, and on the first block of a stage
               down_w [4w, cin, 1, 1], down BN x4,
    fc_w [1000, 2048], fc_b [1000].

bf16 tensors are returned as uint16 bit patterns (numpy has no bf16 type),
rounded from an fp32 draw to nearest-even.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Tuple

import numpy as np

# ----------------------------------------------------------------------------
# Model dimensions
# ----------------------------------------------------------------------------

F32, BF16 = 0, 1


@dataclasses.dataclass(frozen=True)
class VitConfig:
    name: str
    img: int
    chans: int
    patch: int
    dim: int
    heads: int
    mlp: int
    layers: int
    classes: int
    dtype: int                      # F32 or BF16: storage of weights and images
    mode_heads: Tuple[int, ...]     # kept heads per layer, one entry per mode (mode 0 = full)
    mode_mlp: Tuple[int, ...]       # kept MLP hidden channels per layer, per mode
    batch: int
    seeds: Tuple[int, int, int]     # weights / tables / images

    @property
    def n_patches(self) -> int:
        return (self.img // self.patch) ** 2

    @property
    def tokens(self) -> int:
        return self.n_patches + 1

    @property
    def head_dim(self) -> int:
        return self.dim // self.heads

    @property
    def n_modes(self) -> int:
        return len(self.mode_heads)


@dataclasses.dataclass(frozen=True)
class ResnetConfig:
    name: str
    img: int
    chans: int
    classes: int
    dtype: int
    blocks: Tuple[int, int, int, int]
    widths: Tuple[int, int, int, int]
    mode_frac: Tuple[float, ...]    # kept fraction of each block's two inner widths, per mode
    batch: int
    seeds: Tuple[int, int, int]

    @property
    def n_modes(self) -> int:
        return len(self.mode_frac)


TINY = VitConfig("tiny", img=32, chans=3, patch=4, dim=192, heads=3, mlp=768, layers=6,
                 classes=10, dtype=F32, mode_heads=(3, 2), mode_mlp=(768, 384), batch=8,
                 seeds=(0, 1, 2))
VIT_S = VitConfig("vit_s16", img=224, chans=3, patch=16, dim=384, heads=6, mlp=1536, layers=12,
                  classes=1000, dtype=BF16, mode_heads=(6, 4, 3, 2),
                  mode_mlp=(1536, 1152, 768, 384), batch=64, seeds=(10, 11, 12))
# 33 % of 3072 is not an integer; 1024 (= 1/3, a multiple of 128) is used.
VIT_B = VitConfig("vit_b16", img=224, chans=3, patch=16, dim=768, heads=12, mlp=3072, layers=12,
                  classes=1000, dtype=BF16, mode_heads=(12, 9, 6, 4, 3),
                  mode_mlp=(3072, 2304, 1536, 1024, 768), batch=256, seeds=(20, 21, 22))
RESNET50 = ResnetConfig("resnet50", img=224, chans=3, classes=1000, dtype=BF16,
                        blocks=(3, 4, 6, 3), widths=(64, 128, 256, 512),
                        mode_frac=(1.0, 0.75, 0.5, 0.25), batch=128, seeds=(30, 31, 32))

VIT_CONFIGS = {c.name: c for c in (TINY, VIT_S, VIT_B)}


def vit_small_variant(base: VitConfig, **kw) -> VitConfig:
    """A copy of `base` with some fields replaced (smaller test shapes)."""
    return dataclasses.replace(base, **kw)


# ----------------------------------------------------------------------------
# Number formats (storage only)
# ----------------------------------------------------------------------------

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """fp32 -> bf16 bit patterns, round to nearest even (finite inputs)."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounded = u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return (rounded >> np.uint32(16)).astype(np.uint16)


def _store(x32: np.ndarray, dtype: int) -> np.ndarray:
    return f32_to_bf16_bits(x32) if dtype == BF16 else np.ascontiguousarray(x32, np.float32)


# ----------------------------------------------------------------------------
# ViT
# ----------------------------------------------------------------------------

def vit_weight_names(cfg: VitConfig) -> List[str]:
    names = ["patch_w", "patch_b", "cls", "pos"]
    for l in range(cfg.layers):
        names += [f"l{l}.{s}" for s in ("ln1_w", "ln1_b", "qkv_w", "qkv_b", "proj_w", "proj_b",
                                          "ln2_w", "ln2_b", "fc1_w", "fc1_b", "fc2_w", "fc2_b")]
    names += ["norm_w", "norm_b", "head_w", "head_b"]
    return names


def vit_weight_shapes(cfg: VitConfig) -> Dict[str, Tuple[int, ...]]:
    d, f, P, C = cfg.dim, cfg.mlp, cfg.patch, cfg.chans
    shapes = {"patch_w": (d, C, P, P), "patch_b": (d,), "cls": (d,), "pos": (cfg.tokens, d),
              "norm_w": (d,), "norm_b": (d,), "head_w": (cfg.classes, d), "head_b": (cfg.classes,)}
    for l in range(cfg.layers):
        shapes.update({f"l{l}.ln1_w": (d,), f"l{l}.ln1_b": (d,), f"l{l}.qkv_w": (3 * d, d),
                       f"l{l}.qkv_b": (3 * d,), f"l{l}.proj_w": (d, d), f"l{l}.proj_b": (d,),
                       f"l{l}.ln2_w": (d,), f"l{l}.ln2_b": (d,), f"l{l}.fc1_w": (f, d),
                       f"l{l}.fc1_b": (f,), f"l{l}.fc2_w": (d, f), f"l{l}.fc2_b": (d,)})
    return shapes


def make_vit_weights(cfg: VitConfig, seed: int | None = None) -> Dict[str, np.ndarray]:
    """All tensors ~ N(0, 0.02); LayerNorm gains 1 + N(0, 0.02). Stored in cfg.dtype."""
    rng = np.random.default_rng(cfg.seeds[0] if seed is None else seed)
    shapes = vit_weight_shapes(cfg)
    out = {}
    for name in vit_weight_names(cfg):
        x = rng.standard_normal(shapes[name], dtype=np.float32) * np.float32(0.02)
        if name.endswith("ln1_w") or name.endswith("ln2_w") or name == "norm_w":
            x = x + np.float32(1.0)
        out[name] = _store(x, cfg.dtype)
    return out


def make_vit_tables(cfg: VitConfig, seed: int | None = None,
                    nested: bool = True) -> List[Dict[str, List[np.ndarray]]]:
    """Per mode, per layer: sorted int32 kept head indices and kept MLP channels.

    Nested (Eq. 8: every larger DN contains the smaller one): one seeded
    permutation per layer; mode m keeps the sorted first k_m entries.
    With nested=False each mode draws its own subsets (the ABI accepts both).
    """
    base = cfg.seeds[1] if seed is None else seed
    modes = [{"heads": [], "mlp": []} for _ in range(cfg.n_modes)]
    for l in range(cfg.layers):
        rng = np.random.default_rng([base, l])
        ph, pf = rng.permutation(cfg.heads), rng.permutation(cfg.mlp)
        for m in range(cfg.n_modes):
            if not nested:
                ph, pf = rng.permutation(cfg.heads), rng.permutation(cfg.mlp)
            modes[m]["heads"].append(np.sort(ph[:cfg.mode_heads[m]]).astype(np.int32))
            modes[m]["mlp"].append(np.sort(pf[:cfg.mode_mlp[m]]).astype(np.int32))
    return modes


def with_embedding(cfg: VitConfig, tables, widths, seed: int | None = None):
    """Copies of the mode tables that also prune the embedding width: mode m
    keeps widths[m] of the d channels (None: all), nested across the modes
    (one seeded permutation, each mode the sorted first widths[m] entries)."""
    rng = np.random.default_rng([cfg.seeds[1] if seed is None else seed, 1_000_003])
    perm = rng.permutation(cfg.dim)
    out = []
    for t, k in zip(tables, widths):
        t = dict(t)
        t["embed"] = None if k is None else np.sort(perm[:k]).astype(np.int32)
        out.append(t)
    return out


def make_images(cfg, batch: int, seed: int | None = None) -> np.ndarray:
    """[B, H, W, C] pixels U[0, 1) (no normalisation), stored in cfg.dtype."""
    rng = np.random.default_rng(cfg.seeds[2] if seed is None else seed)
    x = rng.random((batch, cfg.img, cfg.img, cfg.chans), dtype=np.float32)
    return _store(x, cfg.dtype)


# ----------------------------------------------------------------------------
# ResNet-50
# ----------------------------------------------------------------------------

def resnet_blocks(cfg: ResnetConfig) -> List[Tuple[int, int, int, bool]]:
    """(cin, width, stride, has_downsample) per bottleneck block, in order."""
    out, cin = [], 64
    for s, (nb, w) in enumerate(zip(cfg.blocks, cfg.widths)):
        for b in range(nb):
            stride = 2 if (b == 0 and s > 0) else 1
            out.append((cin, w, stride, b == 0))
            cin = 4 * w
    return out


def resnet_weight_names(cfg: ResnetConfig) -> List[str]:
    bn = ("g", "b", "mean", "var")
    names = ["stem_w"] + [f"stem_bn.{s}" for s in bn]
    for i, (_, _, _, down) in enumerate(resnet_blocks(cfg)):
        for c in ("1", "2", "3"):
            names += [f"b{i}.conv{c}_w"] + [f"b{i}.bn{c}.{s}" for s in bn]
        if down:
            names += [f"b{i}.down_w"] + [f"b{i}.down_bn.{s}" for s in bn]
    return names + ["fc_w", "fc_b"]


def resnet_weight_shapes(cfg: ResnetConfig) -> Dict[str, Tuple[int, ...]]:
    shapes = {"stem_w": (64, cfg.chans, 7, 7), "fc_w": (cfg.classes, 4 * cfg.widths[-1]),
              "fc_b": (cfg.classes,)}
    for s in ("g", "b", "mean", "var"):
        shapes[f"stem_bn.{s}"] = (64,)
    for i, (cin, w, _, down) in enumerate(resnet_blocks(cfg)):
        shapes[f"b{i}.conv1_w"] = (w, cin, 1, 1)
        shapes[f"b{i}.conv2_w"] = (w, w, 3, 3)
        shapes[f"b{i}.conv3_w"] = (4 * w, w, 1, 1)
        for s in ("g", "b", "mean", "var"):
            shapes[f"b{i}.bn1.{s}"] = (w,)
            shapes[f"b{i}.bn2.{s}"] = (w,)
            shapes[f"b{i}.bn3.{s}"] = (4 * w,)
        if down:
            shapes[f"b{i}.down_w"] = (4 * w, cin, 1, 1)
            for s in ("g", "b", "mean", "var"):
                shapes[f"b{i}.down_bn.{s}"] = (4 * w,)
    return shapes


def make_resnet_weights(cfg: ResnetConfig, seed: int | None = None) -> Dict[str, np.ndarray]:
    """He-normal convs; BN gamma U(0.5, 1) (U(0.1, 0.3) on bn3, the last BN of a
    block's residual branch),
    beta N(0, 0.05), running mean N(0, 0.1), running var U(0.5, 1.5); FC N(0, 0.01)."""
    rng = np.random.default_rng(cfg.seeds[0] if seed is None else seed)
    shapes = resnet_weight_shapes(cfg)
    out = {}
    for name in resnet_weight_names(cfg):
        shp = shapes[name]
        if name.endswith("_w") and len(shp) == 4:
            fan_in = shp[1] * shp[2] * shp[3]
            x = rng.standard_normal(shp, dtype=np.float32) * np.float32(np.sqrt(2.0 / fan_in))
        elif name == "fc_w" or name == "fc_b":
            x = rng.standard_normal(shp, dtype=np.float32) * np.float32(0.01)
        elif name.endswith(".g"):
            # only the BN closing a block's residual branch is small (bounds the
            # growth of the residual sum); the shortcut projection's BN is not,
            # or four projections would shrink the image signal ~0.2^4 against
            # the constant BN shifts and every image would get the same logits
            lo, hi = (0.1, 0.3) if ".bn3." in name else (0.5, 1.0)
            x = rng.uniform(lo, hi, shp).astype(np.float32)
        elif name.endswith(".b"):
            x = rng.standard_normal(shp, dtype=np.float32) * np.float32(0.05)
        elif name.endswith(".mean"):
            x = rng.standard_normal(shp, dtype=np.float32) * np.float32(0.1)
        elif name.endswith(".var"):
            x = rng.uniform(0.5, 1.5, shp).astype(np.float32)
        else:
            raise AssertionError(name)
        out[name] = _store(x, cfg.dtype)
    return out


def make_resnet_tables(cfg: ResnetConfig, seed: int | None = None) -> List[Dict[str, List[np.ndarray]]]:
    """Per mode, per block: sorted kept inner channels S_a (conv1 out = conv2 in)
    and S_b (conv2 out = conv3 in), nested across modes (Eq. 8)."""
    base = cfg.seeds[1] if seed is None else seed
    modes = [{"a": [], "b": []} for _ in range(cfg.n_modes)]
    for i, (_, w, _, _) in enumerate(resnet_blocks(cfg)):
        rng = np.random.default_rng([base, i])
        pa, pb = rng.permutation(w), rng.permutation(w)
        for m, frac in enumerate(cfg.mode_frac):
            k = int(round(w * frac))
            modes[m]["a"].append(np.sort(pa[:k]).astype(np.int32))
            modes[m]["b"].append(np.sort(pb[:k]).astype(np.int32))
    return modes


# ----------------------------------------------------------------------------
# Mixed-mode serving stream (ViT-B weights)
# ----------------------------------------------------------------------------

def make_stream_schedule(n_requests: int, n_modes: int, seed: int = 43,
                         batch_choices=(1, 8, 32, 128), p_stay: float = 0.8):
    """Markov mode schedule (stay with p_stay, else uniform over the other modes,
    starting at mode 0) and per-request batch sizes uniform over batch_choices."""
    rng = np.random.default_rng(seed)
    modes = np.empty(n_requests, np.int32)
    m = 0
    for i in range(n_requests):
        if i > 0 and rng.random() >= p_stay:
            others = [k for k in range(n_modes) if k != m]
            m = others[int(rng.integers(len(others)))]
        modes[i] = m
    batches = np.asarray(batch_choices, np.int32)[rng.integers(len(batch_choices), size=n_requests)]
    return modes, batches
