"""fp64 oracle: elastic ResNet-50 descendant-network forward pass.

Test infrastructure only (see the package docstring).

Network: ResNet-50 v1.5 in NHWC: 7x7/2 stem conv + BN + ReLU, 3x3/2 max pool
(padding 1, padded cells never win), 16 bottleneck blocks [3, 4, 6, 3] of
widths 64..512 (1x1 -> 3x3 (stride here) -> 1x1 to 4x width, each conv with
BN, ReLU after the first two and after the residual sum; a 1x1 strided
projection + BN on the first block of each stage), global average pool,
linear classifier.

Elastic descendant networks (Eq. 7): W_conv is multiplied by a 0/1 mask over
(C_out, C_in, K, K). The masks here are structured by channel: per block a
kept set S_a of conv1's output channels (= conv2's input channels) and a kept
set S_b of conv2's output channels (= conv3's input channels). Masking whole
channels to zero equals deleting them, so the DN forward is the forward of
the sliced convolutions. The stem, block outputs, projections and the
classifier are never pruned. BN eps = 1e-5.
"""
from __future__ import annotations

import numpy as np

from .counts import mm
from .vit import widen

BN_EPS = 1e-5


def conv2d(x: np.ndarray, W: np.ndarray, stride: int, pad: int) -> np.ndarray:
    """out[b, y, x, o] = sum_{ky, kx, c} xpad[b, y*s + ky, x*s + kx, c] * W[o, c, ky, kx].
    x: [B, H, W, Cin] (NHWC), W: [Cout, Cin, kh, kw] (PyTorch layout), zero padding."""
    B, H, Wd, Cin = x.shape
    Cout, _, kh, kw = W.shape
    Ho = (H + 2 * pad - kh) // stride + 1
    Wo = (Wd + 2 * pad - kw) // stride + 1
    xp = np.pad(x, ((0, 0), (pad, pad), (pad, pad), (0, 0)))
    out = np.zeros((B, Ho, Wo, Cout))
    for ky in range(kh):
        for kx in range(kw):
            tap = xp[:, ky:ky + stride * (Ho - 1) + 1:stride, kx:kx + stride * (Wo - 1) + 1:stride, :]
            out += mm(tap, W[:, :, ky, kx].T, "conv")
    return out


def batch_norm(x: np.ndarray, g, b, mean, var, eps: float = BN_EPS) -> np.ndarray:
    """Inference BN over the channel (last) axis with running statistics."""
    return (x - mean) / np.sqrt(var + eps) * g + b


def relu(x: np.ndarray) -> np.ndarray:
    return np.maximum(x, 0.0)


def max_pool_3x3_s2(x: np.ndarray) -> np.ndarray:
    """3x3 window, stride 2, padding 1 (padding cells are -inf)."""
    B, H, W, C = x.shape
    Ho, Wo = (H + 2 - 3) // 2 + 1, (W + 2 - 3) // 2 + 1
    xp = np.pad(x, ((0, 0), (1, 1), (1, 1), (0, 0)), constant_values=-np.inf)
    out = np.full((B, Ho, Wo, C), -np.inf)
    for ky in range(3):
        for kx in range(3):
            out = np.maximum(out, xp[:, ky:ky + 2 * (Ho - 1) + 1:2, kx:kx + 2 * (Wo - 1) + 1:2, :])
    return out


def _bn(w, name, x, idx=None):
    g, b, m, v = (w[f"{name}.{s}"] for s in ("g", "b", "mean", "var"))
    if idx is not None:
        g, b, m, v = g[idx], b[idx], m[idx], v[idx]
    return batch_norm(x, g, b, m, v)


def block_list(cfg):
    """(cin, width, stride, has_projection) for each bottleneck, in order."""
    out, cin = [], 64
    for s, (nb, wdt) in enumerate(zip(cfg.blocks, cfg.widths)):
        for i in range(nb):
            out.append((cin, wdt, 2 if (i == 0 and s > 0) else 1, i == 0))
            cin = 4 * wdt
    return out


def stem(w: dict, images: np.ndarray) -> np.ndarray:
    x = relu(_bn(w, "stem_bn", conv2d(widen(images), w["stem_w"], 2, 3)))
    return max_pool_3x3_s2(x)


def head(w: dict, x: np.ndarray) -> np.ndarray:
    pooled = x.mean(axis=(1, 2))
    return mm(pooled, w["fc_w"].T, "fc") + w["fc_b"]


def resnet_forward_dense(w: dict, cfg, images: np.ndarray) -> np.ndarray:
    """The unmodified base network. `w` widened to float64. Logits [B, classes]."""
    x = stem(w, images)
    for i, (_, _, stride, proj) in enumerate(block_list(cfg)):
        p = f"b{i}."
        y = relu(_bn(w, p + "bn1", conv2d(x, w[p + "conv1_w"], 1, 0)))
        y = relu(_bn(w, p + "bn2", conv2d(y, w[p + "conv2_w"], stride, 1)))
        y = _bn(w, p + "bn3", conv2d(y, w[p + "conv3_w"], 1, 0))
        sc = _bn(w, p + "down_bn", conv2d(x, w[p + "down_w"], stride, 0)) if proj else x
        x = relu(y + sc)
    return head(w, x)


def resnet_forward_sliced(w: dict, cfg, kept_a, kept_b, images: np.ndarray) -> np.ndarray:
    """DN forward: block i keeps inner channels kept_a[i] after conv1 and
    kept_b[i] after conv2 (ascending index arrays)."""
    x = stem(w, images)
    for i, (_, _, stride, proj) in enumerate(block_list(cfg)):
        p = f"b{i}."
        A = np.asarray(kept_a[i], dtype=np.int64)
        Bk = np.asarray(kept_b[i], dtype=np.int64)
        y = relu(_bn(w, p + "bn1", conv2d(x, w[p + "conv1_w"][A], 1, 0), A))
        y = relu(_bn(w, p + "bn2", conv2d(y, w[p + "conv2_w"][Bk][:, A], stride, 1), Bk))
        y = _bn(w, p + "bn3", conv2d(y, w[p + "conv3_w"][:, Bk], 1, 0))
        sc = _bn(w, p + "down_bn", conv2d(x, w[p + "down_w"], stride, 0)) if proj else x
        x = relu(y + sc)
    return head(w, x)


def resnet_masked_weights(w: dict, cfg, kept_a, kept_b) -> dict:
    """Eq. 7 literally: M_conv (.) W_conv with M zero on pruned channels:
    conv1 rows outside S_a, conv2 rows outside S_b and columns outside S_a,
    conv3 columns outside S_b. BN parameters are left whole (a pruned
    channel's BN output only ever meets zero weights downstream)."""
    out = dict(w)
    for i, (_, wdt, _, _) in enumerate(block_list(cfg)):
        p = f"b{i}."
        ma = np.zeros(wdt)
        ma[np.asarray(kept_a[i], dtype=np.int64)] = 1.0
        mb = np.zeros(wdt)
        mb[np.asarray(kept_b[i], dtype=np.int64)] = 1.0
        out[p + "conv1_w"] = w[p + "conv1_w"] * ma[:, None, None, None]
        out[p + "conv2_w"] = w[p + "conv2_w"] * mb[:, None, None, None] * ma[None, :, None, None]
        out[p + "conv3_w"] = w[p + "conv3_w"] * mb[None, :, None, None]
    return out


def fold_bn(W: np.ndarray, g, b, mean, var, eps: float = BN_EPS):
    """BN(conv(x, W)) = conv(x, W * s) + (b - mean * s) with s = g / sqrt(var + eps)
    per output channel. Returns (W', bias') in float64."""
    s = g / np.sqrt(var + eps)
    return W * s[:, None, None, None], b - mean * s


def resnet_forward_folded(w: dict, cfg, kept_a, kept_b, images: np.ndarray) -> np.ndarray:
    """The sliced forward with every BN folded into its conv (an algebraic
    identity of inference BN); pins the folding the packed CNN weights use."""
    def cbr(x, W, name, stride, pad, idx=None, act=True):
        g, b, m, v = (w[f"{name}.{s}"] for s in ("g", "b", "mean", "var"))
        if idx is not None:
            g, b, m, v = g[idx], b[idx], m[idx], v[idx]
        Wf, bf = fold_bn(W, g, b, m, v)
        y = conv2d(x, Wf, stride, pad) + bf
        return relu(y) if act else y

    x = max_pool_3x3_s2(cbr(widen(images), w["stem_w"], "stem_bn", 2, 3))
    for i, (_, _, stride, proj) in enumerate(block_list(cfg)):
        p = f"b{i}."
        A = np.asarray(kept_a[i], dtype=np.int64)
        Bk = np.asarray(kept_b[i], dtype=np.int64)
        y = cbr(x, w[p + "conv1_w"][A], p + "bn1", 1, 0, A)
        y = cbr(y, w[p + "conv2_w"][Bk][:, A], p + "bn2", stride, 1, Bk)
        y = cbr(y, w[p + "conv3_w"][:, Bk], p + "bn3", 1, 0, act=False)
        sc = cbr(x, w[p + "down_w"], p + "down_bn", stride, 0, act=False) if proj else x
        x = relu(y + sc)
    return head(w, x)
