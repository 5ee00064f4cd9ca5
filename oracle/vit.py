"""fp64 oracle: elastic ViT descendant-network forward pass.

Test infrastructure only (see the package docstring).

Model (Section 4.1 and 5.2: ViT "following the original implementation"):
  tokens      n = N + 1, N = HW / P^2 patches of P x P x C, linearly projected
              to d, a class token prepended, a learned position embedding added;
  block       pre-norm: X += MHA(LN1(X)); X += MLP(LN2(X));
  MHA         Eq. 2-3, h heads of width d_i = d / h, scale 1 / sqrt(d_i);
  MLP         Eq. 5, W2 phi(W1 x + b1) + b2, phi = exact (erf) GELU;
  head        LN of the class token, then a linear classifier.

Elastic descendant networks (Eq. 4 and 6): a DN multiplies the projection
weights by binary masks. Here the masks are structured: a DN keeps a set of
heads H per layer (rows of W^Q, W^K, W^V and the matching input columns of
W^O) and a set of MLP hidden channels F per layer (rows of W1, columns of W2).
Multiplying by a 0/1 mask that zeroes whole rows/columns is the same as
deleting them, so the DN forward is the forward of the sliced matrices.
Readings where the paper is silent:
  - attention scale stays 1 / sqrt(d / h) of the base model (Eq. 3 with the
    base d_i); it does not depend on how many heads are kept;
  - biases of deleted rows (q, k, v, fc1) are deleted with them; b^O and b2
    are kept whole;
  - LayerNorm eps = 1e-6;
  - embedding-width pruning (Section 4.1: the compress stage also shrinks the
    hidden size of the LayerNorm and patch-embedding layers) keeps a set E of
    the d channels in every layer alike (the residual stream has one width):
    the DN is the ViT of width |E| whose weights are the kept sub-blocks, so
    each LayerNorm normalises over the kept channels only. Heads keep their
    width d_i = d / h of the base model (and the 1 / sqrt(d_i) scale). With
    no embedding table every channel is kept.
"""
from __future__ import annotations

import numpy as np
from scipy.special import erf

from .counts import mm

LN_EPS = 1e-6


# ----------------------------------------------------------------------------
# Input widening (exact)
# ----------------------------------------------------------------------------

def widen(a) -> np.ndarray:
    """Stored values -> float64, exactly. uint16 arrays are bf16 bit patterns."""
    a = np.asarray(a)
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def widen_all(weights: dict) -> dict:
    return {k: widen(v) for k, v in weights.items()}


# ----------------------------------------------------------------------------
# Building blocks
# ----------------------------------------------------------------------------

def layer_norm(x: np.ndarray, gamma: np.ndarray, beta: np.ndarray, eps: float = LN_EPS) -> np.ndarray:
    """Per row: (x - mean) / sqrt(var + eps) * gamma + beta, biased variance."""
    mu = x.mean(axis=-1, keepdims=True)
    var = ((x - mu) ** 2).mean(axis=-1, keepdims=True)
    return (x - mu) / np.sqrt(var + eps) * gamma + beta


def gelu(x: np.ndarray) -> np.ndarray:
    """phi in Eq. 5: exact GELU, x * Phi(x) = 0.5 x (1 + erf(x / sqrt 2))."""
    return 0.5 * x * (1.0 + erf(x / np.sqrt(2.0)))


def softmax_rows(s: np.ndarray) -> np.ndarray:
    """Row softmax, exp(s - max) / sum (shifting by the row max changes nothing
    mathematically and keeps exp finite)."""
    e = np.exp(s - s.max(axis=-1, keepdims=True))
    return e / e.sum(axis=-1, keepdims=True)


def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, d_i: int) -> np.ndarray:
    """Eq. 3: softmax(q k^T / sqrt(d_i)) v over the last two axes."""
    s = mm(q, np.swapaxes(k, -1, -2), "attn") / np.sqrt(d_i)
    return mm(softmax_rows(s), v, "attn")


def attention_naive(q: np.ndarray, k: np.ndarray, v: np.ndarray, d_i: int) -> np.ndarray:
    """Eq. 3 written element by element (pure loops; tiny inputs only).
    q: [n, d_i], k, v: [m, d_i]."""
    n, m, dv = q.shape[0], k.shape[0], v.shape[1]
    out = np.zeros((n, dv))
    for i in range(n):
        scores = [sum(q[i, c] * k[j, c] for c in range(d_i)) / np.sqrt(d_i) for j in range(m)]
        top = max(scores)
        ex = [np.exp(s - top) for s in scores]
        z = sum(ex)
        for c in range(dv):
            out[i, c] = sum(ex[j] / z * v[j, c] for j in range(m))
    return out


def patchify(images: np.ndarray, P: int) -> np.ndarray:
    """[B, H, W, C] -> [B, N, C*P*P]; patch p = (py, px) row-major; within a
    patch the flattened order is (c, ky, kx), matching a [d, C, P, P] kernel."""
    B, H, W, C = images.shape
    t = images.reshape(B, H // P, P, W // P, P, C)          # b, py, ky, px, kx, c
    t = t.transpose(0, 1, 3, 5, 2, 4)                        # b, py, px, c, ky, kx
    return t.reshape(B, (H // P) * (W // P), C * P * P)


def embed(w: dict, cfg, images: np.ndarray) -> np.ndarray:
    """Section 4.1: N = HW/P^2 patches linearly projected to d; n = N + 1 with
    the class token; plus the position embedding. Returns X0 [B, n, d] (d =
    the rows of patch_w: the kept width after embedding pruning)."""
    d = w["patch_w"].shape[0]
    patches = patchify(widen(images), cfg.patch)
    t = mm(patches, w["patch_w"].reshape(d, -1).T, "patch") + w["patch_b"]
    B = t.shape[0]
    cls = np.broadcast_to(w["cls"], (B, 1, d))
    return np.concatenate([cls, t], axis=1) + w["pos"]


def classify(w: dict, X: np.ndarray) -> np.ndarray:
    """LN of the class token, then the linear head: logits [B, C]."""
    c = layer_norm(X[:, 0], w["norm_w"], w["norm_b"])
    return mm(c, w["head_w"].T, "head") + w["head_b"]


# ----------------------------------------------------------------------------
# Forward passes
# ----------------------------------------------------------------------------

def vit_forward_dense(w: dict, cfg, images: np.ndarray) -> np.ndarray:
    """The unmodified base model (all heads, all MLP channels). `w` must be
    widened (float64). Returns logits [B, classes]."""
    d, h = cfg.dim, cfg.heads
    di = d // h
    X = embed(w, cfg, images)
    B, n, _ = X.shape
    for l in range(cfg.layers):
        p = f"l{l}."
        Y = layer_norm(X, w[p + "ln1_w"], w[p + "ln1_b"])
        qkv = mm(Y, w[p + "qkv_w"].T, "qkv") + w[p + "qkv_b"]              # [B, n, 3d]
        qkv = qkv.reshape(B, n, 3, h, di).transpose(2, 0, 3, 1, 4)          # 3, B, h, n, di
        O = attention(qkv[0], qkv[1], qkv[2], di)                            # B, h, n, di
        O = O.transpose(0, 2, 1, 3).reshape(B, n, d)                         # concat heads (Eq. 2)
        X = X + mm(O, w[p + "proj_w"].T, "proj") + w[p + "proj_b"]
        Y2 = layer_norm(X, w[p + "ln2_w"], w[p + "ln2_b"])
        Hid = gelu(mm(Y2, w[p + "fc1_w"].T, "fc1") + w[p + "fc1_b"])
        X = X + mm(Hid, w[p + "fc2_w"].T, "fc2") + w[p + "fc2_b"]
    return classify(w, X)


def slice_embedding(w: dict, cfg, embed_kept) -> dict:
    """Embedding-width pruning as deletion: every axis of length d that is the
    residual-stream width keeps the channels E = embed_kept (ascending). The
    patch embedding, class token, position embedding, LayerNorm parameters,
    b^O and b2 keep entries E; W^O and W2 keep output rows E; W^Q, W^K, W^V
    and W1 keep input columns E; the classifier keeps input columns E. The
    head axes (rows of W_qkv, columns of W^O) are not embedding channels."""
    E = np.asarray(embed_kept, dtype=np.int64)
    out = dict(w)
    out["patch_w"] = w["patch_w"][E]
    for k in ("patch_b", "cls", "norm_w", "norm_b"):
        out[k] = w[k][E]
    out["pos"] = w["pos"][:, E]
    out["head_w"] = w["head_w"][:, E]
    for l in range(cfg.layers):
        p = f"l{l}."
        for k in ("ln1_w", "ln1_b", "ln2_w", "ln2_b", "proj_b", "fc2_b"):
            out[p + k] = w[p + k][E]
        out[p + "qkv_w"] = w[p + "qkv_w"][:, E]
        out[p + "fc1_w"] = w[p + "fc1_w"][:, E]
        out[p + "proj_w"] = w[p + "proj_w"][E]
        out[p + "fc2_w"] = w[p + "fc2_w"][E]
    # row-major like the inputs (a column gather is column-major in numpy),
    # so the matrix products see the same layout as without pruning
    return {k: np.ascontiguousarray(v) for k, v in out.items()}


def vit_forward_sliced(w: dict, cfg, heads_kept, mlp_kept, images: np.ndarray,
                       embed_kept=None) -> np.ndarray:
    """DN forward (Eq. 2-6 with structured masks applied as deletion).

    heads_kept[l]: ascending kept head indices of layer l (subset of [0, h)).
    mlp_kept[l]:   ascending kept MLP hidden channels of layer l.
    embed_kept:    ascending kept embedding channels (None: all d).
    """
    d, h = cfg.dim, cfg.heads
    di = d // h
    if embed_kept is not None:
        w = slice_embedding(w, cfg, embed_kept)
    X = embed(w, cfg, images)
    for l in range(cfg.layers):
        p = f"l{l}."
        Wqkv, bqkv = w[p + "qkv_w"], w[p + "qkv_b"]
        Y = layer_norm(X, w[p + "ln1_w"], w[p + "ln1_b"])
        outs, cols = [], []
        for j in heads_kept[l]:
            r = np.arange(j * di, (j + 1) * di)
            q = mm(Y, Wqkv[r].T, "qkv") + bqkv[r]
            k = mm(Y, Wqkv[d + r].T, "qkv") + bqkv[d + r]
            v = mm(Y, Wqkv[2 * d + r].T, "qkv") + bqkv[2 * d + r]
            outs.append(attention(q, k, v, di))
            cols.append(r)
        if outs:
            O = np.concatenate(outs, axis=-1)                                # Concat(head_j), j in H
            X = X + mm(O, w[p + "proj_w"][:, np.concatenate(cols)].T, "proj") + w[p + "proj_b"]
        else:                                                                # no head kept: b^O only
            X = X + w[p + "proj_b"]
        Y2 = layer_norm(X, w[p + "ln2_w"], w[p + "ln2_b"])
        F = np.asarray(mlp_kept[l], dtype=np.int64)
        if F.size:
            Hid = gelu(mm(Y2, w[p + "fc1_w"][F].T, "fc1") + w[p + "fc1_b"][F])
            X = X + mm(Hid, w[p + "fc2_w"][:, F].T, "fc2") + w[p + "fc2_b"]
        else:                                                                # no channel kept: b2 only
            X = X + w[p + "fc2_b"]
    return classify(w, X)


def vit_masked_weights(w: dict, cfg, heads_kept, mlp_kept) -> dict:
    """Eq. 4 and 6 literally: full-shape weights multiplied by 0/1 masks.
    M^Q, M^K, M^V keep the rows of the kept heads, M^O keeps the matching
    input columns of W^O, M1 keeps rows of W1, M2 keeps columns of W2; the
    biases of masked rows are zeroed with them."""
    d, h = cfg.dim, cfg.heads
    di = d // h
    out = dict(w)
    for l in range(cfg.layers):
        p = f"l{l}."
        head_on = np.zeros(d)
        for j in heads_kept[l]:
            head_on[j * di:(j + 1) * di] = 1.0
        row3 = np.concatenate([head_on] * 3)
        out[p + "qkv_w"] = w[p + "qkv_w"] * row3[:, None]
        out[p + "qkv_b"] = w[p + "qkv_b"] * row3
        out[p + "proj_w"] = w[p + "proj_w"] * head_on[None, :]
        ch_on = np.zeros(cfg.mlp)
        ch_on[np.asarray(mlp_kept[l], dtype=np.int64)] = 1.0
        out[p + "fc1_w"] = w[p + "fc1_w"] * ch_on[:, None]
        out[p + "fc1_b"] = w[p + "fc1_b"] * ch_on
        out[p + "fc2_w"] = w[p + "fc2_w"] * ch_on[None, :]
    return out


# ----------------------------------------------------------------------------
# Packed layout of one mode (the per-mode index gather done at create time)
# ----------------------------------------------------------------------------

def _bf16_bits_rne(x32: np.ndarray) -> np.ndarray:
    """fp32 values -> bf16 bit patterns, round to nearest, ties to even."""
    u = np.ascontiguousarray(x32, dtype=np.float32).view(np.uint32).astype(np.uint64)
    hi, rem = u >> np.uint64(16), u & np.uint64(0xFFFF)
    up = (rem > 0x8000) | ((rem == 0x8000) & ((hi & np.uint64(1)) == 1))
    return (hi + up.astype(np.uint64)).astype(np.uint16)


def _as_bf16_bits(a: np.ndarray) -> np.ndarray:
    a = np.asarray(a)
    return a if a.dtype == np.uint16 else _bf16_bits_rne(a.astype(np.float32))


def _as_f32(a: np.ndarray) -> np.ndarray:
    return widen(a).astype(np.float32)


def vit_pack_layer(stored: dict, cfg, layer: int, heads, mlp) -> dict:
    """The packed per-mode buffers of one layer, from the STORED (not widened)
    weights. Matrices are bf16 bit patterns, bias vectors fp32:

      qkv_w [3 w_m, d]  rows {blk*d + j*d_i + r : blk in (q, k, v), j in H asc, r < d_i}
      qkv_b [3 w_m]     the same rows of b_qkv
      proj_w [d, w_m]   columns {j*d_i + r : j in H asc, r < d_i} of W^O
      fc1_w [f_m, d]    rows F of W1
      fc1_b [f_m]       entries F of b1
      fc2_w [d, f_m]    columns F of W2
    """
    d, di = cfg.dim, cfg.dim // cfg.heads
    p = f"l{layer}."
    cols = np.array([j * di + r for j in heads for r in range(di)], dtype=np.int64)
    rows = np.array([blk * d + c for blk in range(3) for c in cols], dtype=np.int64)
    F = np.asarray(mlp, dtype=np.int64)
    return {
        "qkv_w": _as_bf16_bits(stored[p + "qkv_w"])[rows] if rows.size else np.zeros((0, d), np.uint16),
        "qkv_b": _as_f32(stored[p + "qkv_b"])[rows],
        "proj_w": np.ascontiguousarray(_as_bf16_bits(stored[p + "proj_w"])[:, cols]),
        "fc1_w": _as_bf16_bits(stored[p + "fc1_w"])[F] if F.size else np.zeros((0, d), np.uint16),
        "fc1_b": _as_f32(stored[p + "fc1_b"])[F],
        "fc2_w": np.ascontiguousarray(_as_bf16_bits(stored[p + "fc2_w"])[:, F]),
    }


PACK_ORDER = ("qkv_w", "qkv_b", "proj_w", "fc1_w", "fc1_b", "fc2_w")
