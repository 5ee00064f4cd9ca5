"""fp64 oracle: L1-norm saliency of the Compress stage (Section 4.1) and the
kept tables it induces.

Test infrastructure only (see the package docstring).

Section 4.1: for each weight matrix, each row's average absolute magnitude is
its saliency; the lowest rows are masked out (Eq. 4 for W^Q, W^K, W^V, W^O,
Eq. 6 for W1, W2, Eq. 7 for convolutions). Readings (structured pruning at
the granularity the descendant networks use, as for the kept tables):
  - a "row" of W^Q, W^K, W^V is an output channel (PyTorch [out, in] rows); a
    "row" of W^O (hd_i x d in the paper's notation) is an input channel, i.e.
    a column of PyTorch's [d, d] W^O; likewise a hidden channel owns a row of
    W1 [d_ff, d] and a column of W2 [d, d_ff];
  - a head's saliency is the mean of the row averages of the 4 x 64 rows it
    owns (its q, k, v output rows and its W^O input rows); an MLP channel's is
    the mean of its W1 row average and its W2 column average;
  - ResNet-50: a channel of S_a owns conv1's output row (over cin) and conv2's
    input slice (over w_out x 3 x 3); a channel of S_b owns conv2's output row
    (over w_in x 3 x 3) and conv3's input column (over 4w); its saliency is the
    mean of its two averages;
  - an embedding channel c (the residual-stream width pruned with the
    LayerNorm and patch-embedding hidden size) owns the rows that write it and
    the columns that read it: row c of the patch projection (over C x P x P),
    of W^O and of W2 in every layer; column c of W_qkv and of W1 in every
    layer and of the classifier. Its saliency is the mean of those 2 + 4L
    averages (LayerNorm gains are scales, not rows, and are left out);
  - a mode keeping k units keeps the k most salient (ties: lower index),
    listed ascending; one ranking for all modes makes the sets nested (Eq. 8).
"""
from __future__ import annotations

import numpy as np


def vit_saliency(w: dict, cfg) -> tuple[np.ndarray, np.ndarray]:
    """`w` widened to float64. Returns head scores [L, h] and MLP channel
    scores [L, d_ff]."""
    d, h = cfg.dim, cfg.heads
    hs = np.zeros((cfg.layers, h))
    fs = np.zeros((cfg.layers, cfg.mlp))
    for l in range(cfg.layers):
        qkv = np.abs(w[f"l{l}.qkv_w"]).mean(axis=1)           # [3d] output rows
        proj = np.abs(w[f"l{l}.proj_w"]).mean(axis=0)         # [d] input columns of W^O
        for j in range(h):
            rows = [qkv[b * d + j * 64: b * d + (j + 1) * 64] for b in range(3)] + [proj[j * 64:(j + 1) * 64]]
            hs[l, j] = np.concatenate(rows).mean()
        fc1 = np.abs(w[f"l{l}.fc1_w"]).mean(axis=1)           # [d_ff] rows
        fc2 = np.abs(w[f"l{l}.fc2_w"]).mean(axis=0)           # [d_ff] columns
        fs[l] = 0.5 * (fc1 + fc2)
    return hs, fs


def vit_embed_saliency(w: dict, cfg) -> np.ndarray:
    """`w` widened to float64. Scores of the d embedding channels."""
    d = cfg.dim
    parts = [np.abs(w["patch_w"]).reshape(d, -1).mean(axis=1),   # patch projection rows
             np.abs(w["head_w"]).mean(axis=0)]                     # classifier columns
    for l in range(cfg.layers):
        p = f"l{l}."
        parts += [np.abs(w[p + "qkv_w"]).mean(axis=0),             # W_qkv columns (inputs)
                  np.abs(w[p + "proj_w"]).mean(axis=1),            # W^O rows (outputs)
                  np.abs(w[p + "fc1_w"]).mean(axis=0),             # W1 columns
                  np.abs(w[p + "fc2_w"]).mean(axis=1)]             # W2 rows
    return np.mean(parts, axis=0)


def resnet_saliency(w: dict, blocks) -> tuple[list, list]:
    """Per block, scores of the S_a and S_b candidate channels."""
    sa, sb = [], []
    for i, (_, wd, _, _) in enumerate(blocks):
        c1, c2, c3 = (w[f"b{i}.conv{k}_w"] for k in (1, 2, 3))
        a = 0.5 * (np.abs(c1).reshape(wd, -1).mean(axis=1) + np.abs(c2).transpose(1, 0, 2, 3).reshape(wd, -1).mean(axis=1))
        b = 0.5 * (np.abs(c2).reshape(wd, -1).mean(axis=1) + np.abs(c3).reshape(c3.shape[0], wd).mean(axis=0))
        sa.append(a)
        sb.append(b)
    return sa, sb


def top_k(scores: np.ndarray, k: int) -> np.ndarray:
    """Indices of the k largest scores (ties: lower index), ascending."""
    order = sorted(range(len(scores)), key=lambda i: (-scores[i], i))
    return np.sort(np.asarray(order[:k], dtype=np.int32))
