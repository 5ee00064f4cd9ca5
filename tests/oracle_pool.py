"""Run the fp64 oracle over many images on all host cores.

Worker processes are started with `spawn` (never forked from a process that
has touched the GPU) and regenerate the seeded weights themselves, so only
the configuration, the kept tables and the images cross the process
boundary. Each worker runs numpy single-threaded; the pool supplies the
parallelism."""
from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np

_CACHE = {}


def _weights(kind: str, cfg):
    from oracle.vit import widen_all
    from paper_2609_10018_gb300 import synth

    key = (kind, cfg)
    if key not in _CACHE:
        make = synth.make_resnet_weights if kind == "resnet" else synth.make_vit_weights
        _CACHE[key] = widen_all(make(cfg))
    return _CACHE[key]


def _resnet_worker(cfg, mode: int, tables, images: np.ndarray) -> np.ndarray:
    from oracle import resnet as orr

    t = tables[mode]
    return orr.resnet_forward_sliced(_weights("resnet", cfg), cfg, t["a"], t["b"], images)


def _vit_worker(cfg, mode: int, tables, images: np.ndarray) -> np.ndarray:
    from oracle import vit as ov

    t = tables[mode]
    return ov.vit_forward_sliced(_weights("vit", cfg), cfg, t["heads"], t["mlp"], images, embed_kept=t.get("embed"))


def _pool_map(worker, cfg, tables, mode: int, images: np.ndarray, chunk: int) -> np.ndarray:
    parts = [images[i:i + chunk] for i in range(0, len(images), chunk)]
    workers = max(1, min(os.cpu_count() or 1, len(parts)))
    saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    for k in saved:
        os.environ[k] = "1"  # inherited by the spawned workers only
    try:
        with mp.get_context("spawn").Pool(workers) as pool:
            outs = pool.starmap(worker, [(cfg, mode, tables, p) for p in parts])
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    return np.concatenate(outs, axis=0)


def resnet_logits(cfg, tables, mode: int, images: np.ndarray, chunk: int = 16) -> np.ndarray:
    """Oracle logits [B, classes] of `mode` (tables as passed to the model)."""
    return _pool_map(_resnet_worker, cfg, tables, mode, images, chunk)


def vit_logits(cfg, tables, mode: int, images: np.ndarray, chunk: int = 4) -> np.ndarray:
    """Oracle logits [B, classes] of the elastic ViT's `mode` (tables as
    passed to the model, an optional "embed" entry included)."""
    return _pool_map(_vit_worker, cfg, tables, mode, images, chunk)
