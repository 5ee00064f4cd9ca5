"""Run the fp64 ResNet oracle over many images on all host cores.

Worker processes are started with `spawn` (never forked from a process that
has touched the GPU) and regenerate the seeded weights and tables themselves,
so only the configuration, the mode and the images cross the process
boundary. Each worker runs numpy single-threaded; the pool supplies the
parallelism."""
from __future__ import annotations

import multiprocessing as mp
import os

import numpy as np

_CACHE = {}


def _resnet_worker(cfg, mode: int, tables, images: np.ndarray) -> np.ndarray:
    from oracle import resnet as orr
    from oracle.vit import widen_all
    from paper_2609_10018_gb300 import synth

    key = (cfg,)
    if key not in _CACHE:
        _CACHE[key] = widen_all(synth.make_resnet_weights(cfg))
    t = tables[mode]
    return orr.resnet_forward_sliced(_CACHE[key], cfg, t["a"], t["b"], images)


def resnet_logits(cfg, tables, mode: int, images: np.ndarray, chunk: int = 16) -> np.ndarray:
    """Oracle logits [B, classes] of `mode` (tables as passed to the model)."""
    workers = max(1, min(os.cpu_count() or 1, (len(images) + chunk - 1) // chunk))
    parts = [images[i:i + chunk] for i in range(0, len(images), chunk)]
    saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    for k in saved:
        os.environ[k] = "1"  # inherited by the spawned workers only
    try:
        with mp.get_context("spawn").Pool(workers) as pool:
            outs = pool.starmap(_resnet_worker, [(cfg, mode, tables, p) for p in parts])
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
    return np.concatenate(outs, axis=0)
