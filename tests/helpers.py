"""Shared test helpers: device buffers via torch (plumbing only) and the
comparison metrics used by the parity tests."""
from __future__ import annotations

import numpy as np


def dev(a: np.ndarray):
    """Copy a host array to a CUDA tensor (uint16 arrays hold bf16 bits)."""
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).cuda()


def empty_dev(shape, dtype):
    import torch
    return torch.empty(shape, dtype=dtype, device="cuda")


def stream_handle() -> int:
    import torch
    return torch.cuda.current_stream().cuda_stream


def bf16_to_f64(bits) -> np.ndarray:
    """bf16 bit patterns (numpy uint16 or a torch uint16 tensor) -> float64."""
    a = bits.cpu().numpy() if hasattr(bits, "cpu") else np.asarray(bits)
    return (a.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def rel_err(got: np.ndarray, ref: np.ndarray) -> float:
    """max |got - ref| / max |ref| (the logit tolerance metric)."""
    return float(np.max(np.abs(got - ref)) / max(float(np.max(np.abs(ref))), 1e-30))


def top1_agreement(got: np.ndarray, ref: np.ndarray) -> float:
    return float(np.mean(got.argmax(axis=1) == ref.argmax(axis=1)))


def margin(ref: np.ndarray) -> np.ndarray:
    """Oracle top-1 minus top-2 logit, per image."""
    s = np.sort(ref, axis=1)
    return s[:, -1] - s[:, -2]


BF16_U = 2.0 ** -9  # unit roundoff of a bf16 activation


def centered(x: np.ndarray) -> np.ndarray:
    """Logits minus their mean over the batch: the part that varies from image
    to image."""
    return x - x.mean(axis=0, keepdims=True)


def centred_tolerance(ref: np.ndarray, layers: int, roundings_per_layer: int = 5) -> float:
    """Bound on the relative error of the centred logits of a bf16 forward.
    Each layer rounds its activations to bf16 (unit roundoff 2^-9) at
    `roundings_per_layer` points (LN output, q/k/v, P, O, MLP hidden); the
    roundings are independent, so their effect on a logit grows like a random
    walk, about 2^-9 * sqrt(5 L) of max|logit|. Relative to the centred part,
    which is a share s of max|logit|, that is 2^-9 * sqrt(5 L) / s; never
    below 2e-2."""
    share = float(np.max(np.abs(centered(ref))) / np.max(np.abs(ref)))
    if share == 0.0:  # one image: nothing varies across the batch
        return float("inf")
    return max(2e-2, BF16_U * np.sqrt(roundings_per_layer * layers) / share)


def check_image_dependent_part(tag: str, got: np.ndarray, ref: np.ndarray, layers: int) -> dict:
    """With random weights most of a logit is the same for every image (the
    ViTs give every image the same top class), so besides max|dlogit| this
    checks the part that the images themselves decide: the centred logits
    within centred_tolerance, and the top class of the centred logits the
    same as the oracle's wherever the oracle's own centred margin exceeds
    twice the largest centred error (where it does not, either class is a
    valid answer)."""
    cg, cr = centered(got), centered(ref)
    cerr = rel_err(cg, cr)
    tol = centred_tolerance(ref, layers)
    dmax = float(np.max(np.abs(cg - cr)))
    cm = margin(cr)
    decided = cm > 2.0 * dmax
    agree_c = cg.argmax(axis=1) == cr.argmax(axis=1)
    out = {"err": rel_err(got, ref), "top1": top1_agreement(got, ref), "centred_err": cerr, "centred_tol": tol,
           "centred_share": float(np.max(np.abs(cr)) / np.max(np.abs(ref))),
           "centred_top1": float(np.mean(agree_c)), "centred_decided": int(decided.sum())}
    print(f"{tag}: err {out['err']:.2e} top1 {out['top1']:.4f} | image-dependent part "
          f"{out['centred_share']:.2e} of max|logit|, its err {cerr:.2e} (bound {tol:.2e}), centred top-1 "
          f"{out['centred_top1']:.4f} ({out['centred_decided']}/{len(ref)} decided by margin)")
    assert cerr <= tol, (tag, cerr, tol)
    assert np.all(agree_c[decided]), (tag, np.flatnonzero(decided & ~agree_c))
    return out
