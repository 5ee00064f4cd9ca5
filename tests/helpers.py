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
