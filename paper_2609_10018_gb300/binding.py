"""ctypes binding to libelasto.so (include/elasto.h, include/elasto_ops.h).

Argument marshalling only: every step of the forward pass runs in the CUDA
library. Functions keep the C names; `ElasticModel` is a small owner of one
handle. Device buffers are passed as integer addresses (e.g. a torch CUDA
tensor's data_ptr()), streams as integer cudaStream_t handles (e.g.
torch.cuda.current_stream().cuda_stream). There is no CPU fallback: if the
library is missing this module raises.
"""
from __future__ import annotations

import ctypes
import os
from typing import Dict, List, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libelasto.so")

ARCH_VIT, ARCH_RESNET50 = 1, 2
F32, BF16 = 0, 1
OK, ERR_INVALID_ARG, ERR_BAD_TABLE, ERR_BAD_MODE, ERR_OOM, ERR_CUDA, ERR_UNSUPPORTED, ERR_TIMEOUT, ERR_GUARD = (
    0, -1, -2, -3, -4, -5, -6, -7, -8)
Q_N_MODES, Q_PACKED_BYTES, Q_SHARED_BYTES, Q_WORKSPACE_BYTES, Q_ARENA_BYTES, Q_MODE_MACS, Q_LAUNCHES = range(7)
Q_PACKED_TOTAL, Q_PREFIX_SHARED, Q_GUARD_ZONES, Q_ONE_LAUNCH = 7, 8, 9, 10
EPI_BIAS_BF16, EPI_BIAS_GELU_BF16, EPI_BIAS_RESID_F32, EPI_BIAS_F32, EPI_BIAS_RELU_BF16, EPI_BIAS_RESID_RELU_BF16 = range(6)
EPI_BIAS_RELU_F16, EPI_BIAS_F16, EPI_BIAS_RESID_RELU_F16 = range(6, 9)  # A, W, resid, out in IEEE f16

c_int, c_void_p, c_size_t, c_int64 = ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int64
P_i32 = ctypes.POINTER(ctypes.c_int32)


class ModelDesc(ctypes.Structure):
    _fields_ = [("arch", c_int), ("img_h", c_int), ("img_w", c_int), ("img_c", c_int), ("patch", c_int),
                ("dim", c_int), ("heads", c_int), ("mlp", c_int), ("layers", c_int), ("classes", c_int),
                ("weight_dtype", c_int), ("max_batch", c_int)]


class Weights(ctypes.Structure):
    _fields_ = [("tensors", ctypes.POINTER(c_void_p)), ("n_tensors", c_int)]


class ModeTables(ctypes.Structure):
    _fields_ = [("heads_kept", P_i32), ("n_heads_kept", P_i32), ("mlp_kept", P_i32), ("n_mlp_kept", P_i32),
                ("conv_kept_a", P_i32), ("n_conv_a", P_i32), ("conv_kept_b", P_i32), ("n_conv_b", P_i32),
                ("embed_kept", P_i32), ("n_embed_kept", ctypes.c_int32)]


K_PATCHIFY, K_GEMM, K_LAYERNORM, K_ATTENTION, K_HEAD, K_IM2COL, K_POOL, K_ONE_LAUNCH = range(8)
KIND_NAMES = {K_PATCHIFY: "patchify", K_GEMM: "gemm", K_LAYERNORM: "layernorm", K_ATTENTION: "attention",
              K_HEAD: "head", K_IM2COL: "im2col", K_POOL: "pool", K_ONE_LAUNCH: "one_launch"}


class DnProfile(ctypes.Structure):
    _fields_ = [("latency_ms", ctypes.c_float), ("memory_bytes", ctypes.c_double), ("gflops", ctypes.c_double),
                ("accuracy", ctypes.c_float)]


class LaunchRecord(ctypes.Structure):
    _fields_ = [("kind", c_int), ("layer", c_int), ("m", c_int), ("n", c_int), ("k", c_int),
                ("ms", ctypes.c_float), ("macs", ctypes.c_double), ("bytes", ctypes.c_double)]


class ElastoError(RuntimeError):
    def __init__(self, status: int, where: str, msg: str):
        super().__init__(f"{where} failed with status {status}: {msg}")
        self.status = status


_lib = None


def lib() -> ctypes.CDLL:
    """Load libelasto.so (raises if it has not been built)."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2609_10018_gb300.build.build()")
    L = ctypes.CDLL(LIB_PATH)
    sig = {
        "elasto_create": [ctypes.POINTER(ModelDesc), ctypes.POINTER(Weights), ctypes.POINTER(ModeTables), c_int,
                          ctypes.POINTER(c_void_p)],
        "elasto_set_mode": [c_void_p, c_int],
        "elasto_get_mode": [c_void_p, ctypes.POINTER(c_int)],
        "elasto_forward": [c_void_p, c_void_p, c_void_p, c_int, c_void_p],
        "elasto_forward_host": [c_void_p, c_void_p, c_void_p, c_int, c_void_p],
        "elasto_forward_host_batches": [c_void_p, c_void_p, c_int, c_int, ctypes.POINTER(c_void_p),
                                        ctypes.POINTER(c_void_p)],
        "elasto_forward_noalloc": [c_void_p, c_void_p, c_void_p, c_int, c_void_p],
        "elasto_sync_status": [c_void_p, c_void_p],
        "elasto_check_guards": [c_void_p, c_void_p, ctypes.POINTER(c_int)],
        "elasto_debug_damage_guard": [c_void_p, c_int],
        "elasto_destroy": [c_void_p],
        "elasto_query": [c_void_p, c_int, c_int, ctypes.POINTER(c_int64)],
        "elasto_debug_export_packed": [c_void_p, c_int, c_int, c_int, c_void_p, c_size_t],
        "elasto_profile_enable": [c_void_p, c_int],
        "elasto_set_one_launch": [c_void_p, c_int],
        "elasto_profile_read": [c_void_p, ctypes.POINTER(LaunchRecord), c_int, ctypes.POINTER(c_int)],
        "elasto_profile_dns": [c_void_p, c_void_p, c_int, c_int, ctypes.POINTER(DnProfile)],
        "elasto_select_dn": [ctypes.POINTER(DnProfile), c_int, ctypes.c_float, ctypes.c_double, ctypes.c_float,
                             ctypes.POINTER(c_int)],
        "elasto_saliency": [ctypes.POINTER(ModelDesc), ctypes.POINTER(Weights), c_void_p, c_void_p],
        "elasto_saliency_embed": [ctypes.POINTER(ModelDesc), ctypes.POINTER(Weights), c_void_p],
        "elasto_topk": [c_void_p, c_int, c_int, c_void_p],
        "elasto_op_gemm": [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_int,
                           c_void_p],
        "elasto_op_conv2d": [c_void_p, c_void_p, c_int, c_int, c_int, c_int, c_void_p, c_int, c_int, c_int, c_int,
                             c_void_p, c_int, c_void_p, c_void_p],
        "elasto_op_layernorm": [c_void_p, c_void_p, c_void_p, c_void_p, c_void_p, c_int, c_int],
        "elasto_op_softmax": [c_void_p, c_void_p, c_void_p, c_int, c_int],
        "elasto_op_attention": [c_void_p, c_void_p, c_void_p, c_int, c_int, c_int, c_void_p],
        "elasto_op_bounded_wait": [c_void_p, c_int, c_void_p, c_void_p],
        "elasto_op_grid_barrier": [c_void_p, c_int, c_void_p, c_void_p, c_void_p],
    }
    for name, args in sig.items():
        f = getattr(L, name)
        f.argtypes = args
        f.restype = c_int
    L.elasto_last_error.argtypes = []
    L.elasto_last_error.restype = ctypes.c_char_p
    _lib = L
    return L


def elasto_last_error() -> str:
    return (lib().elasto_last_error() or b"").decode()


def _check(st: int, where: str) -> None:
    if st != OK:
        raise ElastoError(st, where, elasto_last_error())


# ----------------------------------------------------------------------------
# Marshalling helpers
# ----------------------------------------------------------------------------

class _Keep:
    """Holds numpy arrays alive while their addresses are in a ctypes struct."""

    def __init__(self):
        self.items: List[object] = []

    def arr(self, a, dtype) -> np.ndarray:
        a = np.ascontiguousarray(a, dtype=dtype)
        self.items.append(a)
        return a

    def i32(self, values) -> ctypes.POINTER(ctypes.c_int32):
        a = self.arr(np.asarray(values, dtype=np.int32).reshape(-1), np.int32)
        return a.ctypes.data_as(P_i32)


def vit_desc(cfg, max_batch: int) -> ModelDesc:
    return ModelDesc(ARCH_VIT, cfg.img, cfg.img, cfg.chans, cfg.patch, cfg.dim, cfg.heads, cfg.mlp, cfg.layers,
                     cfg.classes, cfg.dtype, max_batch)


def resnet_desc(cfg, max_batch: int) -> ModelDesc:
    return ModelDesc(ARCH_RESNET50, cfg.img, cfg.img, cfg.chans, 0, 0, 0, 0, 0, cfg.classes, cfg.dtype, max_batch)


def vit_mode_tables(keep: _Keep, tables: Sequence[Dict[str, Sequence[np.ndarray]]]):
    arr = (ModeTables * len(tables))()
    for m, t in enumerate(tables):
        heads = [np.asarray(h, np.int32) for h in t["heads"]]
        mlp = [np.asarray(f, np.int32) for f in t["mlp"]]
        arr[m].heads_kept = keep.i32(np.concatenate(heads) if heads else [])
        arr[m].n_heads_kept = keep.i32([len(h) for h in heads])
        arr[m].mlp_kept = keep.i32(np.concatenate(mlp) if mlp else [])
        arr[m].n_mlp_kept = keep.i32([len(f) for f in mlp])
        if t.get("embed") is not None:  # kept embedding channels (absent: all)
            arr[m].embed_kept = keep.i32(t["embed"])
            arr[m].n_embed_kept = len(t["embed"])
    return arr


def resnet_mode_tables(keep: _Keep, tables):
    arr = (ModeTables * len(tables))()
    for m, t in enumerate(tables):
        a = [np.asarray(x, np.int32) for x in t["a"]]
        b = [np.asarray(x, np.int32) for x in t["b"]]
        arr[m].conv_kept_a = keep.i32(np.concatenate(a))
        arr[m].n_conv_a = keep.i32([len(x) for x in a])
        arr[m].conv_kept_b = keep.i32(np.concatenate(b))
        arr[m].n_conv_b = keep.i32([len(x) for x in b])
    return arr


def weights_struct(keep: _Keep, tensors: Sequence[np.ndarray]) -> Weights:
    ptrs = (c_void_p * len(tensors))()
    for i, t in enumerate(tensors):
        a = np.ascontiguousarray(t)
        keep.items.append(a)
        ptrs[i] = a.ctypes.data
    keep.items.append(ptrs)
    return Weights(ptrs, len(tensors))


# ----------------------------------------------------------------------------
# C-ABI calls (same names)
# ----------------------------------------------------------------------------

def elasto_create(desc: ModelDesc, tensors: Sequence[np.ndarray], mode_tables, n_modes: int | None = None,
                  keep: _Keep | None = None) -> int:
    keep = keep or _Keep()
    w = weights_struct(keep, tensors)
    h = c_void_p()
    n = len(mode_tables) if n_modes is None else n_modes
    _check(lib().elasto_create(ctypes.byref(desc), ctypes.byref(w), mode_tables, n, ctypes.byref(h)),
           "elasto_create")
    return h.value


def elasto_set_mode(h: int, mode: int) -> None:
    _check(lib().elasto_set_mode(h, mode), "elasto_set_mode")


def elasto_get_mode(h: int) -> int:
    v = c_int()
    _check(lib().elasto_get_mode(h, ctypes.byref(v)), "elasto_get_mode")
    return v.value


def elasto_forward(h: int, stream: int, images_ptr: int, batch: int, logits_ptr: int) -> None:
    _check(lib().elasto_forward(h, stream, images_ptr, batch, logits_ptr), "elasto_forward")


def elasto_forward_noalloc(h: int, stream: int, images_ptr: int, batch: int, logits_ptr: int) -> None:
    """Forward with the library's fixed static scratch; allocates nothing."""
    _check(lib().elasto_forward_noalloc(h, stream, images_ptr, batch, logits_ptr), "elasto_forward_noalloc")


def elasto_forward_host(h: int, stream: int, images: np.ndarray, batch: int, logits: np.ndarray) -> None:
    assert images.flags["C_CONTIGUOUS"] and logits.flags["C_CONTIGUOUS"] and logits.dtype == np.float32
    _check(lib().elasto_forward_host(h, stream, images.ctypes.data, batch, logits.ctypes.data),
           "elasto_forward_host")


def elasto_forward_host_batches(h: int, stream: int, images: List[np.ndarray], logits: List[np.ndarray]) -> None:
    """Batches from host memory, copies overlapped with the forwards (all
    batches the same size; pinned host arrays for the overlap)."""
    n = len(images)
    assert n == len(logits) and n > 0
    for a in list(images) + list(logits):
        assert a.flags["C_CONTIGUOUS"]
    assert all(l.dtype == np.float32 for l in logits)
    ip = (c_void_p * n)(*[a.ctypes.data for a in images])
    lp = (c_void_p * n)(*[a.ctypes.data for a in logits])
    _check(lib().elasto_forward_host_batches(h, stream, n, images[0].shape[0], ip, lp),
           "elasto_forward_host_batches")


def elasto_sync_status(h: int, stream: int = 0) -> None:
    _check(lib().elasto_sync_status(h, stream), "elasto_sync_status")


def elasto_check_guards(h: int, stream: int = 0) -> int:
    """Number of damaged guard zones; raises ElastoError (ERR_GUARD) if any."""
    n = c_int(0)
    _check(lib().elasto_check_guards(h, stream, ctypes.byref(n)), "elasto_check_guards")
    return n.value


def elasto_debug_damage_guard(h: int, zone: int) -> None:
    _check(lib().elasto_debug_damage_guard(h, zone), "elasto_debug_damage_guard")


def elasto_destroy(h: int) -> None:
    _check(lib().elasto_destroy(h), "elasto_destroy")


def elasto_query(h: int, what: int, mode: int = 0) -> int:
    v = c_int64()
    _check(lib().elasto_query(h, what, mode, ctypes.byref(v)), "elasto_query")
    return v.value


def elasto_debug_export_packed(h: int, mode: int, layer: int, which: int, out: np.ndarray) -> np.ndarray:
    assert out.flags["C_CONTIGUOUS"]
    _check(lib().elasto_debug_export_packed(h, mode, layer, which, out.ctypes.data, out.nbytes),
           "elasto_debug_export_packed")
    return out


def elasto_set_one_launch(h: int, enable: bool) -> None:
    _check(lib().elasto_set_one_launch(h, 1 if enable else 0), "elasto_set_one_launch")


def elasto_profile_enable(h: int, enable: bool) -> None:
    _check(lib().elasto_profile_enable(h, 1 if enable else 0), "elasto_profile_enable")


def elasto_profile_read(h: int, capacity: int = 1024) -> List[dict]:
    """Per-launch records of the most recent forward (synchronises)."""
    buf = (LaunchRecord * capacity)()
    n = c_int()
    _check(lib().elasto_profile_read(h, buf, capacity, ctypes.byref(n)), "elasto_profile_read")
    return [{"kind": KIND_NAMES.get(r.kind, str(r.kind)), "layer": r.layer, "m": r.m, "n": r.n, "k": r.k,
             "ms": r.ms, "macs": r.macs, "bytes": r.bytes} for r in buf[:n.value]]


def elasto_profile_dns(h: int, stream: int, batch: int, trials: int, n_modes: int) -> List[dict]:
    """Measured look-up table of the handle's modes (Eq. 10 inputs)."""
    buf = (DnProfile * n_modes)()
    _check(lib().elasto_profile_dns(h, stream, batch, trials, buf), "elasto_profile_dns")
    return [{"latency_ms": e.latency_ms, "memory_bytes": e.memory_bytes, "gflops": e.gflops,
             "accuracy": e.accuracy} for e in buf]


def elasto_select_dn(lut: Sequence[dict], max_latency_ms: float, max_memory_bytes: float,
                     min_accuracy: float):
    """Eq. 10 through the C-ABI; None when no DN satisfies the constraints."""
    buf = (DnProfile * len(lut))()
    for i, e in enumerate(lut):
        buf[i] = DnProfile(e["latency_ms"], e["memory_bytes"], e["gflops"], e["accuracy"])
    mode = c_int(-1)
    st = lib().elasto_select_dn(buf, len(lut), max_latency_ms, max_memory_bytes, min_accuracy, ctypes.byref(mode))
    if st == ERR_BAD_MODE:
        return None
    _check(st, "elasto_select_dn")
    return mode.value


def elasto_saliency(desc: ModelDesc, tensors: Sequence[np.ndarray], n_a: int, n_b: int):
    """Compress-stage L1 saliency (scores_a, scores_b) computed on the GPU."""
    keep = _Keep()
    w = weights_struct(keep, tensors)
    a = np.zeros(n_a, np.float32)
    b = np.zeros(n_b, np.float32)
    _check(lib().elasto_saliency(ctypes.byref(desc), ctypes.byref(w), a.ctypes.data, b.ctypes.data),
           "elasto_saliency")
    return a, b


def elasto_saliency_embed(desc: ModelDesc, tensors: Sequence[np.ndarray]) -> np.ndarray:
    """L1 saliency of the ViT's embedding channels, computed on the GPU."""
    keep = _Keep()
    w = weights_struct(keep, tensors)
    e = np.zeros(desc.dim, np.float32)
    _check(lib().elasto_saliency_embed(ctypes.byref(desc), ctypes.byref(w), e.ctypes.data), "elasto_saliency_embed")
    return e


def elasto_topk(scores: np.ndarray, k: int) -> np.ndarray:
    s = np.ascontiguousarray(scores, dtype=np.float32)
    out = np.zeros(k, np.int32)
    _check(lib().elasto_topk(s.ctypes.data, len(s), k, out.ctypes.data), "elasto_topk")
    return out


def saliency_tables_vit(cfg, weights, names=None, embed_widths=None):
    """Kept tables for cfg's modes from the GPU saliency: per layer the most
    salient heads / MLP channels, and with embed_widths (one per mode, None =
    all) the most salient embedding channels; nested across modes (Eq. 8)."""
    from . import synth
    names = names or synth.vit_weight_names(cfg)
    tensors = [weights[k] for k in names]
    a, b = elasto_saliency(vit_desc(cfg, 1), tensors, cfg.layers * cfg.heads, cfg.layers * cfg.mlp)
    a = a.reshape(cfg.layers, cfg.heads)
    b = b.reshape(cfg.layers, cfg.mlp)
    tables = [{"heads": [elasto_topk(a[l], kh) for l in range(cfg.layers)],
               "mlp": [elasto_topk(b[l], kf) for l in range(cfg.layers)]}
              for kh, kf in zip(cfg.mode_heads, cfg.mode_mlp)]
    if embed_widths is not None:
        e = elasto_saliency_embed(vit_desc(cfg, 1), tensors)
        for t, k in zip(tables, embed_widths):
            t["embed"] = None if k is None else elasto_topk(e, k)
    return tables


def elasto_op_gemm(stream, A, W, bias, out, resid, M, N, K, epilogue, status=0) -> None:
    _check(lib().elasto_op_gemm(stream, A, W, bias, out, resid, M, N, K, epilogue, status), "elasto_op_gemm")


def elasto_op_conv2d(stream, x, B, H, W, C, w, N, k, stride, pad, bias, relu, out, status=0) -> None:
    _check(lib().elasto_op_conv2d(stream, x, B, H, W, C, w, N, k, stride, pad, bias, int(relu), out, status),
           "elasto_op_conv2d")


def elasto_op_layernorm(stream, x, gamma, beta, y, rows, d) -> None:
    _check(lib().elasto_op_layernorm(stream, x, gamma, beta, y, rows, d), "elasto_op_layernorm")


def elasto_op_softmax(stream, x, y, rows, cols) -> None:
    _check(lib().elasto_op_softmax(stream, x, y, rows, cols), "elasto_op_softmax")


def elasto_op_attention(stream, qkv, out, batch, n, heads, status=0) -> None:
    _check(lib().elasto_op_attention(stream, qkv, out, batch, n, heads, status), "elasto_op_attention")


def elasto_op_bounded_wait(stream, armed: bool, status, elapsed_ns) -> None:
    _check(lib().elasto_op_bounded_wait(stream, 1 if armed else 0, status, elapsed_ns), "elasto_op_bounded_wait")


def elasto_op_grid_barrier(stream, unreachable: bool, sync, status, elapsed_ns) -> None:
    _check(lib().elasto_op_grid_barrier(stream, 1 if unreachable else 0, sync, status, elapsed_ns),
           "elasto_op_grid_barrier")


# ----------------------------------------------------------------------------
# Owner object
# ----------------------------------------------------------------------------

class ElasticModel:
    """One elastic model (libelasto handle) on the current CUDA device."""

    def __init__(self, desc: ModelDesc, tensors: Sequence[np.ndarray], mode_tables, n_modes: int):
        keep = _Keep()
        self.desc = desc
        self.n_modes = n_modes
        self.handle = elasto_create(desc, tensors, mode_tables, n_modes, keep)

    @classmethod
    def vit(cls, cfg, weights: Dict[str, np.ndarray], tables, max_batch: int, names=None):
        from . import synth
        keep = _Keep()
        names = names or synth.vit_weight_names(cfg)
        mt = vit_mode_tables(keep, tables)
        return cls(vit_desc(cfg, max_batch), [weights[k] for k in names], mt, len(tables))

    @classmethod
    def resnet(cls, cfg, weights: Dict[str, np.ndarray], tables, max_batch: int):
        from . import synth
        keep = _Keep()
        mt = resnet_mode_tables(keep, tables)
        return cls(resnet_desc(cfg, max_batch), [weights[k] for k in synth.resnet_weight_names(cfg)], mt,
                   len(tables))

    def set_mode(self, mode: int) -> None:
        elasto_set_mode(self.handle, mode)

    @property
    def mode(self) -> int:
        return elasto_get_mode(self.handle)

    def forward(self, stream: int, images_ptr: int, batch: int, logits_ptr: int) -> None:
        elasto_forward(self.handle, stream, images_ptr, batch, logits_ptr)

    def forward_host(self, images: np.ndarray, logits: np.ndarray, stream: int = 0) -> None:
        elasto_forward_host(self.handle, stream, images, images.shape[0], logits)

    def forward_host_batches(self, images: List[np.ndarray], logits: List[np.ndarray], stream: int = 0) -> None:
        elasto_forward_host_batches(self.handle, stream, images, logits)

    def sync_status(self, stream: int = 0) -> None:
        elasto_sync_status(self.handle, stream)

    def check_guards(self, stream: int = 0) -> None:
        """Raise ElastoError (ERR_GUARD) if any kernel wrote past the end of
        one of the handle's device buffers."""
        elasto_check_guards(self.handle, stream)

    def query(self, what: int, mode: int = 0) -> int:
        return elasto_query(self.handle, what, mode)

    def profile(self, enable: bool) -> None:
        elasto_profile_enable(self.handle, enable)

    def set_one_launch(self, enable: bool) -> None:
        """One-image forwards as one persistent launch, or kernel by kernel (the default)."""
        elasto_set_one_launch(self.handle, enable)

    def profile_read(self) -> List[dict]:
        return elasto_profile_read(self.handle)

    def profile_dns(self, stream: int = 0, batch: int = 1, trials: int = 20) -> List[dict]:
        return elasto_profile_dns(self.handle, stream, batch, trials, self.n_modes)

    def export_packed(self, mode: int, layer: int, which: int, out: np.ndarray) -> np.ndarray:
        return elasto_debug_export_packed(self.handle, mode, layer, which, out)

    def close(self) -> None:
        if self.handle:
            elasto_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, exc_type, exc, tb):
        # a `with` block that ended normally also proves that no kernel wrote
        # past the end of a buffer of this handle
        try:
            if exc_type is None and self.handle:
                self.check_guards()
        finally:
            self.close()
