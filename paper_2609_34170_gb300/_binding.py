"""ctypes binding of libravel: the C ABI of include/ravel.h, same names, with
argument marshalling only (every step of the path runs in the CUDA kernels).

The library must have been built (``paper_2609_34170_gb300.build.build()``);
there is no fallback: a missing library raises on first use.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

from . import build as _build

RAVEL_FP32, RAVEL_BF16 = 0, 1
RAVEL_MASK_FULL, RAVEL_MASK_SLOT_ISOLATED = 0, 1
RAVEL_FAULT_PREFIX_LEN, RAVEL_FAULT_WITHHOLD_ARRIVAL = 1, 2

STATUS = ["RAVEL_OK", "RAVEL_EINVAL", "RAVEL_ESHAPE", "RAVEL_ENOMEM", "RAVEL_ECUDA", "RAVEL_ENOCONTEXT",
          "RAVEL_EBUSY", "RAVEL_EDEVICE", "RAVEL_ETIMEOUT", "RAVEL_ENOTREADY"]


class RavelConfig(C.Structure):
    _fields_ = [(n, C.c_int) for n in (
        "layers", "width", "n_q_heads", "n_kv_heads", "head_dim", "mlp_dim", "slots", "action_dim",
        "max_prefix", "fop_tokens", "max_batch", "dtype", "mask_mode", "fop_adapter_every", "per_robot_times")]


WEIGHT_FIELDS = ("t_w1", "t_b1", "t_w2", "t_b2", "d_w1", "d_b1", "d_w2", "d_b2", "mod_w", "mod_b",
                 "in_w", "in_b", "fop_gamma", "w_qkv", "w_o", "w_gate", "w_up", "w_down", "out_w", "out_b")


ADAPTER_FIELDS = ("a_gamma", "a_zgamma", "a_wq", "a_wkv", "a_wo", "a_gate")


class RavelWeights(C.Structure):
    _fields_ = ([(n, C.c_void_p) for n in WEIGHT_FIELDS] + [("on_device", C.c_int)]
                + [(n, C.c_void_p) for n in ADAPTER_FIELDS])


class RavelError(RuntimeError):
    def __init__(self, status: int, msg: str):
        self.status = status
        name = STATUS[status] if 0 <= status < len(STATUS) else str(status)
        super().__init__(f"{name}: {msg}")


_lib = None


def lib_path() -> str:
    return _build.LIB


def load(path: str | None = None):
    """Load libravel.so (once).  Raises OSError if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or lib_path()
    if not os.path.exists(path):
        raise OSError(f"{path} is missing: build it with paper_2609_34170_gb300.build.build()")
    L = C.CDLL(path)
    vp, i, pp = C.c_void_p, C.c_int, C.POINTER(C.c_void_p)
    sig = {
        "ravel_create": (i, [C.POINTER(RavelConfig), C.POINTER(RavelWeights), i, pp]),
        "ravel_destroy": (None, [vp]),
        "ravel_reset": (i, [vp, i, vp, vp, vp]),
        "ravel_set_context": (i, [vp, vp, vp, i, vp]),
        "ravel_set_context_robots": (i, [vp, vp, i, vp, vp, i, vp]),
        "ravel_roll_step": (i, [vp, vp, vp, vp, vp, vp, vp, vp]),
        "ravel_denoise_chunk": (i, [vp, vp, i, vp, vp, vp, vp]),
        "ravel_roll_step_rel": (i, [vp, vp, vp, vp, vp, vp, vp, vp, vp]),
        "ravel_set_relative_dims": (i, [vp, vp]),
        "ravel_get_state": (i, [vp, vp]),
        "ravel_set_state": (i, [vp, vp]),
        "ravel_step_kernel_count": (i, [vp]),
        "ravel_profile_step": (i, [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, i, vp]),
        "ravel_kernel_kind_name": (C.c_char_p, [i]),
        "ravel_gemm": (i, [vp, vp, i, i, i, vp, i, i, i, vp, i, i, vp, vp]),
        "ravel_gemm_noalloc": (i, [vp, i, i, i, vp, i, i, i, vp, i, i, vp, vp]),
        "ravel_gemm_noalloc_status": (i, [vp]),
        "ravel_debug_inject": (i, [vp, i, i, vp]),
        "ravel_status_string": (C.c_char_p, [i]),
        "ravel_last_error": (C.c_char_p, [vp]),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype, f.argtypes = res, args
    _lib = L
    return L


def _check(h, status: int, what: str):
    if status != 0:
        msg = load().ravel_last_error(h).decode() if h else ""
        raise RavelError(status, f"{what}: {msg}")


def _dptr(t, dtype=None, name="tensor"):
    """Device pointer of a contiguous CUDA tensor (or None)."""
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous CUDA tensor")
    if dtype is not None and t.dtype != dtype:
        raise ValueError(f"{name} must have dtype {dtype}, got {t.dtype}")
    return t.data_ptr()


def _stream_ptr(stream):
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream if hasattr(stream, "cuda_stream") else int(stream)


def ravel_create(cfg, weights: dict, device: int = 0, max_batch: int | None = None,
                 max_prefix: int | None = None, mask_mode: int = RAVEL_MASK_FULL):
    """cfg: an object with the ExpertConfig fields; weights: name -> float32
    array in math layout (numpy host arrays or CUDA tensors, not mixed)."""
    L = load()
    c = RavelConfig(cfg.layers, cfg.width, cfg.n_q_heads, cfg.n_kv_heads, cfg.head_dim, cfg.mlp_dim, cfg.slots,
                    cfg.action_dim, max_prefix or cfg.prefix, cfg.fop_tokens, max_batch or cfg.batch,
                    RAVEL_BF16 if cfg.dtype == "bf16" else RAVEL_FP32, mask_mode,
                    getattr(cfg, "fop_adapter_every", 0), getattr(cfg, "per_robot_times", 0))
    on_dev = None
    keep = []
    w = RavelWeights()
    for n in WEIGHT_FIELDS + ADAPTER_FIELDS:
        if n not in weights:   # adapter tensors of a network without adapters
            continue
        a = weights[n]
        if isinstance(a, np.ndarray):
            a = np.ascontiguousarray(a, dtype=np.float32)
            keep.append(a)
            ptr, dev = a.ctypes.data, False
        else:
            ptr, dev = _dptr(a, name=n), True
            keep.append(a)
        if on_dev is None:
            on_dev = dev
        elif on_dev != dev:
            raise ValueError("weights must be all host arrays or all CUDA tensors")
        setattr(w, n, ptr)
    w.on_device = int(bool(on_dev))
    h = C.c_void_p()
    st = L.ravel_create(C.byref(c), C.byref(w), device, C.byref(h))
    if st != 0:
        raise RavelError(st, "ravel_create failed (see stderr)")
    return h


def ravel_destroy(h):
    load().ravel_destroy(h)


def ravel_reset(h, batch: int, seeds, buffer, stream=None):
    seeds = np.ascontiguousarray(seeds, dtype=np.uint64)
    import torch
    _check(h, load().ravel_reset(h, batch, seeds.ctypes.data, _dptr(buffer, torch.float32, "buffer"),
                                 _stream_ptr(stream)), "ravel_reset")


def ravel_set_context(h, k, v, prefix_len: int, side_stream=None):
    _check(h, load().ravel_set_context(h, _dptr(k, name="k"), _dptr(v, name="v"), prefix_len,
                                       _stream_ptr(side_stream)), "ravel_set_context")


def ravel_set_context_robots(h, robots, k, v, prefix_len: int, side_stream=None):
    """New contexts for the listed robots only (k, v [L, len(robots), Hkv, prefix_len, hd])."""
    idx = np.ascontiguousarray(np.asarray(robots, dtype=np.int32))
    _check(h, load().ravel_set_context_robots(h, idx.ctypes.data, int(idx.size), _dptr(k, name="k"), _dptr(v, name="v"),
                                              prefix_len, _stream_ptr(side_stream)), "ravel_set_context_robots")


def ravel_roll_step(h, buffer, slot_times, obs_tokens, delta, released, velocity=None, stream=None):
    import torch
    f32 = torch.float32
    _check(h, load().ravel_roll_step(
        h, _dptr(buffer, f32, "buffer"), _dptr(slot_times, f32, "slot_times"), _dptr(obs_tokens, name="obs_tokens"),
        _dptr(delta, f32, "delta"), _dptr(released, f32, "released"), _dptr(velocity, f32, "velocity"),
        _stream_ptr(stream)), "ravel_roll_step")


def ravel_roll_step_rel(h, buffer, slot_times, obs_tokens, delta, state, released, velocity=None, stream=None):
    import torch
    f32 = torch.float32
    _check(h, load().ravel_roll_step_rel(
        h, _dptr(buffer, f32, "buffer"), _dptr(slot_times, f32, "slot_times"), _dptr(obs_tokens, name="obs_tokens"),
        _dptr(delta, f32, "delta"), _dptr(state, f32, "state"), _dptr(released, f32, "released"),
        _dptr(velocity, f32, "velocity"), _stream_ptr(stream)), "ravel_roll_step_rel")


def ravel_set_relative_dims(h, mask):
    m = np.ascontiguousarray(mask, dtype=np.float32)
    _check(h, load().ravel_set_relative_dims(h, m.ctypes.data), "ravel_set_relative_dims")


def ravel_denoise_chunk(h, chunk, n_steps: int, obs_tokens, delta, velocity=None, stream=None):
    import torch
    f32 = torch.float32
    _check(h, load().ravel_denoise_chunk(h, _dptr(chunk, f32, "chunk"), n_steps, _dptr(obs_tokens, name="obs_tokens"),
                                         _dptr(delta, f32, "delta"), _dptr(velocity, f32, "velocity"),
                                         _stream_ptr(stream)), "ravel_denoise_chunk")


def ravel_profile_step(h, buffer, slot_times, obs_tokens, delta, released, velocity=None, stream=None,
                       cap: int = 4096):
    """Eager step with per-launch timing: returns [(kind_name, ms), ...]."""
    import torch
    f32 = torch.float32
    ms = np.zeros(cap, np.float32)
    kinds = np.zeros(cap, np.int32)
    n = C.c_int(0)
    _check(h, load().ravel_profile_step(
        h, _dptr(buffer, f32, "buffer"), _dptr(slot_times, f32, "slot_times"), _dptr(obs_tokens, name="obs_tokens"),
        _dptr(delta, f32, "delta"), _dptr(released, f32, "released"), _dptr(velocity, f32, "velocity"),
        _stream_ptr(stream), ms.ctypes.data, kinds.ctypes.data, cap, C.byref(n)), "ravel_profile_step")
    k = min(n.value, cap)
    return [(load().ravel_kernel_kind_name(int(kinds[i])).decode(), float(ms[i])) for i in range(k)]


def ravel_gemm(h, X, W, epi: int, out, bias=None, K: int | None = None, stream=None):
    """out (op)= X[:, :K] @ W[:, :K]^T (+ bias) on the device; see ravel.h."""
    import torch
    M, lda = X.shape
    N, ldw = W.shape
    K = lda if K is None else K
    od = 1 if out.dtype == torch.bfloat16 else 0
    _check(h, load().ravel_gemm(h, _dptr(X, name="X"), M, K, lda, _dptr(W, name="W"), N, ldw, epi,
                                _dptr(out, name="out"), out.shape[1], od, _dptr(bias, torch.float32, "bias"),
                                _stream_ptr(stream)), "ravel_gemm")


def ravel_gemm_noalloc(X, W, epi: int, out, bias=None, K: int | None = None, stream=None):
    """ravel_gemm without a handle and without device allocation (see ravel.h)."""
    import torch
    M, lda = X.shape
    N, ldw = W.shape
    K = lda if K is None else K
    od = 1 if out.dtype == torch.bfloat16 else 0
    _check(None, load().ravel_gemm_noalloc(_dptr(X, torch.bfloat16, "X"), M, K, lda, _dptr(W, torch.bfloat16, "W"),
                                           N, ldw, epi, _dptr(out, name="out"), out.shape[1], od,
                                           _dptr(bias, torch.float32, "bias"), _stream_ptr(stream)),
           "ravel_gemm_noalloc")


def ravel_gemm_noalloc_status(stream=None) -> int:
    """Status of the allocation-free GEMM's device error word (read and
    cleared); returned as the raw ravel_status value."""
    return int(load().ravel_gemm_noalloc_status(_stream_ptr(stream)))


def ravel_debug_inject(h, fault: int, count: int = 1, stream=None):
    """Fault injection of the failure-path tests (see ravel.h)."""
    _check(h, load().ravel_debug_inject(h, fault, count, _stream_ptr(stream)), "ravel_debug_inject")


def ravel_get_state(h, batch: int) -> np.ndarray:
    out = np.zeros(batch, dtype=np.uint64)
    _check(h, load().ravel_get_state(h, out.ctypes.data), "ravel_get_state")
    return out


def ravel_set_state(h, counters):
    c = np.ascontiguousarray(counters, dtype=np.uint64)
    _check(h, load().ravel_set_state(h, c.ctypes.data), "ravel_set_state")


def ravel_step_kernel_count(h) -> int:
    return int(load().ravel_step_kernel_count(h))


def ravel_status_string(status: int) -> str:
    return load().ravel_status_string(status).decode()


def ravel_last_error(h) -> str:
    return load().ravel_last_error(h).decode()
