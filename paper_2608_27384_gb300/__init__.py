"""Python binding of libfva, the FlashVLA streaming action-decode library.

Argument marshalling only: every function forwards to the C ABI of the same name
declared in include/fva.h and raises FvaError when it returns an error code.
All compute runs in the library's CUDA kernels; there is no Python or CPU
fallback.  Device pointers may be passed as ints or as objects with a
``data_ptr()`` method (e.g. torch tensors); streams as ints, None (legacy
default stream) or objects with ``cuda_stream``.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional, Sequence

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libfva.so")

FVA_ABI_VERSION = 1
FVA_FP32, FVA_BF16 = 0, 1
FVA_FLAG_NO_GRAPH = 1
FVA_FLAG_BLOCK_DIAGONAL = 2
FVA_FLAG_NO_PERSISTENT_GEMM = 4
FVA_FLAG_NO_ATTN_CLUSTER = 8
FVA_FLAG_FULL_A_BOX = 16
FVA_PARAM_RING = 8

STATUS = {0: "FVA_OK", 1: "FVA_ERR_INVALID_ARG", 2: "FVA_ERR_STATE", 3: "FVA_ERR_OOM",
          4: "FVA_ERR_CUDA", 5: "FVA_ERR_UNSUPPORTED", 6: "FVA_ERR_TIMEOUT"}


class FvaError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS.get(status, status)}: {message}")
        self.status = status
        self.name = STATUS.get(status, str(status))


class fva_config(ctypes.Structure):
    _fields_ = [("abi_version", ctypes.c_int32), ("dtype", ctypes.c_int32),
                ("n_layers", ctypes.c_int32), ("width", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("mlp_dim", ctypes.c_int32),
                ("action_dim", ctypes.c_int32), ("n_chunks", ctypes.c_int32),
                ("chunk_tokens", ctypes.c_int32), ("max_batch", ctypes.c_int32),
                ("max_prefix", ctypes.c_int32), ("flags", ctypes.c_uint32),
                ("rms_eps", ctypes.c_float), ("rope_theta", ctypes.c_float),
                ("t_min_period", ctypes.c_float), ("t_max_period", ctypes.c_float),
                ("noise_seed", ctypes.c_uint64)]


class fva_step_opts(ctypes.Structure):
    _fields_ = [("fresh_noise", ctypes.c_void_p), ("velocity_out", ctypes.c_void_p),
                ("trace_layer", ctypes.c_int32), ("flags", ctypes.c_uint32),
                ("trace_out", ctypes.c_void_p), ("n_valid", ctypes.c_void_p)]


class fva_kernel_time(ctypes.Structure):
    _fields_ = [("kind", ctypes.c_int32), ("layer", ctypes.c_int32),
                ("microseconds", ctypes.c_float)]


KERNEL_KINDS = ["timestep_embed", "time_mlp", "film", "embed_norm", "qkv", "attention",
                "out_proj", "resid_norm", "gate_up", "down", "final_norm", "attn_merge",
                "velocity", "params"]

EXPORTS = ["fva_create", "fva_destroy", "fva_num_weights", "fva_weight_shape",
           "fva_load_weights", "fva_set_prefix_kv", "fva_step", "fva_step_ex",
           "fva_trace_floats", "fva_set_step_index", "fva_get_step_index", "fva_mask_table",
           "fva_step_profile", "fva_chunk_attention", "fva_chunk_attention_noalloc",
           "fva_check_bounded_wait", "fva_geglu_gelu", "fva_share_prefix_kv",
           "fva_last_error"]

_lib_handle: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    """Load libfva.so (built by __graft_entry__.build()); raises if it is missing."""
    global _lib_handle
    if _lib_handle is not None:
        return _lib_handle
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is not built; run `python -c \"import __graft_entry__ as g; "
                           "g.build()\"` first (there is no fallback implementation)")
    L = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, u64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_uint64
    P = ctypes.POINTER
    sig = {
        "fva_create": (i32, [P(fva_config), P(vp)]),
        "fva_destroy": (None, [vp]),
        "fva_num_weights": (i32, [P(fva_config)]),
        "fva_weight_shape": (i32, [P(fva_config), i32, P(i64), P(i64)]),
        "fva_load_weights": (i32, [vp, P(vp), i32, i32]),
        "fva_set_prefix_kv": (i32, [vp, i32, i32, vp, vp, i32, i32, vp]),
        "fva_step": (i32, [vp, vp, P(ctypes.c_float), vp, i32, vp]),
        "fva_step_ex": (i32, [vp, vp, P(ctypes.c_float), vp, i32, P(fva_step_opts), vp]),
        "fva_trace_floats": (i64, [vp, i32]),
        "fva_set_step_index": (i32, [vp, u64]),
        "fva_get_step_index": (i32, [vp, P(u64)]),
        "fva_mask_table": (i32, [vp, i32, vp, vp]),
        "fva_check_bounded_wait": (i32, [vp, i32, vp]),
        "fva_share_prefix_kv": (i32, [vp, i32, i32, vp]),
        "fva_geglu_gelu": (i32, [vp, vp, ctypes.c_int64, vp]),
        "fva_step_profile": (i32, [vp, vp, P(ctypes.c_float), vp, i32, P(fva_kernel_time), i32,
                                   P(i32), vp]),
        "fva_chunk_attention": (i32, [vp, vp, vp, vp, vp, i32, i32, vp, vp]),
        "fva_chunk_attention_noalloc": (i32, [vp, vp, vp, vp, i32, i32, i32, i32, i32, i32, vp,
                                              vp]),
        "fva_last_error": (ctypes.c_char_p, []),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    _lib_handle = L
    return L


def fva_last_error() -> str:
    return lib().fva_last_error().decode()


def _check(status: int) -> None:
    if status != 0:
        raise FvaError(status, fva_last_error())


def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        return int(x.data_ptr())
    if isinstance(x, np.ndarray):
        return int(x.ctypes.data)
    raise TypeError(f"cannot pass {type(x)} as a pointer")


def _stream(s) -> Optional[int]:
    if s is None or isinstance(s, int):
        return s
    if hasattr(s, "cuda_stream"):
        return int(s.cuda_stream)
    raise TypeError(f"cannot pass {type(s)} as a stream")


def make_config(*, dtype: int, n_layers: int, width: int, n_q_heads: int, head_dim: int,
                mlp_dim: int, action_dim: int, n_chunks: int, chunk_tokens: int,
                max_batch: int, max_prefix: int, rms_eps: float = 1e-6,
                rope_theta: float = 1e4, t_min_period: float = 4e-3, t_max_period: float = 4.0,
                noise_seed: int = 0, flags: int = 0, n_kv_heads: int = 1,
                abi_version: int = FVA_ABI_VERSION) -> fva_config:
    return fva_config(abi_version, dtype, n_layers, width, n_q_heads, n_kv_heads, head_dim,
                      mlp_dim, action_dim, n_chunks, chunk_tokens, max_batch, max_prefix, flags,
                      rms_eps, rope_theta, t_min_period, t_max_period, noise_seed)


def fva_create(cfg: fva_config) -> int:
    h = ctypes.c_void_p()
    _check(lib().fva_create(ctypes.byref(cfg), ctypes.byref(h)))
    return h.value


def fva_destroy(handle: Optional[int]) -> None:
    lib().fva_destroy(handle)


def fva_num_weights(cfg: fva_config) -> int:
    return lib().fva_num_weights(ctypes.byref(cfg))


def fva_weight_shape(cfg: fva_config, index: int):
    r, c = ctypes.c_int64(), ctypes.c_int64()
    _check(lib().fva_weight_shape(ctypes.byref(cfg), index, ctypes.byref(r), ctypes.byref(c)))
    return r.value, c.value


def fva_load_weights(handle: int, tensors: Sequence, on_device: bool) -> None:
    arr = (ctypes.c_void_p * len(tensors))(*[_ptr(t) for t in tensors])
    _check(lib().fva_load_weights(handle, arr, len(tensors), int(bool(on_device))))


def fva_set_prefix_kv(handle: int, request: int, layer: int, k, v, length: int,
                      on_device: bool, stream=None) -> None:
    _check(lib().fva_set_prefix_kv(handle, request, layer, _ptr(k), _ptr(v), length,
                                   int(bool(on_device)), _stream(stream)))


def _tau_ptr(noise_levels):
    tau = np.ascontiguousarray(noise_levels, dtype=np.float32)
    return tau, tau.ctypes.data_as(ctypes.POINTER(ctypes.c_float))


def fva_step(handle: int, buffer, noise_levels, out_chunk, batch: int, stream=None) -> None:
    tau, tp = _tau_ptr(noise_levels)
    _check(lib().fva_step(handle, _ptr(buffer), tp, _ptr(out_chunk), batch, _stream(stream)))


FVA_STEP_REUSE_FILM = 1
FVA_STEP_SERIAL_FILM = 2


def fva_step_ex(handle: int, buffer, noise_levels, out_chunk, batch: int, fresh_noise=None,
                velocity_out=None, trace_layer: int = -1, trace_out=None, stream=None,
                n_valid=None, reuse_film: bool = False, serial_film: bool = False) -> None:
    """n_valid: per-request real chunks (cold start), a sequence of ints or None."""
    tau, tp = _tau_ptr(noise_levels)
    nv = None
    if n_valid is not None:
        import numpy as _np
        nv = _np.ascontiguousarray(n_valid, dtype=_np.int32)
    opts = fva_step_opts(_ptr(fresh_noise), _ptr(velocity_out), trace_layer,
                         (FVA_STEP_REUSE_FILM if reuse_film else 0) |
                         (FVA_STEP_SERIAL_FILM if serial_film else 0), _ptr(trace_out),
                         nv.ctypes.data if nv is not None else None)
    _check(lib().fva_step_ex(handle, _ptr(buffer), tp, _ptr(out_chunk), batch,
                             ctypes.byref(opts), _stream(stream)))


def fva_trace_floats(handle: int, batch: int) -> int:
    return lib().fva_trace_floats(handle, batch)


def fva_set_step_index(handle: int, step: int) -> None:
    _check(lib().fva_set_step_index(handle, step))


def fva_get_step_index(handle: int) -> int:
    s = ctypes.c_uint64()
    _check(lib().fva_get_step_index(handle, ctypes.byref(s)))
    return s.value


def fva_mask_table(handle: int, batch: int, key_limit, stream=None) -> None:
    _check(lib().fva_mask_table(handle, batch, _ptr(key_limit), _stream(stream)))


def fva_share_prefix_kv(handle: int, request: int, src_request: int, stream=None) -> None:
    _check(lib().fva_share_prefix_kv(handle, request, src_request, _stream(stream)))


def fva_geglu_gelu(x, y, n: int, stream=None) -> None:
    _check(lib().fva_geglu_gelu(_ptr(x), _ptr(y), n, _stream(stream)))


def fva_check_bounded_wait(handle: int, limit_us: int, stream=None) -> None:
    _check(lib().fva_check_bounded_wait(handle, limit_us, _stream(stream)))


def fva_step_profile(handle: int, buffer, noise_levels, out_chunk, batch: int, stream=None):
    """One step launched kernel by kernel with CUDA events; returns a list of
    (kind name, layer, microseconds) in launch order."""
    tau, tp = _tau_ptr(noise_levels)
    cap = 4096
    recs = (fva_kernel_time * cap)()
    n = ctypes.c_int32()
    _check(lib().fva_step_profile(handle, _ptr(buffer), tp, _ptr(out_chunk), batch, recs, cap,
                                  ctypes.byref(n), _stream(stream)))
    return [(KERNEL_KINDS[recs[i].kind], recs[i].layer, recs[i].microseconds)
            for i in range(n.value)]


def fva_chunk_attention(handle: int, q, k, v, prefix_len, batch: int, kv_rows: int, out,
                        stream=None) -> None:
    _check(lib().fva_chunk_attention(handle, _ptr(q), _ptr(k), _ptr(v), _ptr(prefix_len), batch,
                                     kv_rows, _ptr(out), _stream(stream)))


def fva_chunk_attention_noalloc(q, k, v, prefix_len, batch: int, n_chunks: int,
                                chunk_tokens: int, n_q_heads: int, head_dim: int, kv_rows: int,
                                out, stream=None) -> None:
    """fva_chunk_attention with the library's fixed scratch: allocates nothing."""
    _check(lib().fva_chunk_attention_noalloc(_ptr(q), _ptr(k), _ptr(v), _ptr(prefix_len), batch,
                                             n_chunks, chunk_tokens, n_q_heads, head_dim,
                                             kv_rows, _ptr(out), _stream(stream)))
