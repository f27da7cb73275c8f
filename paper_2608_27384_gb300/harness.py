"""Upload a synthetic workload (see workloads.py) into a libfva handle.

Plumbing for tests, the benchmark and smoke runs: converts host arrays to the
library's storage formats and calls the C ABI.  Holds none of the method's
arithmetic.
"""
from __future__ import annotations

from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

from . import (FVA_BF16, FVA_FLAG_BLOCK_DIAGONAL, FVA_FP32, fva_create, fva_destroy,
               fva_load_weights, fva_set_prefix_kv, make_config)


def _bits(x: np.ndarray) -> np.ndarray:
    """bf16 bit patterns of bf16-exact fp32 values."""
    return (np.ascontiguousarray(x, dtype=np.float32).view(np.uint32) >> 16).astype(np.uint16)


def storage(arr: np.ndarray, bf16: bool) -> np.ndarray:
    return _bits(arr) if bf16 else np.ascontiguousarray(arr, dtype=np.float32)


def config_for(wl, max_batch: Optional[int] = None, max_prefix: Optional[int] = None,
               flags: int = 0, noise_seed: int = 0):
    bf16 = wl.dtype == "bf16"
    if getattr(wl, "mask", "chunk_causal") == "block_diagonal":
        flags |= FVA_FLAG_BLOCK_DIAGONAL
    return make_config(dtype=FVA_BF16 if bf16 else FVA_FP32, n_layers=wl.n_layers,
                       width=wl.width, n_q_heads=wl.n_q_heads, head_dim=wl.head_dim,
                       mlp_dim=wl.mlp_dim, action_dim=wl.action_dim, n_chunks=wl.n_chunks,
                       chunk_tokens=wl.chunk_tokens,
                       max_batch=max_batch if max_batch is not None else wl.batch,
                       max_prefix=max_prefix if max_prefix is not None else wl.max_prefix,
                       rms_eps=wl.rms_eps, rope_theta=wl.rope_theta,
                       t_min_period=wl.t_min_period, t_max_period=wl.t_max_period,
                       noise_seed=noise_seed, flags=flags)


class Decoder:
    """A libfva handle with a workload's weights and prefixes installed."""

    def __init__(self, wl, flat_weights: Sequence[np.ndarray],
                 prefix: Sequence[Tuple[np.ndarray, np.ndarray]], max_batch: Optional[int] = None,
                 max_prefix: Optional[int] = None, flags: int = 0, noise_seed: int = 0,
                 weights_on_device: bool = False, stream=None):
        self.wl = wl
        self.bf16 = wl.dtype == "bf16"
        self.cfg = config_for(wl, max_batch, max_prefix, flags, noise_seed)
        self.handle = fva_create(self.cfg)
        try:
            self.load_weights(flat_weights, weights_on_device)
            for r, (k, v) in enumerate(prefix):
                self.set_prefix(r, k, v, stream=stream)
        except Exception:
            self.close()
            raise

    def load_weights(self, flat: Sequence[np.ndarray], on_device: bool = False) -> None:
        host = [storage(t, self.bf16) for t in flat]
        if on_device:
            import torch
            dev = [torch.from_numpy(h.view(np.int16) if self.bf16 else h).cuda() for h in host]
            fva_load_weights(self.handle, dev, True)
        else:
            fva_load_weights(self.handle, host, False)

    def set_prefix(self, request: int, k: np.ndarray, v: np.ndarray, layer: int = -1,
                   stream=None) -> None:
        ks, vs = storage(k, self.bf16), storage(v, self.bf16)
        length = k.shape[-2]
        fva_set_prefix_kv(self.handle, request, layer, ks, vs, length, False, stream)
        if stream is None:
            import torch
            torch.cuda.synchronize()  # host arrays are released after this call

    def close(self) -> None:
        if getattr(self, "handle", None):
            fva_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
