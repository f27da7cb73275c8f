"""Seeded synthetic inputs for the streaming action-decode step.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic.  Both the CPU oracle (through the tests and the bench's
CPU baseline) and the CUDA library consume what it returns, so the two sides
see bit-identical inputs.

The workloads stand in for the paper's pi0.5 deployments on LIBERO / RoboTwin
(§4.1, Tab. 2): no trained weights or datasets are available, so every tensor
is drawn from a fixed recipe:

* weights and biases ~ N(0, 0.02), drawn in the library's tensor order
  (``weight_names``), then rounded to bf16 (round-to-nearest-even) for the bf16
  workloads;
* prefix K and V (one observation's cached VLM keys/values, one KV head) ~ N(0, 1),
  bf16-rounded for bf16 workloads;
* the streaming buffer ~ N(0, 1) in fp32;
* noise levels: evenly spaced tau_k = k/K, or (serving workload) the Eq. 2
  staircase tau_k = 0.001 + 0.999 (k-1+u_k)/K with u_k ~ Beta(1.5, 1).

Recipe ``unit_gate`` adds 1.0 to the residual-gate slices of the FiLM biases so
that every layer's attention and MLP branch moves the residual stream by O(1);
with the plain recipe the 0.02-scale gates make the layers almost invisible in
the velocity, which would let a broken layer pass a parity test.
"""
from __future__ import annotations

import dataclasses
from typing import Dict, List, Optional

import numpy as np

DTYPE_FP32 = "fp32"
DTYPE_BF16 = "bf16"


@dataclasses.dataclass
class Workload:
    """One synthetic workload: shapes of the action expert and of the step."""

    name: str
    dtype: str
    n_layers: int
    width: int
    n_q_heads: int
    head_dim: int
    mlp_dim: int
    action_dim: int
    n_chunks: int
    chunk_tokens: int
    batch: int
    prefix_lens: List[int]
    tau_mode: str = "even"          # "even" (tau_k = k/K) or "beta" (Eq. 2 staircase)
    rms_eps: float = 1e-6
    rope_theta: float = 1e4
    t_min_period: float = 4e-3
    t_max_period: float = 4.0
    seed: int = 0
    mask: str = "chunk_causal"      # or "block_diagonal" (no-causal ablation)

    @property
    def tokens(self) -> int:
        return self.n_chunks * self.chunk_tokens

    @property
    def max_prefix(self) -> int:
        return max(self.prefix_lens) if self.prefix_lens else 0

    def as_config(self) -> Dict[str, float]:
        """Model/step configuration as plain numbers (shared field names with fva_config)."""
        return dict(
            dtype=self.dtype, n_layers=self.n_layers, width=self.width,
            n_q_heads=self.n_q_heads, head_dim=self.head_dim, mlp_dim=self.mlp_dim,
            action_dim=self.action_dim, n_chunks=self.n_chunks,
            chunk_tokens=self.chunk_tokens, rms_eps=self.rms_eps,
            rope_theta=self.rope_theta, t_min_period=self.t_min_period,
            t_max_period=self.t_max_period, mask=self.mask)


def _serving_prefix_lens(n: int, lo: int, hi: int, seed: int) -> List[int]:
    rng = np.random.default_rng(seed)
    return [int(v) for v in rng.integers(lo, hi + 1, size=n)]


def standard_workloads() -> Dict[str, Workload]:
    """The workloads of the hot-path study, by name: the five of the main study,
    then the paper's own deployment buffer shapes (App. A.1 and A.2: chunk size
    10 / 20 with buffer length 4 / 5) on the same pi0.5-sized expert."""
    expert = dict(dtype=DTYPE_BF16, n_layers=18, width=1024, n_q_heads=8, head_dim=256,
                  mlp_dim=4096, action_dim=32, chunk_tokens=50)
    return {
        # 2 layers, width 256, 4q/1kv heads of 64, MLP 1024, prefix 64, K=2 x H=8, A=7.
        "tiny_fp32": Workload("tiny_fp32", DTYPE_FP32, 2, 256, 4, 64, 1024, 7, 2, 8, 1, [64]),
        # pi0.5-shaped expert, 2 camera views: 2 x 256 image + 48 text prefix tokens.
        "pi05_2view": Workload("pi05_2view", n_chunks=10, batch=1, prefix_lens=[560], **expert),
        # 3 camera views: 3 x 256 + 48 = 816 prefix tokens, K=5.
        "pi05_3view": Workload("pi05_3view", n_chunks=5, batch=1, prefix_lens=[816], **expert),
        # 16 independent requests, ragged prefixes U[300, 900], per-request staircases.
        "serving16": Workload("serving16", n_chunks=10, batch=16,
                              prefix_lens=_serving_prefix_lens(16, 300, 900, 0),
                              tau_mode="beta", **expert),
        # Long buffer: K=20 x H=50 = 1000 action tokens, prefix 1024, batch 4.
        "long_b4": Workload("long_b4", n_chunks=20, batch=4, prefix_lens=[1024] * 4, **expert),
        # LIBERO setting: chunk size 10, buffer length 4 (40 action tokens), 2 views.
        "libero_k4h10": Workload("libero_k4h10", n_chunks=4, batch=1, prefix_lens=[560],
                                 **dict(expert, chunk_tokens=10)),
        # RoboTwin / real-robot setting: chunk size 20, buffer length 4, 3 views.
        "robotwin_k4h20": Workload("robotwin_k4h20", n_chunks=4, batch=1, prefix_lens=[816],
                                   **dict(expert, chunk_tokens=20)),
        # SmolVLA setting's buffer: chunk size 10, buffer length 5, 2 views.
        "k5h10": Workload("k5h10", n_chunks=5, batch=1, prefix_lens=[560],
                          **dict(expert, chunk_tokens=10)),
    }


def small_bf16_workload(**over) -> Workload:
    """A reduced bf16 expert that the oracle runs in well under a second but that
    still spans several GEMM / attention tiles with ragged tails."""
    base = dict(name="small_bf16", dtype=DTYPE_BF16, n_layers=2, width=256, n_q_heads=8,
                head_dim=256, mlp_dim=512, action_dim=32, n_chunks=3, chunk_tokens=50,
                batch=1, prefix_lens=[100])
    base.update(over)
    return Workload(**base)


# --------------------------------------------------------------------------
# bf16 helpers (storage format only)
# --------------------------------------------------------------------------

def bf16_round(x: np.ndarray) -> np.ndarray:
    """Round fp32 values to the nearest bf16 (ties to even); returns fp32."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    # finite inputs only: the sum stays below 2^32
    r = ((u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16))
    return (r << np.uint32(16)).view(np.float32)


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """The bf16 bit patterns (uint16) of fp32 values that are already bf16-exact."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    return (u >> 16).astype(np.uint16)


# --------------------------------------------------------------------------
# tensors
# --------------------------------------------------------------------------

GLOBAL_TENSORS = ["w_in", "b_in", "w_t1", "b_t1", "w_t2", "b_t2"]
LAYER_TENSORS = ["w_mod1", "b_mod1", "w_mod2", "b_mod2", "w_q", "w_k", "w_v", "w_o",
                 "w_g", "w_u", "w_d"]
FINAL_TENSORS = ["w_modf", "b_modf", "w_out", "b_out"]


def tensor_shapes(wl: Workload) -> Dict[str, tuple]:
    W, A, F = wl.width, wl.action_dim, wl.mlp_dim
    Dq, dh = wl.n_q_heads * wl.head_dim, wl.head_dim
    return {
        "w_in": (W, A), "b_in": (W,), "w_t1": (W, W), "b_t1": (W,), "w_t2": (W, W),
        "b_t2": (W,), "w_mod1": (3 * W, W), "b_mod1": (3 * W,), "w_mod2": (3 * W, W),
        "b_mod2": (3 * W,), "w_q": (Dq, W), "w_k": (dh, W), "w_v": (dh, W), "w_o": (W, Dq),
        "w_g": (F, W), "w_u": (F, W), "w_d": (W, F), "w_modf": (2 * W, W),
        "b_modf": (2 * W,), "w_out": (A, W), "b_out": (A,),
    }


def weight_names(n_layers: int) -> List[str]:
    """Flat tensor order used by fva_load_weights: globals, layer 0..L-1, final."""
    names = list(GLOBAL_TENSORS)
    for l in range(n_layers):
        names += [f"layers.{l}.{t}" for t in LAYER_TENSORS]
    names += FINAL_TENSORS
    return names


def make_weights(wl: Workload, recipe: str = "paper", std: float = 0.02,
                 seed: Optional[int] = None) -> Dict[str, object]:
    """Draw every weight and bias (fp32 arrays; bf16-exact for bf16 workloads).

    Returns {"w_in": ..., ..., "layers": [ {"w_q": ...}, ... ], ...}.
    """
    rng = np.random.default_rng(wl.seed if seed is None else seed)
    shapes = tensor_shapes(wl)
    W = wl.width
    out: Dict[str, object] = {"layers": [dict() for _ in range(wl.n_layers)]}
    for name in weight_names(wl.n_layers):
        key = name.split(".")[-1]
        arr = rng.standard_normal(shapes[key], dtype=np.float32) * np.float32(std)
        if recipe == "unit_gate" and key in ("b_mod1", "b_mod2"):
            arr[2 * W:3 * W] += np.float32(1.0)          # gate slice of (scale, shift, gate)
        if wl.dtype == DTYPE_BF16:
            arr = bf16_round(arr)
        if name.startswith("layers."):
            out["layers"][int(name.split(".")[1])][key] = arr
        else:
            out[key] = arr
    return out


def flat_weights(wl: Workload, weights: Dict[str, object]) -> List[np.ndarray]:
    """Weights as a list in fva_load_weights order."""
    flat = []
    for name in weight_names(wl.n_layers):
        if name.startswith("layers."):
            _, l, key = name.split(".")
            flat.append(weights["layers"][int(l)][key])
        else:
            flat.append(weights[name])
    return flat


def make_prefix_kv(wl: Workload, seed: Optional[int] = None):
    """Per request r: (K, V), each [L, P_r, head_dim] fp32 (bf16-exact for bf16)."""
    rng = np.random.default_rng((wl.seed if seed is None else seed) + 1)
    out = []
    for p in wl.prefix_lens:
        k = rng.standard_normal((wl.n_layers, p, wl.head_dim), dtype=np.float32)
        v = rng.standard_normal((wl.n_layers, p, wl.head_dim), dtype=np.float32)
        if wl.dtype == DTYPE_BF16:
            k, v = bf16_round(k), bf16_round(v)
        out.append((k, v))
    return out


def make_buffer(wl: Workload, seed: Optional[int] = None) -> np.ndarray:
    """Streaming buffer [B, K, H, A] fp32, N(0, 1)."""
    rng = np.random.default_rng((wl.seed if seed is None else seed) + 2)
    return rng.standard_normal((wl.batch, wl.n_chunks, wl.chunk_tokens, wl.action_dim),
                               dtype=np.float32)


def make_noise_levels(wl: Workload, seed: Optional[int] = None) -> np.ndarray:
    """Noise levels [B, K] fp32, strictly increasing per request, in (0, 1]."""
    K = wl.n_chunks
    if wl.tau_mode == "even":
        row = (np.arange(1, K + 1, dtype=np.float64) / K).astype(np.float32)
        return np.tile(row, (wl.batch, 1))
    rng = np.random.default_rng((wl.seed if seed is None else seed) + 3)
    u = rng.beta(1.5, 1.0, size=(wl.batch, K))
    i = np.arange(K, dtype=np.float64)[None, :]
    return (0.001 + 0.999 * (i + u) / K).astype(np.float32)


def make_fresh_noise(wl: Workload, n_steps: int, seed: Optional[int] = None) -> np.ndarray:
    """Tail chunks to inject, one per step: [S, B, H, A] fp32, N(0, 1)."""
    rng = np.random.default_rng((wl.seed if seed is None else seed) + 4)
    return rng.standard_normal((n_steps, wl.batch, wl.chunk_tokens, wl.action_dim),
                               dtype=np.float32)
