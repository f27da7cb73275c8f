"""Plain fp64 CPU oracle of FlashVLA's streaming action-decode step.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
CPU-baseline / reference legs of ``bench.py`` may import this module.  The CUDA
library never calls it and shares no code, header, table or constant with it.

What it computes (FlashVLA, arXiv 2608.27384):

* §3.1, Eq. 1 -- flow matching: x_tau = (1 - tau) a + tau z, velocity
  v = dx/dtau = z - a; tau = 1 is pure noise and tau = 0 the clean action, so a
  step from tau_k down to tau_{k-1} is the Euler update x += (tau_{k-1} - tau_k) v.
* §3.1, Eq. 2 -- the streaming buffer B_t = [x^(1)_{tau_1}, ..., x^(N)_{tau_N}]
  with tau_1 < ... < tau_N.
* §3.1 -- chunk-wise causal attention: a noisier (later) chunk attends to the
  cleaner (earlier) chunks and to itself, never to a later one.
* App. A.4 -- FiLM conditioning: each chunk's own timestep embedding produces a
  scale, a shift and a gate for every normalisation / residual branch.
* §3.2 and Algorithm 1 (steady streaming) -- one forward pass advances every
  chunk by one level, the head chunk is popped for execution, the rest shift
  forward and fresh N(0, I) noise is pushed at the tail.

Readings where the paper is silent (the CUDA library takes the same ones):

* R1/R2 tau_0 = 0: the head chunk lands exactly on the clean level.
* R3 within-chunk attention is bidirectional; every action token sees the whole
  prefix of its own request; the prefix is a fixed input.
* R4 MQA, one KV head, softmax scale 1/sqrt(head_dim).
* R5 sinusoidal timestep embedding, periods geometric in [t_min, t_max], sin half
  first, then a 2-layer SiLU MLP.
* R6 FiLM: per normalisation Linear(W -> 3W) = (scale, shift, gate); pre-norm
  modulation x (1 + scale) + shift; gated residual h += gate * branch; the final
  normalisation has (scale, shift) only.  RMSNorm has no separate learned weight.
* R7 RMSNorm eps from the config.
* R8 rotate-half RoPE with theta from the config at absolute position P_r + t;
  the prefix keys arrive already rotated; theta = 0 disables RoPE.
* R9 gated MLP with tanh-approximate GELU on the gate branch.
* R10 cold start (§3.2 "Cold start", Algorithm 1): a request whose buffer holds
  n_valid < K real chunks keeps them in the noisiest slots K-n_valid .. K-1 and
  padding in the cleaner slots; padding tokens are never keys, and their outputs
  (velocity, emitted chunk, buffer slots) are meaningless.  A query with no
  visible key at all (a padding token of a request without prefix) gets a zero
  attention output.
* R11 the queue has a fixed length: PushBack evicts the front slot during cold
  start too, so a chunk receives exactly K updates between entering at the tail
  and being emitted.
* R12 the tail chunk z is either passed in or drawn from Philox4x32-10 +
  Box-Muller (``philox_normal_tail``).
* Mask variants: "chunk_causal" (§3.1, the method) and "block_diagonal" (each
  chunk sees the prefix and itself only: the no-causal ablation of App. A.3).
* R13 expert projections have no bias; in/out projections, time MLP and FiLM do.

Parity: pinned by the tests in tests/test_oracle_pins.py (K=1 reduction to a
plain flow-matching step, causality, brute-force attention, zero-weight closed
form, prefix consistency, queue semantics, primitive identities, Philox KAT).
"""
from __future__ import annotations

import math
from typing import Dict, List, Optional, Sequence, Tuple

import numpy as np

f64 = np.float64


# ---------------------------------------------------------------------------
# scalar pieces
# ---------------------------------------------------------------------------

def delta_t(tau: np.ndarray) -> np.ndarray:
    """Per-chunk Euler step Delta t_k = tau_{k-1} - tau_k with tau_0 = 0 (Eq. 1, Alg. 1).

    tau: [..., K] strictly increasing in (0, 1].  Chunk k moves from level tau_k to
    the level of the slot in front of it; the head chunk moves to 0 (clean).
    """
    tau = np.asarray(tau, dtype=f64)
    prev = np.concatenate([np.zeros_like(tau[..., :1]), tau[..., :-1]], axis=-1)
    return prev - tau


def silu(x):
    return x / (1.0 + np.exp(-x))


def gelu_tanh(x):
    """tanh approximation of GELU."""
    return 0.5 * x * (1.0 + np.tanh(math.sqrt(2.0 / math.pi) * (x + 0.044715 * (x * x * x))))


def rms_norm(h: np.ndarray, eps: float) -> np.ndarray:
    """h / sqrt(mean(h^2) + eps) over the last axis (no learned weight, R6/R7)."""
    return h / np.sqrt(np.mean(h * h, axis=-1, keepdims=True) + eps)


def timestep_embedding(tau: np.ndarray, width: int, t_min: float, t_max: float) -> np.ndarray:
    """Sinusoidal embedding of noise levels (R5). tau [n] -> [n, width].

    Periods p_j = t_min (t_max / t_min)^(j / (width/2 - 1)), j < width/2;
    e = [sin(2 pi tau / p_j) | cos(2 pi tau / p_j)].
    """
    half = width // 2
    j = np.arange(half, dtype=f64)
    period = t_min * (t_max / t_min) ** (j / (half - 1))
    arg = 2.0 * math.pi * np.asarray(tau, dtype=f64)[:, None] / period[None, :]
    return np.concatenate([np.sin(arg), np.cos(arg)], axis=-1)


def rope(x: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotate-half RoPE (R8).  x [n, ..., dh], pos [n] integer positions.

    Pair (i, i + dh/2) is rotated by angle pos * theta^(-2 i / dh).
    """
    if theta == 0.0:
        return np.array(x, dtype=f64)
    x = np.asarray(x, dtype=f64)
    dh = x.shape[-1]
    half = dh // 2
    inv = theta ** (-2.0 * np.arange(half, dtype=f64) / dh)
    ang = np.asarray(pos, dtype=f64)[:, None] * inv[None, :]          # [n, half]
    shape = (x.shape[0],) + (1,) * (x.ndim - 2) + (half,)
    c, s = np.cos(ang).reshape(shape), np.sin(ang).reshape(shape)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


# ---------------------------------------------------------------------------
# chunk-wise causal attention (§3.1)
# ---------------------------------------------------------------------------

def chunk_of_token(n_tokens: int, chunk_tokens: int) -> np.ndarray:
    """c(t) = floor(t / H): the buffer slot (0 = cleanest) of action token t."""
    return np.arange(n_tokens) // chunk_tokens


def visible_keys(prefix_len: int, chunk: int, chunk_tokens: int, first_real: int = 0,
                 mask: str = "chunk_causal") -> Tuple[np.ndarray, np.ndarray]:
    """Explicit key index lists seen by every token of chunk ``chunk`` (§3.1, R3).

    Returns (prefix indices, action-token indices): the whole prefix, and every
    action token s with first_real <= c(s) <= chunk (own chunk bidirectional,
    earlier real chunks fully, later chunks and padding never; R10).  With
    mask="block_diagonal" only the chunk's own tokens (if it is real).
    """
    lo = chunk if mask == "block_diagonal" else first_real
    lo = max(lo, first_real)
    hi = chunk + 1
    return np.arange(prefix_len), np.arange(lo * chunk_tokens, max(lo, hi) * chunk_tokens)


def key_limit_table(prefix_len: int, n_chunks: int, chunk_tokens: int) -> np.ndarray:
    """Per action token t: number of keys in the concatenated [prefix ; action] key
    sequence that it attends to (they are always a leading range)."""
    c = chunk_of_token(n_chunks * chunk_tokens, chunk_tokens)
    return prefix_len + (c + 1) * chunk_tokens


def chunk_causal_attention(q: np.ndarray, k_pre: np.ndarray, v_pre: np.ndarray,
                           k_act: np.ndarray, v_act: np.ndarray, chunk_tokens: int,
                           scale: float, first_real: int = 0,
                           mask: str = "chunk_causal") -> np.ndarray:
    """MQA over unmasked keys only (R3, R4, R10).

    q [T, nq, dh]; k_pre/v_pre [P, dh]; k_act/v_act [T, dh] -> o [T, nq, dh].
    Each chunk's rows gather their visible keys by index and take an ordinary
    softmax over exactly those keys: masked keys never enter the sum.  Chunks
    before ``first_real`` are padding (never keys); rows without any visible key
    get zeros.
    """
    T = q.shape[0]
    o = np.zeros_like(q, dtype=f64)
    for c in range(T // chunk_tokens):
        rows = slice(c * chunk_tokens, (c + 1) * chunk_tokens)
        ip, ia = visible_keys(k_pre.shape[0], c, chunk_tokens, first_real, mask)
        if ip.size + ia.size == 0:
            continue
        keys = np.concatenate([k_pre[ip], k_act[ia]], axis=0)          # [S, dh]
        vals = np.concatenate([v_pre[ip], v_act[ia]], axis=0)
        qr = q[rows].reshape(-1, q.shape[-1])                          # [H*nq, dh]
        s = (qr @ keys.T) * scale                                        # [H*nq, S]
        s = s - s.max(axis=-1, keepdims=True)
        p = np.exp(s)
        p = p / p.sum(axis=-1, keepdims=True)
        o[rows] = (p @ vals).reshape(q[rows].shape)
    return o


# ---------------------------------------------------------------------------
# the action expert
# ---------------------------------------------------------------------------

def _w(a) -> np.ndarray:
    return np.asarray(a, dtype=f64)


def time_condition(weights: Dict, cfg: Dict, tau: np.ndarray) -> np.ndarray:
    """Per-chunk FiLM condition c_k = silu(W_t2 silu(W_t1 e_k + b_t1) + b_t2) (R5)."""
    e = timestep_embedding(tau, cfg["width"], cfg["t_min_period"], cfg["t_max_period"])
    hid = silu(e @ _w(weights["w_t1"]).T + _w(weights["b_t1"]))
    return silu(hid @ _w(weights["w_t2"]).T + _w(weights["b_t2"]))


def film(cond: np.ndarray, w, b, parts: int) -> List[np.ndarray]:
    """FiLM projection of the per-chunk condition, split into ``parts`` slices (R6)."""
    m = cond @ _w(w).T + _w(b)
    return np.split(m, parts, axis=-1)


def expert_velocity(weights: Dict, cfg: Dict, x: np.ndarray, tau: np.ndarray,
                    prefix_k: np.ndarray, prefix_v: np.ndarray,
                    trace: Optional[Dict] = None, trace_layer: int = -1,
                    n_valid: Optional[int] = None) -> np.ndarray:
    """One forward pass of the flow-matching action expert over one request's buffer.

    x [K, H, A] (slot 0 cleanest), tau [K], prefix_k/v [L, P, dh] (already rotated).
    Returns the velocity v [K, H, A] (fp64).  If ``trace`` is a dict, the inputs and
    outputs of every sub-step of layer ``trace_layer`` are stored in it.
    n_valid (R10): real chunks in slots K-n_valid .. K-1, padding before them
    (None: all K real).  cfg["mask"] selects the mask variant (default
    "chunk_causal").
    """
    K, H, A = x.shape
    T = K * H
    first_real = 0 if n_valid is None else K - int(n_valid)
    mask = cfg.get("mask", "chunk_causal")
    W, nq, dh = cfg["width"], cfg["n_q_heads"], cfg["head_dim"]
    eps = cfg["rms_eps"]
    P = prefix_k.shape[1]
    c_tok = chunk_of_token(T, H)
    pos = P + np.arange(T)
    cond = time_condition(weights, cfg, tau)                              # [K, W]

    h = _w(x).reshape(T, A) @ _w(weights["w_in"]).T + _w(weights["b_in"])
    for l, lw in enumerate(weights["layers"]):
        s1, b1, g1 = film(cond, lw["w_mod1"], lw["b_mod1"], 3)
        s2, b2, g2 = film(cond, lw["w_mod2"], lw["b_mod2"], 3)
        y = rms_norm(h, eps) * (1.0 + s1[c_tok]) + b1[c_tok]
        q = (y @ _w(lw["w_q"]).T).reshape(T, nq, dh)
        k = y @ _w(lw["w_k"]).T
        v = y @ _w(lw["w_v"]).T
        q = rope(q, pos, cfg["rope_theta"])
        k = rope(k, pos, cfg["rope_theta"])
        o = chunk_causal_attention(q, _w(prefix_k[l]), _w(prefix_v[l]), k, v, H,
                                   1.0 / math.sqrt(dh), first_real, mask)
        h_mid = h + g1[c_tok] * (o.reshape(T, nq * dh) @ _w(lw["w_o"]).T)
        y2 = rms_norm(h_mid, eps) * (1.0 + s2[c_tok]) + b2[c_tok]
        m = gelu_tanh(y2 @ _w(lw["w_g"]).T) * (y2 @ _w(lw["w_u"]).T)
        h_out = h_mid + g2[c_tok] * (m @ _w(lw["w_d"]).T)
        if trace is not None and l == trace_layer:
            trace.update(h_in=h, y1=y, q=q, k=k, v=v, attn=o.reshape(T, nq * dh),
                         h_mid=h_mid, y2=y2, mlp=m, h_out=h_out)
        h = h_out
    sF, bF = film(cond, weights["w_modf"], weights["b_modf"], 2)
    yF = rms_norm(h, eps) * (1.0 + sF[c_tok]) + bF[c_tok]
    vel = yF @ _w(weights["w_out"]).T + _w(weights["b_out"])
    if trace is not None:
        trace.update(cond=cond, h_final=h)
    return vel.reshape(K, H, A)


def stream_step(weights: Dict, cfg: Dict, buffer: np.ndarray, tau: np.ndarray,
                prefix: Sequence[Tuple[np.ndarray, np.ndarray]],
                fresh: np.ndarray, n_valid: Optional[Sequence[int]] = None
                ) -> Tuple[np.ndarray, np.ndarray, np.ndarray]:
    """One streaming step (§3.2, Algorithm 1) for a batch of requests.

    buffer [B, K, H, A]; tau [B, K]; prefix[r] = (K_r, V_r) each [L, P_r, dh];
    fresh [B, H, A] (the N(0, I) tail chunk); n_valid [B] real chunks per request
    (None: all K, steady streaming; fewer: a cold-start step, R10/R11).
    Returns (out [B, H, A], new buffer [B, K, H, A], velocity [B, K, H, A]), fp64.

    Per request: advance every chunk one level (x_k += Delta t_k v_k), pop the
    head chunk (now at tau_0 = 0) as the executable chunk, shift slots k+1 -> k,
    push ``fresh`` into the tail slot.  In a cold-start step the popped chunk is
    padding (the caller executes its default action instead).
    """
    B = buffer.shape[0]
    outs, news, vels = [], [], []
    for r in range(B):
        nv = None if n_valid is None else int(n_valid[r])
        vel = expert_velocity(weights, cfg, buffer[r], tau[r], prefix[r][0], prefix[r][1],
                              n_valid=nv)
        dt = delta_t(tau[r])
        adv = _w(buffer[r]) + dt[:, None, None] * vel
        outs.append(adv[0])
        news.append(np.concatenate([adv[1:], _w(fresh[r])[None]], axis=0))
        vels.append(vel)
    return np.stack(outs), np.stack(news), np.stack(vels)


# ---------------------------------------------------------------------------
# tail noise: Philox4x32-10 (Salmon, Moraes, Dror, Shaw, SC'11) + Box-Muller
# ---------------------------------------------------------------------------

_PHILOX_M = (0xD2511F53, 0xCD9E8D57)
_PHILOX_W = (0x9E3779B9, 0xBB67AE85)
_MASK32 = 0xFFFFFFFF


def philox4x32_10(counter: Sequence[int], key: Sequence[int]) -> Tuple[int, int, int, int]:
    """Philox4x32 with 10 rounds, written from its published definition."""
    c0, c1, c2, c3 = (int(v) & _MASK32 for v in counter)
    k0, k1 = (int(v) & _MASK32 for v in key)
    for rnd in range(10):
        if rnd:
            k0 = (k0 + _PHILOX_W[0]) & _MASK32
            k1 = (k1 + _PHILOX_W[1]) & _MASK32
        p0 = _PHILOX_M[0] * c0
        p1 = _PHILOX_M[1] * c2
        hi0, lo0 = p0 >> 32, p0 & _MASK32
        hi1, lo1 = p1 >> 32, p1 & _MASK32
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return c0, c1, c2, c3


def uniform_open0(bits: int) -> float:
    """32 random bits -> uniform in (0, 1] on a 2^-24 grid: ((bits >> 8) + 1) 2^-24."""
    return ((bits >> 8) + 1) * 2.0 ** -24


def philox_normal_tail(seed: int, step: int, request: int, n: int) -> np.ndarray:
    """The tail chunk the library draws for (seed, step, request): n N(0,1) values.

    Element e uses Philox counter (e // 4, request, step_lo, step_hi) under key
    (seed_lo, seed_hi); the four words give two Box-Muller pairs:
    z = sqrt(-2 ln u_a) * (cos 2 pi u_b, sin 2 pi u_b).
    """
    out = np.empty(n, dtype=f64)
    for g in range((n + 3) // 4):
        x = philox4x32_10((g, request, step & _MASK32, (step >> 32) & _MASK32),
                          (seed & _MASK32, (seed >> 32) & _MASK32))
        for pair in range(2):
            ua, ub = uniform_open0(x[2 * pair]), uniform_open0(x[2 * pair + 1])
            rad = math.sqrt(-2.0 * math.log(ua))
            for j, val in enumerate((rad * math.cos(2 * math.pi * ub),
                                     rad * math.sin(2 * math.pi * ub))):
                e = 4 * g + 2 * pair + j
                if e < n:
                    out[e] = val
    return out
