"""Pins of the CPU oracle against facts fixed by the paper and by mathematics.

Each test would fail on a plausible mistake in the oracle: a dropped term, a
wrong sign or index, a transposed operand, a mask leaking a later chunk, a roll
in the wrong direction.  None of them needs a GPU.
"""
import math

import numpy as np
import pytest
from scipy import special

import oracle as O
import workloads as WL


def tiny_wl(**over):
    base = dict(name="pin", dtype=WL.DTYPE_FP32, n_layers=2, width=32, n_q_heads=2,
                head_dim=8, mlp_dim=48, action_dim=3, n_chunks=3, chunk_tokens=4,
                batch=1, prefix_lens=[5])
    base.update(over)
    return WL.Workload(**base)


def setup(wl, recipe="unit_gate", std=0.3):
    w = WL.make_weights(wl, recipe=recipe, std=std)
    pre = WL.make_prefix_kv(wl)
    buf = WL.make_buffer(wl)
    tau = WL.make_noise_levels(wl)
    return w, pre, buf, tau


# ---------------------------------------------------------------------------
# 1. K = 1 reduces to a plain flow-matching Euler step (§3.1, Eq. 1)
# ---------------------------------------------------------------------------

def plain_flow_step(w, cfg, x, tau1, pk, pv):
    """pi0-style isolated decode step of one chunk, written independently of the
    oracle: full attention over [prefix ; chunk], one noise level, one Euler step
    from tau1 to 0.  Formulated differently on purpose (complex-number RoPE, norms
    via np.linalg.norm, joint softmax over a concatenated key matrix)."""
    W, nq, dh = cfg["width"], cfg["n_q_heads"], cfg["head_dim"]
    H, A = x.shape
    P = pk.shape[1]
    half = W // 2
    periods = cfg["t_min_period"] * np.exp(
        np.log(cfg["t_max_period"] / cfg["t_min_period"]) * np.arange(half) / (half - 1))
    ph = np.exp(1j * 2 * math.pi * float(tau1) / periods)
    emb = np.concatenate([ph.imag, ph.real])
    sig = lambda z: z * special.expit(z)
    cond = sig(w["w_t2"].astype(float) @ sig(w["w_t1"].astype(float) @ emb + w["b_t1"])
               + w["b_t2"])

    def rms(hh):
        return hh * math.sqrt(W) / np.sqrt(np.linalg.norm(hh, axis=1) ** 2 + W * cfg["rms_eps"])[:, None]

    def rot(v, pos):
        th = cfg["rope_theta"]
        freqs = th ** (-np.arange(dh // 2) * 2.0 / dh)
        z = (v[..., :dh // 2] + 1j * v[..., dh // 2:])
        shp = (len(pos),) + (1,) * (v.ndim - 2) + (dh // 2,)
        z = z * np.exp(1j * np.outer(pos, freqs)).reshape(shp)
        return np.concatenate([z.real, z.imag], axis=-1)

    h = x.astype(float) @ w["w_in"].astype(float).T + w["b_in"]
    pos = np.arange(P, P + H)
    for l, lw in enumerate(w["layers"]):
        m1 = lw["w_mod1"].astype(float) @ cond + lw["b_mod1"]
        m2 = lw["w_mod2"].astype(float) @ cond + lw["b_mod2"]
        y = rms(h) * (1 + m1[:W]) + m1[W:2 * W]
        q = rot((y @ lw["w_q"].T).reshape(H, nq, dh), pos)
        k = rot(y @ lw["w_k"].T, pos)
        v = y @ lw["w_v"].T
        keys = np.vstack([pk[l], k])
        vals = np.vstack([pv[l], v])
        logits = np.einsum("hnd,sd->hns", q, keys) / math.sqrt(dh)
        att = special.softmax(logits, axis=-1) @ vals
        h = h + m1[2 * W:] * (att.reshape(H, nq * dh) @ lw["w_o"].T)
        y2 = rms(h) * (1 + m2[:W]) + m2[W:2 * W]
        g = y2 @ lw["w_g"].T
        act = 0.5 * g * (1 + np.tanh(math.sqrt(2 / math.pi) * (g + 0.044715 * g ** 3)))
        h = h + m2[2 * W:] * ((act * (y2 @ lw["w_u"].T)) @ lw["w_d"].T)
    mf = w["w_modf"].astype(float) @ cond + w["b_modf"]
    vel = (rms(h) * (1 + mf[:W]) + mf[W:]) @ w["w_out"].T + w["b_out"]
    return x + (0.0 - float(tau1)) * vel


@pytest.mark.parametrize("tau1", [1.0, 0.37])
def test_k1_reduces_to_plain_flow_step(tau1):
    wl = tiny_wl(n_chunks=1, chunk_tokens=6)
    w, pre, buf, _ = setup(wl)
    tau = np.array([[tau1]], dtype=np.float32)
    fresh = WL.make_fresh_noise(wl, 1)[0]
    out, new, _ = O.stream_step(w, wl.as_config(), buf, tau, pre, fresh)
    ref = plain_flow_step(w, wl.as_config(), buf[0, 0], tau[0, 0], pre[0][0], pre[0][1])
    np.testing.assert_allclose(out[0], ref, rtol=1e-11, atol=1e-11)
    np.testing.assert_array_equal(new[0, 0], fresh[0])


# ---------------------------------------------------------------------------
# 2. causality (§3.1): later chunks never influence earlier ones
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("i", [0, 1])
def test_causality_bit_identical(i):
    wl = tiny_wl(n_chunks=4)
    w, pre, buf, tau = setup(wl)
    cfg = wl.as_config()
    v0 = O.expert_velocity(w, cfg, buf[0], tau[0], pre[0][0], pre[0][1])
    buf2 = buf.copy()
    tau2 = tau.copy()
    rng = np.random.default_rng(7)
    buf2[0, i + 1:] += rng.standard_normal(buf2[0, i + 1:].shape).astype(np.float32)
    tau2[0, i + 1:] = np.sort(rng.uniform(tau[0, i], 1.0, size=wl.n_chunks - i - 1))
    v1 = O.expert_velocity(w, cfg, buf2[0], tau2[0], pre[0][0], pre[0][1])
    np.testing.assert_array_equal(v0[:i + 1], v1[:i + 1])
    assert not np.allclose(v0[i + 1:], v1[i + 1:])
    # and the earlier chunks DO influence the later ones (the mask is not block-diagonal)
    buf3 = buf.copy()
    buf3[0, 0] += 1.0
    v3 = O.expert_velocity(w, cfg, buf3[0], tau[0], pre[0][0], pre[0][1])
    assert not np.allclose(v0[1:], v3[1:])


# ---------------------------------------------------------------------------
# 3. attention against brute force with an explicit per-pair mask predicate
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("P,H,K,nq,dh", [(5, 3, 3, 2, 8), (1, 2, 3, 1, 4), (0, 3, 2, 2, 6),
                                          (4, 1, 3, 3, 8)])
def test_attention_brute_force(P, H, K, nq, dh):
    rng = np.random.default_rng(P * 100 + H * 10 + K)
    T = H * K
    q = rng.standard_normal((T, nq, dh))
    kp, vp = rng.standard_normal((P, dh)), rng.standard_normal((P, dh))
    ka, va = rng.standard_normal((T, dh)), rng.standard_normal((T, dh))
    scale = 1 / math.sqrt(dh)
    got = O.chunk_causal_attention(q, kp, vp, ka, va, H, scale)
    keys = [kp[s] for s in range(P)] + [ka[s] for s in range(T)]
    vals = [vp[s] for s in range(P)] + [va[s] for s in range(T)]

    def visible(t, s):
        if s < P:
            return True
        return (s - P) // H <= t // H

    for t in range(T):
        for hh in range(nq):
            logits, vs = [], []
            for s in range(P + T):
                if visible(t, s):
                    logits.append(sum(q[t, hh, d] * keys[s][d] for d in range(dh)) * scale)
                    vs.append(vals[s])
            mx = max(logits)
            ex = [math.exp(z - mx) for z in logits]
            tot = sum(ex)
            ref = [sum(ex[j] * vs[j][d] for j in range(len(ex))) / tot for d in range(dh)]
            np.testing.assert_allclose(got[t, hh], ref, rtol=1e-12, atol=1e-12)
    # the key-limit table gives the same visible set as the predicate
    lim = O.key_limit_table(P, K, H)
    for t in range(T):
        assert lim[t] == sum(visible(t, s) for s in range(P + T))


# ---------------------------------------------------------------------------
# 4. closed form with a constant velocity field
# ---------------------------------------------------------------------------

def zero_expert(w, b):
    z = {k: (np.zeros_like(v) if isinstance(v, np.ndarray) else v) for k, v in w.items()}
    z["w_in"], z["b_in"] = w["w_in"], w["b_in"]
    z["w_t1"], z["b_t1"], z["w_t2"], z["b_t2"] = w["w_t1"], w["b_t1"], w["w_t2"], w["b_t2"]
    z["layers"] = [{k: np.zeros_like(v) for k, v in lw.items()} for lw in w["layers"]]
    z["b_out"] = b.astype(np.float32)
    return z


def test_zero_weights_closed_form():
    wl = tiny_wl(n_chunks=4, batch=2, prefix_lens=[5, 2], tau_mode="beta")
    w, pre, buf, tau = setup(wl)
    b = np.linspace(-1, 2, wl.action_dim)
    z = zero_expert(w, b)
    fresh = WL.make_fresh_noise(wl, 1)[0]
    out, new, vel = O.stream_step(z, wl.as_config(), buf, tau, pre, fresh)
    assert np.array_equal(vel, np.broadcast_to(b, vel.shape))
    dt = O.delta_t(tau)
    np.testing.assert_array_equal(out, buf[:, 0] + dt[:, 0, None, None] * b)
    np.testing.assert_array_equal(new[:, :-1], buf[:, 1:] + dt[:, 1:, None, None] * b)
    np.testing.assert_array_equal(new[:, -1], fresh)


# ---------------------------------------------------------------------------
# 5. prefix consistency: chunk i sees only chunks 1..i
# ---------------------------------------------------------------------------

def test_prefix_consistency():
    wl = tiny_wl(n_chunks=4)
    w, pre, buf, tau = setup(wl)
    cfg = wl.as_config()
    full = O.expert_velocity(w, cfg, buf[0], tau[0], pre[0][0], pre[0][1])
    for i in range(1, wl.n_chunks + 1):
        part = O.expert_velocity(w, cfg, buf[0, :i], tau[0, :i], pre[0][0], pre[0][1])
        np.testing.assert_allclose(part, full[:i], rtol=1e-12, atol=1e-12)


# ---------------------------------------------------------------------------
# 6. queue semantics over many steps (Algorithm 1, §3.2)
# ---------------------------------------------------------------------------

def test_queue_semantics_constant_velocity():
    K = 4
    wl = tiny_wl(n_chunks=K)
    w, pre, buf, tau = setup(wl)
    b = np.linspace(0.5, -0.5, wl.action_dim)
    z = zero_expert(w, b)
    S = 3 * K
    fresh = WL.make_fresh_noise(wl, S)
    state = buf.astype(np.float64)
    emitted = []
    for s in range(S):
        out, state, _ = O.stream_step(z, wl.as_config(), state, tau, pre, fresh[s])
        emitted.append(out)
    # the chunk pushed at step s is popped at step s + K after a total Euler
    # displacement of sum_k Delta t_k = -tau_K = -1: it exits as z - b (Eq. 1)
    for s in range(S - K):
        np.testing.assert_allclose(emitted[s + K], fresh[s] - b, rtol=0, atol=1e-12)
    # the initial buffer's chunk k is popped at step k after k+1 updates
    for k in range(K):
        np.testing.assert_allclose(emitted[k][0], buf[0, k] - tau[0, k] * b, atol=1e-12)


def test_flow_matching_recovers_clean_action():
    """A chunk on the interpolant x_tau = (1-tau) a + tau z with the exact velocity
    z - a lands on a when stepped from its level to 0 (Eq. 1)."""
    wl = tiny_wl(n_chunks=1)
    w, pre, buf, _ = setup(wl)
    rng = np.random.default_rng(3)
    a = rng.standard_normal((wl.chunk_tokens, wl.action_dim))
    zz = a + np.linspace(-1, 1, wl.action_dim)            # z - a = constant field b
    bvec = zz[0] - a[0]
    tau1 = 0.625
    x = ((1 - tau1) * a + tau1 * zz)[None, None].astype(np.float64)
    out, _, _ = O.stream_step(zero_expert(w, bvec), wl.as_config(), x,
                              np.array([[tau1]]), pre, np.zeros((1,) + a.shape))
    np.testing.assert_allclose(out[0], a, atol=1e-12)


# ---------------------------------------------------------------------------
# 7. primitives
# ---------------------------------------------------------------------------

def test_delta_t():
    tau = np.array([[0.1, 0.25, 0.7, 1.0]])
    dt = O.delta_t(tau)
    np.testing.assert_allclose(dt, [[-0.1, -0.15, -0.45, -0.3]], atol=1e-15)
    np.testing.assert_allclose(dt.sum(), -1.0, atol=1e-15)


def test_gelu_tanh_against_exact_gelu():
    x = np.linspace(-6, 6, 2001)
    exact = 0.5 * x * (1 + special.erf(x / math.sqrt(2)))
    assert np.max(np.abs(O.gelu_tanh(x) - exact)) < 1e-3
    np.testing.assert_allclose(O.gelu_tanh(x) - O.gelu_tanh(-x), x, atol=1e-12)
    assert O.gelu_tanh(np.array([0.0]))[0] == 0.0


def test_silu():
    x = np.linspace(-20, 20, 401)
    np.testing.assert_allclose(O.silu(x), x * special.expit(x), rtol=1e-13, atol=1e-300)


def test_rms_norm():
    rng = np.random.default_rng(0)
    h = rng.standard_normal((5, 64)) * 3
    y = O.rms_norm(h, 0.0)
    np.testing.assert_allclose(np.sqrt(np.mean(y * y, axis=1)), 1.0, rtol=1e-13)
    np.testing.assert_allclose(O.rms_norm(7 * h, 0.0), y, rtol=1e-13)
    eps = 1e-2
    np.testing.assert_allclose(O.rms_norm(h, eps),
                               h / np.sqrt((h ** 2).mean(1, keepdims=True) + eps), rtol=1e-14)


def test_rope_pairing_sign_and_relative_position():
    dh = 16
    e0 = np.zeros((1, dh))
    e0[0, 0] = 1.0
    r = O.rope(e0, np.array([1]), 1e4)
    expect = np.zeros(dh)
    expect[0], expect[dh // 2] = math.cos(1.0), math.sin(1.0)     # frequency of pair 0 is 1
    np.testing.assert_allclose(r[0], expect, atol=1e-15)
    e1 = np.zeros((1, dh))
    e1[0, 1] = 1.0
    r1 = O.rope(e1, np.array([3]), 1e4)
    ang = 3 * 1e4 ** (-2.0 / dh)
    assert abs(r1[0, 1] - math.cos(ang)) < 1e-15 and abs(r1[0, dh // 2 + 1] - math.sin(ang)) < 1e-15
    rng = np.random.default_rng(1)
    q, k = rng.standard_normal((1, dh)), rng.standard_normal((1, dh))
    for m, n, d in [(5, 2, 7), (100, 40, 13)]:
        a = O.rope(q, np.array([m]), 1e4) @ O.rope(k, np.array([n]), 1e4).T
        b = O.rope(q, np.array([m + d]), 1e4) @ O.rope(k, np.array([n + d]), 1e4).T
        np.testing.assert_allclose(a, b, rtol=1e-10)
    np.testing.assert_allclose(np.linalg.norm(O.rope(q, np.array([9]), 1e4)), np.linalg.norm(q))
    np.testing.assert_array_equal(O.rope(q, np.array([9]), 0.0), q)


def test_timestep_embedding():
    W, tmin, tmax = 16, 4e-3, 4.0
    e = O.timestep_embedding(np.array([0.0, tmin / 4, tmax / 4]), W, tmin, tmax)
    np.testing.assert_allclose(e[0], np.r_[np.zeros(W // 2), np.ones(W // 2)], atol=0)
    assert abs(e[1, 0] - 1.0) < 1e-15                  # period t_min: quarter turn
    assert abs(e[2, W // 2 - 1] - 1.0) < 1e-15         # period t_max: quarter turn


def test_philox_known_answers():
    import os
    path = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")
    n = 0
    for line in open(path):
        if line.startswith("#") or not line.strip():
            continue
        v = [int(x, 16) for x in line.split()]
        assert O.philox4x32_10(v[:4], v[4:6]) == tuple(v[6:])
        n += 1
    assert n == 3


def test_philox_tail_statistics():
    z = np.concatenate([O.philox_normal_tail(1234, s, r, 1600) for s in range(3) for r in range(2)])
    assert abs(z.mean()) < 0.05 and abs(z.var() - 1) < 0.06
    from scipy import stats
    assert stats.kstest(z, "norm").pvalue > 1e-3
    np.testing.assert_array_equal(O.philox_normal_tail(1234, 2, 1, 50),
                                  O.philox_normal_tail(1234, 2, 1, 50))
    assert not np.array_equal(O.philox_normal_tail(1234, 2, 1, 50),
                              O.philox_normal_tail(1234, 3, 1, 50))


def test_key_limits_and_chunks():
    np.testing.assert_array_equal(O.chunk_of_token(6, 2), [0, 0, 1, 1, 2, 2])
    np.testing.assert_array_equal(O.key_limit_table(10, 3, 2), [12, 12, 14, 14, 16, 16])


# ---------------------------------------------------------------------------
# 8. cold start (§3.2 "Cold start", Algorithm 1; readings R10, R11)
# ---------------------------------------------------------------------------

def test_cold_start_all_valid_is_the_steady_step():
    wl = tiny_wl(n_chunks=3, batch=2, prefix_lens=[5, 2])
    w, pre, buf, tau = setup(wl)
    fresh = WL.make_fresh_noise(wl, 1)[0]
    a = O.stream_step(w, wl.as_config(), buf, tau, pre, fresh)
    b = O.stream_step(w, wl.as_config(), buf, tau, pre, fresh, n_valid=[3, 3])
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)


@pytest.mark.parametrize("n_valid", [1, 2, 3])
def test_cold_start_padding_is_invisible(n_valid):
    """Real chunks do not depend on the padding slots' contents or noise levels."""
    K = 4
    wl = tiny_wl(n_chunks=K)
    w, pre, buf, tau = setup(wl)
    cfg = wl.as_config()
    c0 = K - n_valid
    v0 = O.expert_velocity(w, cfg, buf[0], tau[0], pre[0][0], pre[0][1], n_valid=n_valid)
    rng = np.random.default_rng(11)
    buf2, tau2 = buf.copy(), tau.copy()
    buf2[0, :c0] = 5 * rng.standard_normal(buf2[0, :c0].shape)
    tau2[0, :c0] = np.sort(rng.uniform(0.001, tau[0, c0], size=c0))
    v1 = O.expert_velocity(w, cfg, buf2[0], tau2[0], pre[0][0], pre[0][1], n_valid=n_valid)
    np.testing.assert_array_equal(v0[c0:], v1[c0:])
    # without the padding mask the same perturbation does reach the real chunks
    if c0 > 0:
        w0 = O.expert_velocity(w, cfg, buf[0], tau[0], pre[0][0], pre[0][1])
        w1 = O.expert_velocity(w, cfg, buf2[0], tau2[0], pre[0][0], pre[0][1])
        assert not np.allclose(w0[c0:], w1[c0:])


@pytest.mark.parametrize("n_valid", [1, 2, 3])
def test_cold_start_equals_shorter_buffer_without_rope(n_valid):
    """Without RoPE positions do not matter, so the real chunks of a cold-start
    buffer move exactly like a K = n_valid buffer holding only them."""
    K = 4
    wl = tiny_wl(n_chunks=K, rope_theta=0.0)
    w, pre, buf, tau = setup(wl)
    cfg = wl.as_config()
    c0 = K - n_valid
    full = O.expert_velocity(w, cfg, buf[0], tau[0], pre[0][0], pre[0][1], n_valid=n_valid)
    short = O.expert_velocity(w, cfg, buf[0, c0:], tau[0, c0:], pre[0][0], pre[0][1])
    np.testing.assert_allclose(full[c0:], short, rtol=1e-12, atol=1e-12)


@pytest.mark.parametrize("P,H,K,nq,dh,first_real,mask",
                         [(3, 2, 3, 2, 4, 1, "chunk_causal"), (0, 3, 3, 1, 4, 2, "chunk_causal"),
                          (2, 2, 3, 2, 4, 0, "block_diagonal"),
                          (0, 2, 4, 1, 6, 1, "block_diagonal")])
def test_masked_attention_brute_force(P, H, K, nq, dh, first_real, mask):
    """Padding and mask variants against an explicit per-pair predicate; rows with
    no visible key give zeros (R10)."""
    rng = np.random.default_rng(P + 10 * H + 100 * K + first_real)
    T = H * K
    q = rng.standard_normal((T, nq, dh))
    kp, vp = rng.standard_normal((P, dh)), rng.standard_normal((P, dh))
    ka, va = rng.standard_normal((T, dh)), rng.standard_normal((T, dh))
    scale = 1 / math.sqrt(dh)
    got = O.chunk_causal_attention(q, kp, vp, ka, va, H, scale, first_real, mask)

    def visible(t, s):
        if s < P:
            return True
        cs, ct = (s - P) // H, t // H
        if cs < first_real:
            return False
        return cs == ct if mask == "block_diagonal" else cs <= ct

    for t in range(T):
        for hh in range(nq):
            idx = [s for s in range(P + T) if visible(t, s)]
            if not idx:
                assert np.all(got[t, hh] == 0)
                continue
            keys = [kp[s] if s < P else ka[s - P] for s in idx]
            vals = [vp[s] if s < P else va[s - P] for s in idx]
            logits = [sum(q[t, hh, d] * kk[d] for d in range(dh)) * scale for kk in keys]
            mx = max(logits)
            ex = [math.exp(z - mx) for z in logits]
            ref = [sum(e * vv[d] for e, vv in zip(ex, vals)) / sum(ex) for d in range(dh)]
            np.testing.assert_allclose(got[t, hh], ref, rtol=1e-12, atol=1e-12)


def test_cold_start_episode_constant_velocity():
    """Algorithm 1 from an empty buffer: K-1 cold-start steps with n_valid = 1..K-1,
    then steady streaming.  The first sample z_0 is emitted at step K after exactly
    K updates (R11), i.e. as z_0 - b when tau_K = 1; every later tail likewise."""
    K = 4
    wl = tiny_wl(n_chunks=K)
    w, pre, _, tau = setup(wl)
    b = np.linspace(0.25, -0.75, wl.action_dim)
    z = zero_expert(w, b)
    S = 3 * K
    noise = WL.make_fresh_noise(wl, S + 1)
    state = np.zeros((1, K, wl.chunk_tokens, wl.action_dim))
    state[0, -1] = noise[0][0]                      # [pad, ..., pad, z_0]
    emitted = []
    for s in range(S):
        nv = [min(K, s + 1)]
        out, state, _ = O.stream_step(z, wl.as_config(), state, tau, pre, noise[s + 1], n_valid=nv)
        emitted.append(out)
    np.testing.assert_allclose(emitted[K - 1][0], noise[0][0] - b, atol=1e-12)
    for s in range(K, S):
        np.testing.assert_allclose(emitted[s][0], noise[s - K + 1][0] - b, atol=1e-12)


# ---------------------------------------------------------------------------
# 9. the no-causal (block-diagonal) ablation mask
# ---------------------------------------------------------------------------

def test_block_diagonal_chunks_are_independent_without_rope():
    """With the block-diagonal mask and no RoPE every chunk moves exactly like a
    K = 1 buffer holding it alone; with the chunk-causal mask it does not."""
    K = 3
    wl = tiny_wl(n_chunks=K, rope_theta=0.0)
    w, pre, buf, tau = setup(wl)
    cfg = dict(wl.as_config(), mask="block_diagonal")
    full = O.expert_velocity(w, cfg, buf[0], tau[0], pre[0][0], pre[0][1])
    for c in range(K):
        alone = O.expert_velocity(w, cfg, buf[0, c:c + 1], tau[0, c:c + 1], pre[0][0], pre[0][1])
        np.testing.assert_allclose(full[c], alone[0], rtol=1e-12, atol=1e-12)
    causal = O.expert_velocity(w, wl.as_config(), buf[0], tau[0], pre[0][0], pre[0][1])
    np.testing.assert_array_equal(causal[0], full[0])   # chunk 0 sees only itself either way
    assert not np.allclose(causal[1:], full[1:])
