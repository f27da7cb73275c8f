"""GPU parity: libfva's streaming step against the CPU oracle on the same seeded
inputs, through the C ABI.

Bars: emitted chunk and updated buffer within max-abs 3e-2 / rel-L2 1e-2 (bf16)
or 1e-4 (fp32); the velocity within rel-L2 2e-2 (bf16) / 1e-4 (fp32); roll, emit,
tail push and mask indices bit-exact; chunk-i velocity bit-identical when later
chunks change (causality).
"""
import numpy as np
import pytest

import oracle
import workloads as WL
from gpu_util import TOL, VEL_REL_L2, Case, assert_close, errors, split_trace

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2608_27384_gb300 as fva
    fva.lib()
    torch.cuda.set_device(0)


def check_step(case, res, ref, dtype):
    out_ref, new_ref, vel_ref = ref
    tol = TOL[dtype]
    assert_close(res["out"], out_ref, what="out", **tol)
    assert_close(res["buffer"], new_ref, what="buffer", **tol)
    if "vel" in res:
        assert_close(res["vel"], vel_ref, rel_l2=VEL_REL_L2[dtype], what="velocity")


SMALL_BF16 = {
    "base": dict(),
    "multi_split": dict(n_chunks=4, prefix_lens=[700]),
    "batch3_ragged": dict(batch=3, prefix_lens=[37, 300, 611], tau_mode="beta"),
    "nq4": dict(n_q_heads=4, width=384, mlp_dim=640, prefix_lens=[129]),
    "nq16": dict(n_q_heads=16, n_chunks=2, prefix_lens=[64]),
    "chunk7": dict(chunk_tokens=7, n_chunks=5, prefix_lens=[260]),
    "no_prefix": dict(prefix_lens=[0]),
    "one_chunk": dict(n_chunks=1, prefix_lens=[300]),
}


@pytest.mark.parametrize("name", list(SMALL_BF16))
def test_small_bf16_step(name):
    wl = WL.small_bf16_workload(**SMALL_BF16[name])
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        res = case.run(fresh=fresh)
        check_step(case, res, case.oracle_step(fresh=fresh), "bf16")
    finally:
        case.close()


@pytest.mark.parametrize("recipe", ["paper", "unit_gate"])
def test_tiny_fp32_step(recipe):
    wl = WL.standard_workloads()["tiny_fp32"]
    case = Case(wl, recipe=recipe)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        res = case.run(fresh=fresh)
        check_step(case, res, case.oracle_step(fresh=fresh), "fp32")
    finally:
        case.close()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_layer_intermediates(dtype):
    if dtype == "bf16":
        wl = WL.small_bf16_workload(n_layers=3, prefix_lens=[333])
        tol = 1.5e-2
    else:
        wl = WL.standard_workloads()["tiny_fp32"]
        tol = 2e-5
    case = Case(wl)
    try:
        for layer in range(wl.n_layers):
            res = case.run(trace_layer=layer)
            tr = split_trace(wl, res["trace"], 1)
            ref = {}
            oracle.expert_velocity(case.w, wl.as_config(), case.buf[0], case.tau[0],
                                   case.prefix[0][0], case.prefix[0][1], trace=ref,
                                   trace_layer=layer)
            T = wl.tokens
            for key in ["h_in", "y1", "q", "k", "v", "attn", "h_mid", "y2", "mlp", "h_out"]:
                r = ref[key].reshape(T, -1)
                assert_close(tr[key], r, rel_l2=tol, what=f"layer {layer} {key}")
            assert_close(tr["cond"], ref["cond"], rel_l2=tol, what="cond")
    finally:
        case.close()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_roll_emit_tail_bit_exact(dtype):
    wl = (WL.small_bf16_workload(batch=2, prefix_lens=[50, 120]) if dtype == "bf16"
          else WL.standard_workloads()["tiny_fp32"])
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        res = case.run(fresh=fresh)
        x, v = case.buf, res["vel"]
        tau = case.tau.astype(np.float32)
        prev = np.concatenate([np.zeros_like(tau[:, :1]), tau[:, :-1]], axis=1)
        dt = (prev - tau).astype(np.float32)                      # fp32 dt_k
        adv = (x + (dt[:, :, None, None] * v).astype(np.float32)).astype(np.float32)
        np.testing.assert_array_equal(res["out"], adv[:, 0])
        np.testing.assert_array_equal(res["buffer"][:, :-1], adv[:, 1:])
        np.testing.assert_array_equal(res["buffer"][:, -1], fresh)
    finally:
        case.close()


def test_mask_table_bit_exact():
    import torch
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(batch=3, chunk_tokens=7, n_chunks=4, prefix_lens=[0, 5, 213])
    case = Case(wl)
    try:
        lim = torch.full((wl.batch * wl.tokens,), -1, dtype=torch.int32, device="cuda")
        fva.fva_mask_table(case.handle, wl.batch, lim)
        torch.cuda.synchronize()
        got = lim.cpu().numpy().reshape(wl.batch, wl.tokens)
        for r, p in enumerate(wl.prefix_lens):
            np.testing.assert_array_equal(got[r], oracle.key_limit_table(p, wl.n_chunks,
                                                                         wl.chunk_tokens))
    finally:
        case.close()


@pytest.mark.parametrize("i", [0, 2])
def test_gpu_causality_bit_identical(i):
    wl = WL.small_bf16_workload(n_chunks=4, chunk_tokens=30, prefix_lens=[410])
    case = Case(wl)
    try:
        base = case.run()
        rng = np.random.default_rng(11)
        buf2 = case.buf.copy()
        buf2[0, i + 1:] += rng.standard_normal(buf2[0, i + 1:].shape).astype(np.float32)
        tau2 = case.tau.copy()
        tau2[0, i + 1:] = np.sort(rng.uniform(tau2[0, i] + 1e-3, 1.0, wl.n_chunks - i - 1))
        pert = case.run(buf=buf2, tau=tau2)
        np.testing.assert_array_equal(base["vel"][0, :i + 1], pert["vel"][0, :i + 1])
        assert not np.array_equal(base["vel"][0, i + 1:], pert["vel"][0, i + 1:])
    finally:
        case.close()


def test_graph_replay_matches_eager_bitwise():
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(batch=2, prefix_lens=[77, 505])
    g = Case(wl)
    e = Case(wl, flags=fva.FVA_FLAG_NO_GRAPH)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        a, b = g.run(fresh=fresh), e.run(fresh=fresh)
        for k in ("out", "buffer", "vel"):
            np.testing.assert_array_equal(a[k], b[k])
        a2 = g.run(fresh=fresh)  # second replay of the cached graph
        np.testing.assert_array_equal(a["out"], a2["out"])
    finally:
        g.close()
        e.close()


def test_weights_from_device_pointers():
    wl = WL.small_bf16_workload()
    a = Case(wl)
    b = Case(wl, weights_on_device=True)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        ra, rb = a.run(fresh=fresh), b.run(fresh=fresh)
        np.testing.assert_array_equal(ra["out"], rb["out"])
    finally:
        a.close()
        b.close()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_multi_step_streaming(dtype):
    """2K steps of Algorithm 1 with injected tails: every emitted chunk tracks the
    oracle run with fp64 state."""
    import torch
    import paper_2608_27384_gb300 as fva
    wl = (WL.small_bf16_workload(n_chunks=3, prefix_lens=[150]) if dtype == "bf16"
          else WL.standard_workloads()["tiny_fp32"])
    case = Case(wl)
    try:
        S = 2 * wl.n_chunks
        fresh = WL.make_fresh_noise(wl, S)
        d_buf = case.dev(case.buf)
        d_out = torch.empty((wl.batch, wl.chunk_tokens, wl.action_dim), device="cuda")
        state = case.buf.astype(np.float64)
        for s in range(S):
            d_fresh = case.dev(fresh[s])
            fva.fva_step_ex(case.handle, d_buf, case.tau, d_out, wl.batch, fresh_noise=d_fresh)
            torch.cuda.synchronize()
            out_ref, state, _ = oracle.stream_step(case.w, wl.as_config(), state, case.tau,
                                                   case.prefix, fresh[s])
            assert_close(d_out.cpu().numpy(), out_ref, what=f"step {s}", **TOL[dtype])
    finally:
        case.close()


def test_philox_tail_matches_oracle_and_resumes():
    import torch
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(batch=2, prefix_lens=[10, 20])
    seed = 0x1234ABCD5678
    case = Case(wl, noise_seed=seed)
    try:
        fva.fva_set_step_index(case.handle, 41)
        r1 = case.run(want_vel=False)
        assert fva.fva_get_step_index(case.handle) == 42
        n = wl.chunk_tokens * wl.action_dim
        for r in range(wl.batch):
            ref = oracle.philox_normal_tail(seed, 41, r, n).reshape(wl.chunk_tokens,
                                                                     wl.action_dim)
            got = r1["buffer"][r, -1]
            assert np.all(np.abs(got - ref) <= 2e-5 * (1 + np.abs(ref))), np.abs(got - ref).max()
        fva.fva_set_step_index(case.handle, 41)
        r2 = case.run(want_vel=False)
        np.testing.assert_array_equal(r1["buffer"], r2["buffer"])
        r3 = case.run(want_vel=False)  # step 42: a different tail
        assert not np.array_equal(r3["buffer"][:, -1], r1["buffer"][:, -1])
    finally:
        case.close()


def test_host_errors_leave_state_untouched():
    import torch
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(batch=2, prefix_lens=[30, 40])
    case = Case(wl)
    try:
        d_buf = case.dev(case.buf)
        d_out = torch.zeros((2, wl.chunk_tokens, wl.action_dim), device="cuda")
        before = d_buf.cpu().numpy()
        bad = case.tau.copy()
        bad[1, 1] = bad[1, 0]
        for tau, batch, status in [(bad, 2, "FVA_ERR_INVALID_ARG"),
                                   (case.tau, 3, "FVA_ERR_INVALID_ARG"),
                                   (case.tau * 2, 2, "FVA_ERR_INVALID_ARG")]:
            with pytest.raises(fva.FvaError) as e:
                fva.fva_step(case.handle, d_buf, tau, d_out, batch)
            assert e.value.name == status
        torch.cuda.synchronize()
        np.testing.assert_array_equal(d_buf.cpu().numpy(), before)
        assert float(d_out.abs().sum()) == 0.0
        # a prefix length that differs between layers of one request
        k1 = case.prefix[1][0][0, :5]
        case.dec.set_prefix(1, k1, k1, layer=0)
        with pytest.raises(fva.FvaError) as e:
            fva.fva_step(case.handle, d_buf, case.tau, d_out, 2)
        assert e.value.name == "FVA_ERR_STATE"
        fva.fva_step(case.handle, d_buf, case.tau[:1], d_out, 1)  # request 0 is still valid
    finally:
        case.close()


def test_step_before_weights_and_prefix():
    import torch
    import paper_2608_27384_gb300 as fva
    from paper_2608_27384_gb300.harness import config_for
    wl = WL.small_bf16_workload()
    h = fva.fva_create(config_for(wl))
    try:
        buf = torch.zeros((1, wl.n_chunks, wl.chunk_tokens, wl.action_dim), device="cuda")
        out = torch.zeros((1, wl.chunk_tokens, wl.action_dim), device="cuda")
        tau = WL.make_noise_levels(wl)
        with pytest.raises(fva.FvaError) as e:
            fva.fva_step(h, buf, tau, out, 1)
        assert e.value.name == "FVA_ERR_STATE"
        w = WL.make_weights(wl)
        from paper_2608_27384_gb300.harness import storage
        fva.fva_load_weights(h, [storage(t, True) for t in WL.flat_weights(wl, w)], False)
        with pytest.raises(fva.FvaError) as e:
            fva.fva_step(h, buf, tau, out, 1)
        assert e.value.name == "FVA_ERR_STATE" and "prefix" in str(e.value)
    finally:
        fva.fva_destroy(h)


def test_step_profile_matches_step_and_counts_launches():
    import torch
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(n_chunks=4, prefix_lens=[600])
    case = Case(wl)
    try:
        d_a, d_b = case.dev(case.buf), case.dev(case.buf)
        o_a = torch.empty((1, wl.chunk_tokens, wl.action_dim), device="cuda")
        o_b = torch.empty_like(o_a)
        fva.fva_set_step_index(case.handle, 5)
        fva.fva_step(case.handle, d_a, case.tau, o_a, 1)
        fva.fva_set_step_index(case.handle, 5)
        recs = fva.fva_step_profile(case.handle, d_b, case.tau, o_b, 1)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(o_a.cpu().numpy(), o_b.cpu().numpy())
        np.testing.assert_array_equal(d_a.cpu().numpy(), d_b.cpu().numpy())
        kinds = [k for k, _, _ in recs]
        L = wl.n_layers
        # the parameter fetch (which also writes the timestep embeddings), 2 time-MLP
        # layers, FiLM, embed+norm; per layer QKV, attention, split merge
        # (prefix 600 + 200 keys: 13 query tiles of 13 key blocks in splits of 2; a
        # cluster of 8 would leave its CTAs as many blocks, so the global form),
        # O-projection, norm, gate/up, down, norm (last layer: final norm); velocity
        assert kinds[0] == "params" and kinds.count("params") == 1, kinds
        assert kinds.count("attention") == L and kinds.count("attn_merge") == L, kinds
        assert kinds[-1] == "velocity" and "timestep_embed" not in kinds
        assert len(recs) == 5 + 8 * L + 1, kinds
        assert kinds[-2] == "final_norm"
        assert all(us > 0 for _, _, us in recs)
    finally:
        case.close()


def test_persistent_gemm_bitwise():
    """The persistent projections (used where a projection has at least two
    output tiles per SM) give the per-operation kernels' results bit for bit:
    the same MMAs in the same order per tile, the same epilogues.  128 requests
    of 160 tokens make every projection of this reduced expert persistent."""
    wl = WL.small_bf16_workload(batch=128, n_chunks=4, chunk_tokens=40, prefix_lens=[64] * 128)
    fresh = WL.make_fresh_noise(wl, 1)[0]
    results = {}
    import paper_2608_27384_gb300 as fva
    for mode, flags in (("persistent", 0), ("per_op", fva.FVA_FLAG_NO_PERSISTENT_GEMM)):
        case = Case(wl, flags=flags)
        try:
            results[mode] = case.run(fresh=fresh)
        finally:
            case.close()
    for key in ("out", "buffer", "vel"):
        a, b = results["persistent"][key], results["per_op"][key]
        assert np.isfinite(a).all()
        assert np.array_equal(a.view(np.uint32), b.view(np.uint32)), key


def test_attention_cluster_step():
    """A step whose attention shares each query tile's key blocks out over a
    thread-block cluster (16 query tiles of up to 17 key blocks: clusters of 6 CTAs
    with at most 3 blocks each, against splits of 4 blocks in the global form) and
    combines them in distributed shared memory, with no merge kernel: matches the
    oracle, and the step with the global form to the bf16 rounding of the split
    results."""
    import torch
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(n_chunks=5, prefix_lens=[816])
    fresh = WL.make_fresh_noise(wl, 1)[0]
    results = {}
    for mode, flags in (("cluster", 0), ("merge", fva.FVA_FLAG_NO_ATTN_CLUSTER)):
        case = Case(wl, flags=flags)
        try:
            results[mode] = case.run(fresh=fresh)
            check_step(case, results[mode], case.oracle_step(fresh=fresh), "bf16")
            d_buf = case.dev(case.buf)
            d_out = torch.empty((1, wl.chunk_tokens, wl.action_dim), device="cuda")
            kinds = [k for k, _, _ in fva.fva_step_profile(case.handle, d_buf, case.tau, d_out, 1)]
            assert kinds.count("attn_merge") == (0 if mode == "cluster" else wl.n_layers), kinds
        finally:
            case.close()
    for key in ("out", "buffer", "vel"):
        assert np.isfinite(results["cluster"][key]).all()
        assert_close(results["cluster"][key], results["merge"][key], rel_l2=5e-3,
                     what=f"cluster vs merge: {key}")


@pytest.mark.parametrize("wl_kw", [
    dict(n_chunks=4, chunk_tokens=10, prefix_lens=[200]),              # 40 rows: 48-row boxes
    dict(batch=2, n_chunks=3, chunk_tokens=8, prefix_lens=[30, 70]),   # 48 rows of two requests
    dict(n_chunks=4, chunk_tokens=20, prefix_lens=[90]),               # 80 rows: 80-row boxes
    dict(n_chunks=2, chunk_tokens=63, prefix_lens=[50]),               # 126 rows: 128-row boxes
])
def test_short_a_boxes_bitwise(wl_kw):
    """Fewer than 128 rows: the QKV and gate/up projections that load their
    activation tile through boxes of the row count rounded up to 16 (the MMA's later
    rows then read stale shared memory and are never stored) give the bits of
    128-row boxes and match the oracle."""
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(**wl_kw)
    fresh = WL.make_fresh_noise(wl, 1)[0]
    results = {}
    for mode, flags in (("short", 0), ("full", fva.FVA_FLAG_FULL_A_BOX)):
        case = Case(wl, flags=flags)
        try:
            results[mode] = case.run(fresh=fresh)
            check_step(case, results[mode], case.oracle_step(fresh=fresh), "bf16")
        finally:
            case.close()
    for key in ("out", "buffer", "vel"):
        a, b = results["short"][key], results["full"][key]
        assert np.isfinite(a).all()
        assert np.array_equal(a.view(np.uint32), b.view(np.uint32)), key


@pytest.mark.parametrize("wl_kw", [
    dict(),                                                   # 2 layers, W 256, 3 chunks
    dict(n_layers=6, width=512, mlp_dim=1024, n_chunks=10, chunk_tokens=8, prefix_lens=[200]),
    dict(n_layers=4, n_chunks=4, chunk_tokens=10, batch=2, prefix_lens=[64, 150]),
    # 800 rows: the QKV launch leaves too few SMs, the gate/up launch takes the rest
    dict(n_chunks=8, chunk_tokens=50, batch=2, prefix_lens=[64, 100]),
], ids=["L2", "L6_K10", "B2_K4", "B2_K8_gate_up"])
def test_film_overlap_matches_serial_bitwise(wl_kw):
    """FiLM modulation carried by the QKV projections (layer 0's scale / shift pair
    first, then each layer's QKV launch computing the next 6W columns in extra CTAs)
    gives the bits of the step that computes all of it before the first layer, step
    after step with new noise levels each time (a norm reading the previous step's
    modulation would differ), and both match the oracle."""
    wl = WL.small_bf16_workload(**wl_kw)
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        base = case.tau.astype(np.float64)
        for i in range(5):
            tau = (base * (0.6 + 0.1 * i)).astype(np.float32)
            res = {mode: case.run(tau=tau, fresh=fresh, serial_film=(mode == "serial"))
                   for mode in ("overlap", "serial", "overlap2")}
            for key in ("out", "buffer", "vel"):
                a = res["overlap"][key]
                assert np.isfinite(a).all()
                for other in ("serial", "overlap2"):
                    assert np.array_equal(a.view(np.uint32), res[other][key].view(np.uint32)), \
                        (i, key, other)
            if i in (0, 4):
                check_step(case, res["overlap"], case.oracle_step(tau=tau, fresh=fresh), "bf16")
    finally:
        case.close()


def test_host_buffers_step_matches_device_step():
    """fva_step_ex on pinned host buffers (the step's kernels read the buffer from and
    write the buffer and the emitted chunk to host memory over the host link) gives
    the bits of the same steps on device buffers, step after step; pageable host
    memory is refused before anything is queued."""
    import torch
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(n_chunks=3, prefix_lens=[80])
    case = Case(wl)
    try:
        fresh = case.dev(WL.make_fresh_noise(wl, 1)[0])
        d_buf = case.dev(case.buf)
        d_out = torch.empty((1, wl.chunk_tokens, wl.action_dim), device="cuda")
        h_buf = torch.from_numpy(np.ascontiguousarray(case.buf)).pin_memory()
        h_out = torch.empty((1, wl.chunk_tokens, wl.action_dim)).pin_memory()
        base = case.tau.astype(np.float64)
        for i in range(4):
            tau = (base * (0.7 + 0.1 * i)).astype(np.float32)
            fva.fva_step_ex(case.handle, d_buf, tau, d_out, 1, fresh_noise=fresh)
            fva.fva_step_ex(case.handle, h_buf, tau, h_out, 1, fresh_noise=fresh)
            torch.cuda.synchronize()
            for dev_t, host_t, what in ((d_out, h_out, "out"), (d_buf, h_buf, "buffer")):
                a = dev_t.cpu().numpy()
                b = host_t.numpy()
                assert np.isfinite(a).all()
                assert np.array_equal(a.view(np.uint32), b.view(np.uint32)), (i, what)
        pageable = torch.from_numpy(np.ascontiguousarray(case.buf))
        assert not pageable.is_pinned()
        with pytest.raises(fva.FvaError) as ei:
            fva.fva_step(case.handle, pageable, case.tau, d_out, 1)
        assert "INVALID_ARG" in str(ei.value)
        torch.cuda.synchronize()
    finally:
        case.close()


def test_step_parameters_follow_every_call():
    """Each step reads its own noise levels through the pinned ring of step
    parameters (8 slots; the step's first kernel copies the slot a device counter
    names): 20 steps on one handle with different levels each, mixing graph replays,
    kernel-by-kernel trace steps and profiled steps, every one checked against the
    oracle."""
    import torch
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(n_chunks=3, prefix_lens=[80])
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        base = case.tau.astype(np.float64)
        for i in range(20):
            # strictly increasing levels in (0, 1], different every step
            tau = (base * (0.55 + 0.45 * ((i * 7) % 20) / 19.0)).astype(np.float32)
            mode = i % 4
            if mode == 3:
                d_buf = case.dev(case.buf)
                d_out = torch.empty((1, wl.chunk_tokens, wl.action_dim), device="cuda")
                fva.fva_step_profile(case.handle, d_buf, tau, d_out, 1)
                torch.cuda.synchronize()
                res = dict(out=d_out.cpu().numpy(), buffer=d_buf.cpu().numpy())
                ref = case.oracle_step(tau=tau)  # the emitted chunk does not see the tail
                assert_close(res["out"], ref[0], what="profiled out", **TOL["bf16"])
                continue
            res = case.run(tau=tau, fresh=fresh, trace_layer=0 if mode == 2 else -1)
            check_step(case, res, case.oracle_step(tau=tau, fresh=fresh), "bf16")
    finally:
        case.close()


def test_reuse_film_matches_recomputed():
    """FVA_STEP_REUSE_FILM: with bit-identical noise levels the previous step's FiLM
    modulation is reused and the step's results are bit-identical to recomputing
    it; with other levels it is recomputed (and matches the oracle)."""
    wl = WL.small_bf16_workload(n_chunks=3, prefix_lens=[120])
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        a = case.run(fresh=fresh)
        b = case.run(fresh=fresh, reuse_film=True)
        for key in ("out", "buffer", "vel"):
            np.testing.assert_array_equal(a[key], b[key])
        tau2 = (case.tau * np.float32(0.9)).astype(np.float32)  # other levels: recomputed
        c = case.run(tau=tau2, fresh=fresh, reuse_film=True)
        check_step(case, c, case.oracle_step(tau=tau2, fresh=fresh), "bf16")
        d = case.run(tau=tau2, fresh=fresh, reuse_film=True)    # same levels again: reused
        for key in ("out", "buffer", "vel"):
            np.testing.assert_array_equal(c[key], d[key])
    finally:
        case.close()
