"""GPU parity of the cold-start steps (padding chunks, Algorithm 1) and of the
block-diagonal mask variant, through the C ABI, against the CPU oracle.

Only real chunks are compared: the velocity of slots K-n_valid .. K-1, the
updated buffer slots they move into, and the emitted chunk once it is real.
"""
import numpy as np
import pytest

import workloads as WL
from gpu_util import TOL, VEL_REL_L2, Case, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import paper_2608_27384_gb300 as fva
    fva.lib()
    torch.cuda.set_device(0)


def _workload(dtype, **over):
    if dtype == "bf16":
        base = dict(n_chunks=4, prefix_lens=[300])
        base.update(over)
        return WL.small_bf16_workload(**base)
    wl = WL.standard_workloads()["tiny_fp32"]
    d = dict(wl.__dict__)
    d.update(dict(n_chunks=4, prefix_lens=[40]))
    d.update(over)
    return WL.Workload(**d)


def check_real(res, ref, n_valid, K, dtype):
    out_ref, new_ref, vel_ref = ref
    tol = TOL[dtype]
    for r, nv in enumerate(n_valid):
        c0 = K - nv
        assert np.all(np.isfinite(res["vel"][r, c0:]))
        assert_close(res["vel"][r, c0:], vel_ref[r, c0:], rel_l2=VEL_REL_L2[dtype],
                     what=f"velocity r={r} n_valid={nv}")
        lo = max(0, c0 - 1)  # slot c moves to c - 1; the tail slot takes the fresh chunk
        assert_close(res["buffer"][r, lo:], new_ref[r, lo:], what=f"buffer r={r}", **tol)
        if nv == K:
            assert_close(res["out"][r], out_ref[r], what=f"out r={r}", **tol)


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
@pytest.mark.parametrize("n_valid", [[1], [2], [3], [4]])
def test_cold_start_step(dtype, n_valid):
    wl = _workload(dtype)
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        res = case.run(fresh=fresh, n_valid=n_valid)
        check_real(res, case.oracle_step(fresh=fresh, n_valid=n_valid), n_valid, wl.n_chunks, dtype)
    finally:
        case.close()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_cold_start_ragged_batch(dtype):
    """One launch, three requests at different cold-start stages and prefixes,
    one of them without any prefix (its padding queries see no key at all)."""
    prefixes = [0, 37, 280] if dtype == "bf16" else [0, 9, 40]
    wl = _workload(dtype, batch=3, prefix_lens=prefixes, tau_mode="beta")
    n_valid = [1, 3, 2]
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        res = case.run(fresh=fresh, n_valid=n_valid)
        check_real(res, case.oracle_step(fresh=fresh, n_valid=n_valid), n_valid, wl.n_chunks, dtype)
    finally:
        case.close()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_padding_is_invisible_bitwise(dtype):
    """Changing the padding slots' contents and noise levels leaves every real
    chunk's velocity bit-identical on the GPU."""
    wl = _workload(dtype)
    K, nv = wl.n_chunks, 2
    c0 = K - nv
    case = Case(wl)
    try:
        a = case.run(n_valid=[nv])
        rng = np.random.default_rng(5)
        buf2, tau2 = case.buf.copy(), case.tau.copy()
        buf2[0, :c0] = 4 * rng.standard_normal(buf2[0, :c0].shape).astype(np.float32)
        tau2[0, :c0] = np.sort(rng.uniform(0.001, case.tau[0, c0], size=c0)).astype(np.float32)
        b = case.run(buf=buf2, tau=tau2, n_valid=[nv])
        np.testing.assert_array_equal(a["vel"][0, c0:], b["vel"][0, c0:])
        c = case.run(buf=buf2, tau=tau2)          # without the padding mask it leaks
        assert not np.array_equal(a["vel"][0, c0:], c["vel"][0, c0:])
    finally:
        case.close()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_cold_start_episode(dtype):
    """Algorithm 1 from [pad, ..., pad, z_0]: K-1 cold-start steps with n_valid =
    1 .. K-1, then steady steps; GPU and oracle run the same sequence with the
    same injected tails, and every real chunk they emit agrees."""
    wl = _workload(dtype, n_chunks=3)
    K = wl.n_chunks
    case = Case(wl)
    try:
        noise = WL.make_fresh_noise(wl, K + 3)
        g = np.zeros_like(case.buf)
        g[0, -1] = noise[0][0]
        o = g.astype(np.float64)
        for s in range(K + 2):
            nv = [min(K, s + 1)]
            res = case.run(buf=g, fresh=noise[s + 1], n_valid=nv)
            out_ref, o, _ = case.oracle_step(buf=o, fresh=noise[s + 1], n_valid=nv)
            g = res["buffer"]
            real = max(0, K - nv[0] - 1)
            assert_close(g[0, real:], o[0, real:], what=f"buffer step {s}", **TOL[dtype])
            if nv[0] == K:
                assert_close(res["out"], out_ref, what=f"emitted step {s}", **TOL[dtype])
    finally:
        case.close()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_block_diagonal_mask(dtype):
    wl = _workload(dtype, mask="block_diagonal", n_chunks=3)
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        res = case.run(fresh=fresh)
        out_ref, new_ref, vel_ref = case.oracle_step(fresh=fresh)
        assert_close(res["out"], out_ref, what="out", **TOL[dtype])
        assert_close(res["buffer"], new_ref, what="buffer", **TOL[dtype])
        assert_close(res["vel"], vel_ref, rel_l2=VEL_REL_L2[dtype], what="velocity")
    finally:
        case.close()


def test_multi_buffer_forward():
    """The packed multi-buffer forward (§3.3, App. A.4): the N cold-start
    configurations of one observation, [pad x (N-j), j real chunks] for j = 1..N,
    reading one shared prefix K/V (fva_share_prefix_kv) and isolated from each
    other, in one launch as a batch of N requests.  Each configuration matches the
    oracle, and equals running it alone bit for bit (no cross-buffer interaction)."""
    K = 3
    base = _workload("bf16", n_chunks=K)
    wl = WL.Workload(**dict(base.__dict__, batch=K, prefix_lens=[base.prefix_lens[0]] * K))
    case = Case(wl)
    try:
        import paper_2608_27384_gb300 as fva
        buf = np.repeat(case.buf[:1], K, axis=0)              # the same future chunks...
        pre = [case.prefix[0]] * K                            # ...and the same observation,
        for r in range(1, K):                                 # read from request 0's rows
            fva.fva_share_prefix_kv(case.handle, r, 0)
        case.prefix = pre
        n_valid = list(range(1, K + 1))
        fresh = WL.make_fresh_noise(wl, 1)[0]
        res = case.run(buf=buf, fresh=fresh, n_valid=n_valid)
        check_real(res, case.oracle_step(buf=buf, fresh=fresh, n_valid=n_valid), n_valid, K, "bf16")
        for r in range(K):
            alone = case.run(buf=buf[r:r + 1], fresh=fresh[r:r + 1], n_valid=[n_valid[r]], batch=1)
            c0 = K - n_valid[r]
            np.testing.assert_array_equal(res["vel"][r, c0:], alone["vel"][0, c0:])
    finally:
        case.close()


@pytest.mark.parametrize("dtype", ["bf16", "fp32"])
def test_shared_prefix_equals_separate_copies(dtype):
    """A request reading another's prefix (fva_share_prefix_kv) gives the same
    results bit for bit as the same prefix uploaded into its own rows; setting the
    source's prefix again drops the share."""
    import paper_2608_27384_gb300 as fva
    base = _workload(dtype, n_chunks=3)
    P = 150 if dtype == "bf16" else base.prefix_lens[0]  # 150 = 2 x 64 + a 22-key tail
    wl = WL.Workload(**dict(base.__dict__, batch=3, prefix_lens=[P] * 3))
    case = Case(wl)
    try:
        buf = case.buf
        fresh = WL.make_fresh_noise(wl, 1)[0]
        for r in range(3):                           # separate copies of request 0's prefix
            case.dec.set_prefix(r, case.prefix[0][0], case.prefix[0][1])
        sep = case.run(buf=buf, fresh=fresh)
        for r in (1, 2):                             # the same prefix, shared
            fva.fva_share_prefix_kv(case.handle, r, 0)
        shr = case.run(buf=buf, fresh=fresh)
        for key in ("out", "buffer", "vel"):
            np.testing.assert_array_equal(sep[key], shr[key])
        case.prefix = [case.prefix[0]] * 3
        out_ref, new_ref, _ = case.oracle_step(buf=buf, fresh=fresh)
        tol = TOL[dtype]
        assert_close(shr["out"], out_ref, what="shared out", **tol)
        assert_close(shr["buffer"], new_ref, what="shared buffer", **tol)
        with pytest.raises(fva.FvaError) as e:
            fva.fva_share_prefix_kv(case.handle, 1, 1)
        assert e.value.name == "FVA_ERR_INVALID_ARG"
        with pytest.raises(fva.FvaError) as e:
            fva.fva_share_prefix_kv(case.handle, 0, 1)    # 1 itself shares 0's prefix
        assert e.value.name == "FVA_ERR_STATE"
        case.dec.set_prefix(0, case.prefix[0][0], case.prefix[0][1])  # drops the shares
        with pytest.raises(fva.FvaError) as e:
            case.run(buf=buf, fresh=fresh)
        assert e.value.name == "FVA_ERR_STATE"
    finally:
        case.close()
