"""GPU parity of the isolated chunk-causal attention (fva_chunk_attention) against
the oracle's attention on seeded bf16 inputs."""
import math

import numpy as np
import pytest

import oracle
import workloads as WL
from gpu_util import assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def attention_inputs(prefix_lens, K, H, nq, dh=256, seed=0, kv_extra=0):
    rng = np.random.default_rng(seed)
    B, T = len(prefix_lens), K * H
    kv_rows = max(prefix_lens) + T + kv_extra
    q = WL.bf16_round(rng.standard_normal((B * T * nq, dh), dtype=np.float32))
    k = WL.bf16_round(rng.standard_normal((B, kv_rows, dh), dtype=np.float32))
    v = WL.bf16_round(rng.standard_normal((B, kv_rows, dh), dtype=np.float32))
    return q, k, v, kv_rows


def oracle_attention(q, k, v, prefix_lens, K, H, nq, dh=256):
    T = K * H
    out = []
    for r, P in enumerate(prefix_lens):
        qr = q[r * T * nq:(r + 1) * T * nq].reshape(T, nq, dh)
        o = oracle.chunk_causal_attention(qr, k[r, :P], v[r, :P], k[r, P:P + T], v[r, P:P + T], H,
                                          1.0 / math.sqrt(dh))
        out.append(o.reshape(T * nq, dh))
    return np.concatenate(out)


def make_handle(prefix_lens, K, H, nq, max_prefix=None, flags=0):
    import paper_2608_27384_gb300 as fva
    from paper_2608_27384_gb300.harness import config_for
    wl = WL.small_bf16_workload(n_q_heads=nq, n_chunks=K, chunk_tokens=H, batch=len(prefix_lens),
                                prefix_lens=list(prefix_lens))
    return fva.fva_create(config_for(wl, max_prefix=max_prefix, flags=flags))


def run_gpu_attention(handle, q, k, v, prefix_lens, kv_rows):
    import torch
    import paper_2608_27384_gb300 as fva
    B = len(prefix_lens)
    bits = lambda a: torch.from_numpy(WL.bf16_bits(a).view(np.int16)).cuda()
    dq, dk, dv = bits(q), bits(k), bits(v)
    dp = torch.tensor(prefix_lens, dtype=torch.int32, device="cuda")
    dout = torch.full_like(dq, -1)
    fva.fva_chunk_attention(handle, dq, dk, dv, dp, B, kv_rows, dout)
    torch.cuda.synchronize()
    o = dout.cpu().numpy().view(np.uint16).astype(np.uint32) << 16
    return o.view(np.float32)


@pytest.mark.parametrize("prefix_lens,K,H,nq", [
    ([560], 10, 50, 8),          # pi0.5 2-view layer
    ([816], 5, 50, 8),           # 3-view
    ([37, 300, 611], 3, 50, 8),  # ragged batch
    ([0, 5], 4, 7, 8),           # no prefix, short chunks straddling query tiles
    ([129], 3, 50, 4),           # 4 query heads
    ([4096], 10, 50, 8),         # longest prefix of the sweep
])
def test_chunk_attention_matches_oracle(prefix_lens, K, H, nq):
    import paper_2608_27384_gb300 as fva
    q, k, v, kv_rows = attention_inputs(prefix_lens, K, H, nq)
    h = make_handle(prefix_lens, K, H, nq)
    try:
        got = run_gpu_attention(h, q, k, v, prefix_lens, kv_rows)
        ref = oracle_attention(q, k, v, prefix_lens, K, H, nq)
        assert_close(got, ref, max_abs=2e-2, rel_l2=1e-2, what=f"attention P={prefix_lens}")
    finally:
        fva.fva_destroy(h)


def test_chunk_attention_rejects_bad_arguments():
    import paper_2608_27384_gb300 as fva
    h = make_handle([10], 2, 8, 8)
    try:
        with pytest.raises(fva.FvaError) as e:
            fva.fva_chunk_attention(h, 16, 16, 16, 16, 1, 10_000, 16)   # kv_rows too large
        assert e.value.name == "FVA_ERR_INVALID_ARG"
        with pytest.raises(fva.FvaError) as e:
            fva.fva_chunk_attention(h, 16, 16, 16, 16, 2, 26, 16)       # batch > max_batch
        assert e.value.name == "FVA_ERR_INVALID_ARG"
        with pytest.raises(fva.FvaError) as e:
            fva.fva_chunk_attention(h, 8, 16, 16, 16, 1, 26, 16)        # misaligned q
        assert e.value.name == "FVA_ERR_INVALID_ARG"
    finally:
        fva.fva_destroy(h)


@pytest.mark.parametrize("prefix_lens,K,H,nq", [
    ([816], 5, 50, 8),           # 16 query tiles of up to 17 key blocks: clusters of 6, 2-3 blocks each
    ([37, 300, 611], 3, 50, 8),  # 30 tiles of up to 12 blocks: clusters of 4, the short request's
                                 # tiles with fewer blocks than CTAs (some CTAs idle)
    ([129], 3, 50, 4),           # 5 tiles of 32 tokens, 5 blocks: clusters of 5, one block each
    ([700], 2, 50, 16),          # 13 tiles of 8 tokens, 13 blocks: clusters of 8
    ([5, 0], 2, 50, 2),          # 4 tiles of 64 tokens, 2 blocks: clusters of 2
])
def test_cluster_combination(prefix_lens, K, H, nq):
    """The key blocks of each query tile shared out over a thread-block cluster and
    combined in distributed shared memory: matches the oracle, and the global-scratch
    form with its merge kernel to the bf16 rounding of the split results."""
    import paper_2608_27384_gb300 as fva
    q, k, v, kv_rows = attention_inputs(prefix_lens, K, H, nq, seed=3)
    got = {}
    for name, flags in (("cluster", 0), ("global", fva.FVA_FLAG_NO_ATTN_CLUSTER)):
        h = make_handle(prefix_lens, K, H, nq, flags=flags)
        try:
            got[name] = run_gpu_attention(h, q, k, v, prefix_lens, kv_rows)
        finally:
            fva.fva_destroy(h)
    ref = oracle_attention(q, k, v, prefix_lens, K, H, nq)
    assert_close(got["cluster"], ref, max_abs=2e-2, rel_l2=1e-2, what=f"cluster P={prefix_lens}")
    assert_close(got["global"], ref, max_abs=2e-2, rel_l2=1e-2, what=f"global P={prefix_lens}")
    assert_close(got["cluster"], got["global"], max_abs=2e-2, rel_l2=5e-3,
                 what=f"cluster vs global P={prefix_lens}")
