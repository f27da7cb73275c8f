"""fva_chunk_attention_noalloc against fva_chunk_attention.

The no-allocation entry point serves callers that cannot allocate device memory
(a fixed-period control loop that cannot afford cudaMalloc's device
synchronisation, a host that owns all device memory through its own pool).  It
runs the same attention kernel with the library's fixed scratch array instead
of a handle's.  This file is collected last so that a stop-at-first-failure run
has run every other test before it.
"""
import numpy as np
import pytest

from gpu_util import assert_close
from test_gpu_attention import attention_inputs, make_handle, oracle_attention

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def _dev_bits(a):
    import torch
    import workloads as WL
    return torch.from_numpy(WL.bf16_bits(a).view(np.int16)).cuda()


def _to_f32(t):
    return (t.cpu().numpy().view(np.uint16).astype(np.uint32) << 16).view(np.float32)


def test_noalloc_matches_allocating_entry_point_twice_in_a_row():
    import torch
    import paper_2608_27384_gb300 as fva
    # two different calls back to back: the fixed scratch keeps the first call's
    # partials, which the second must not pick up.  Slots used: 32 tiles x 5 splits =
    # 160, then 2 requests x 32 tiles x 4 splits = 256, exactly the array's 256 slots.
    cases = [([560], 10, 50, 8, 1), ([300, 200], 10, 50, 8, 2)]
    for prefix_lens, K, H, nq, seed in cases:
        q, k, v, kv_rows = attention_inputs(prefix_lens, K, H, nq, seed=seed)
        B = len(prefix_lens)
        dq, dk, dv = _dev_bits(q), _dev_bits(k), _dev_bits(v)
        dp = torch.tensor(prefix_lens, dtype=torch.int32, device="cuda")
        out_ref = torch.full_like(dq, -1)
        out_new = torch.full_like(dq, -1)
        h = make_handle(prefix_lens, K, H, nq)
        try:
            fva.fva_chunk_attention(h, dq, dk, dv, dp, B, kv_rows, out_ref)
        finally:
            torch.cuda.synchronize()
            fva.fva_destroy(h)
        fva.fva_chunk_attention_noalloc(dq, dk, dv, dp, B, K, H, nq, 256, kv_rows, out_new)
        torch.cuda.synchronize()
        got, ref = _to_f32(out_new), _to_f32(out_ref)
        assert np.all(np.isfinite(got))
        assert_close(got, ref, max_abs=2e-2, rel_l2=1e-2, what=f"noalloc P={prefix_lens}")


@pytest.mark.parametrize("prefix_lens,K,H,nq", [
    # slots = batch * ceil(K*H*nq / 128) * ceil(kv_rows / 256)
    ([129], 3, 50, 4),           # 5 tiles x 2 splits = 10 slots
    ([300, 45], 2, 50, 16),      # 2 requests x 13 tiles x 2 splits = 52 slots
    ([560], 10, 50, 8),          # 32 tiles x 5 splits = 160 slots
])
def test_noalloc_matches_oracle(prefix_lens, K, H, nq):
    """The no-allocation entry point against the fp64 oracle directly, for several
    query-head counts (each changes the tokens per 128-row tile and the tile count)."""
    import torch
    import paper_2608_27384_gb300 as fva
    q, k, v, kv_rows = attention_inputs(prefix_lens, K, H, nq, seed=3)
    B = len(prefix_lens)
    dq, dk, dv = _dev_bits(q), _dev_bits(k), _dev_bits(v)
    dp = torch.tensor(prefix_lens, dtype=torch.int32, device="cuda")
    out = torch.full_like(dq, -1)
    for _ in range(2):  # twice in a row: the shared scratch keeps the last call's data
        fva.fva_chunk_attention_noalloc(dq, dk, dv, dp, B, K, H, nq, 256, kv_rows, out)
        torch.cuda.synchronize()
        got = _to_f32(out)
        ref = oracle_attention(q, k, v, prefix_lens, K, H, nq)
        assert_close(got, ref, max_abs=2e-2, rel_l2=1e-2, what=f"noalloc vs oracle nq={nq}")


def test_noalloc_rejects_calls_beyond_its_fixed_scratch():
    import paper_2608_27384_gb300 as fva
    # batch 4, K*H = 1000 tokens, 1024-token prefix: 4 * 63 * 8 slots > 256
    with pytest.raises(fva.FvaError) as e:
        fva.fva_chunk_attention_noalloc(16, 16, 16, 16, 4, 20, 50, 8, 256, 2024, 16)
    assert e.value.name == "FVA_ERR_INVALID_ARG"
    assert "scratch" in fva.fva_last_error()
    with pytest.raises(fva.FvaError) as e:
        fva.fva_chunk_attention_noalloc(16, 16, 16, 16, 1, 2, 8, 8, 128, 64, 16)
    assert e.value.name == "FVA_ERR_UNSUPPORTED"
