"""Bounded waits on the GPU, tested without a GPU fault: a kernel whose only wait
can never complete gives up after a short limit, records a timeout code in the
handle's error word and returns; the next step reports FVA_ERR_TIMEOUT once and the
step after it runs normally and correctly (the context stays usable)."""
import time

import numpy as np
import pytest

import workloads as WL
from gpu_util import TOL, Case, assert_close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def test_bounded_wait_reports_timeout_then_recovers():
    import torch
    import paper_2608_27384_gb300 as fva
    wl = WL.small_bf16_workload(n_layers=1, n_chunks=2, prefix_lens=[70])
    case = Case(wl)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        out_ref, new_ref, _ = case.oracle_step(fresh=fresh)
        first = case.run(fresh=fresh, want_vel=False)
        assert_close(first["out"], out_ref, what="before", **TOL["bf16"])

        t0 = time.perf_counter()
        fva.fva_check_bounded_wait(case.handle, 2000)  # 2 ms
        torch.cuda.synchronize()
        waited = time.perf_counter() - t0
        assert 0.002 <= waited < 1.0, waited  # the wait ran its limit, then returned

        with pytest.raises(fva.FvaError) as e:
            case.run(fresh=fresh, want_vel=False)
        assert e.value.name == "FVA_ERR_TIMEOUT"
        assert "bounded wait" in fva.fva_last_error()

        again = case.run(fresh=fresh, want_vel=False)  # reported once, then cleared
        assert_close(again["out"], out_ref, what="after", **TOL["bf16"])
        assert_close(again["buffer"], new_ref, what="after buffer", **TOL["bf16"])
        np.testing.assert_array_equal(again["out"], first["out"])

        for bad in (0, -5, 1000001):
            with pytest.raises(fva.FvaError) as e:
                fva.fva_check_bounded_wait(case.handle, bad)
            assert e.value.name == "FVA_ERR_INVALID_ARG"
    finally:
        case.close()
