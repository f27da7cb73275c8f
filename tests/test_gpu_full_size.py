"""Full-size parity of the five standard workloads (the shapes the benchmark
times), through the C ABI with CUDA-graph replay, against the CPU oracle on every
output element."""
import numpy as np
import pytest

import workloads as WL
from gpu_util import TOL, VEL_REL_L2, Case, assert_close

pytestmark = [pytest.mark.gpu, pytest.mark.slow]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


@pytest.mark.parametrize("name,recipe", [("tiny_fp32", "paper"), ("pi05_2view", "paper"),
                                         ("pi05_2view", "unit_gate"), ("pi05_3view", "paper"),
                                         ("serving16", "paper"), ("long_b4", "paper"),
                                         ("libero_k4h10", "paper"), ("robotwin_k4h20", "paper"),
                                         ("k5h10", "paper")])
def test_full_size_workload(name, recipe):
    wl = WL.standard_workloads()[name]
    case = Case(wl, recipe=recipe)
    try:
        fresh = WL.make_fresh_noise(wl, 1)[0]
        res = case.run(fresh=fresh)
        out_ref, new_ref, vel_ref = case.oracle_step(fresh=fresh)
        tol = TOL[wl.dtype]
        assert_close(res["out"], out_ref, what=f"{name} out", **tol)
        assert_close(res["buffer"], new_ref, what=f"{name} buffer", **tol)
        assert_close(res["vel"], vel_ref, rel_l2=VEL_REL_L2[wl.dtype], what=f"{name} velocity")
        # per request as well (a broken request must not hide in the batch norm)
        for r in range(wl.batch):
            assert_close(res["out"][r], out_ref[r], what=f"{name} out[{r}]", **tol)
    finally:
        case.close()
