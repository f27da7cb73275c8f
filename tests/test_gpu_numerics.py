"""Device arithmetic whose accuracy a kernel relies on, against fp64 definitions.

The bf16 gate/up epilogue evaluates tanh(u) with the PTX tanh.approx.f32
instruction and states that the GELU it returns is within |x| 2^-12 of the exact
tanh-form GELU (before the bf16 rounding of the product)."""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    torch = pytest.importorskip("torch")
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.set_device(0)


def gelu_tanh_fp64(x):
    x = np.asarray(x, dtype=np.float64)
    return 0.5 * x * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3)))


def test_geglu_gelu_within_its_bound():
    import torch
    import paper_2608_27384_gb300 as fva
    rng = np.random.default_rng(0)
    x = np.concatenate([np.linspace(-12.0, 12.0, 200001), rng.standard_normal(100000) * 3.0,
                        np.array([0.0, -0.0, 1e-30, -1e-30, 40.0, -40.0, 1e4, -1e4])])
    x = x.astype(np.float32)
    dx = torch.from_numpy(x).cuda()
    dy = torch.empty_like(dx)
    fva.fva_geglu_gelu(dx, dy, x.size)
    torch.cuda.synchronize()
    y = dy.cpu().numpy().astype(np.float64)
    ref = gelu_tanh_fp64(x)
    err = np.abs(y - ref)
    bound = np.abs(x.astype(np.float64)) * 2.0 ** -12 + np.abs(ref) * 2.0 ** -22
    worst = float(np.max(err / np.maximum(bound, 1e-300)))
    print(f"geglu gelu: max |err| = {err.max():.3e}, max err / bound = {worst:.3f}")
    assert np.all(np.isfinite(y))
    assert np.all(err <= bound), worst
