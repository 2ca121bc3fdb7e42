"""Shared helpers of the GPU parity tests: device setup, conversions, tolerances."""
import numpy as np
import pytest
import torch


def cuda_or_skip():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA device")
    from paper_2608_23167_gb300 import build_lib, ssm
    build_lib.build()
    ssm.lib()
    return torch.device("cuda:0")


def f64(t: torch.Tensor) -> np.ndarray:
    return t.detach().to("cpu").to(torch.float64).numpy()


def bf16_ulp(x: np.ndarray) -> np.ndarray:
    """Spacing of bfloat16 numbers at |x| (2**(e-7) for |x| in [2**e, 2**(e+1)))."""
    ax = np.abs(x)
    e = np.floor(np.log2(np.maximum(ax, 2.0 ** -126)))
    return np.ldexp(1.0, (e - 7).astype(int))


def assert_attention_close(got: np.ndarray, ref: np.ndarray, what=""):
    """The attention tolerance: max-abs <= 2e-2 and mean-abs <= 2e-3 against fp64."""
    err = np.abs(got - ref)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert err.max() <= 2e-2, f"{what}: max-abs {err.max():.3e}"
    assert err.mean() <= 2e-3, f"{what}: mean-abs {err.mean():.3e}"
    return float(err.max()), float(err.mean())


def check_device_error(expect=0):
    from paper_2608_23167_gb300 import ssm
    assert ssm.ssm_get_device_error() == expect
