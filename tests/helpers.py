"""Shared helpers of the GPU tests: seeded tensors and comparisons."""
import numpy as np
import torch

import synth


def bf16_values(x: np.ndarray) -> np.ndarray:
    return synth.to_bf16_values(np.asarray(x, dtype=np.float32))


def randn(shape, seed, scale=1.0, stream=0) -> np.ndarray:
    n = int(np.prod(shape))
    return (synth.normal(seed, stream, n) * np.float32(scale)).reshape(shape)


def dev(x: np.ndarray, dtype=None) -> torch.Tensor:
    t = torch.from_numpy(np.ascontiguousarray(x))
    if dtype is not None:
        t = t.to(dtype)
    return t.cuda()


def f64(x) -> torch.Tensor:
    if torch.is_tensor(x):
        return x.detach().cpu().to(torch.float64)
    return torch.from_numpy(np.asarray(x)).to(torch.float64)


def assert_close_scaled(got, want, rel: float, what: str = "") -> None:
    """|got - want| <= rel * max|want| element-wise (tolerance scaled to the output range)."""
    got, want = f64(got), f64(want)
    assert got.shape == want.shape, (got.shape, want.shape)
    scale = max(float(want.abs().max()), 1e-30)
    err = float((got - want).abs().max())
    assert err <= rel * scale, f"{what}: max err {err:.3e} > {rel} * {scale:.3e}"


def pixel_errors(got, want):
    d = (f64(got) - f64(want)).abs()
    return float(d.max()), float(d.mean())
