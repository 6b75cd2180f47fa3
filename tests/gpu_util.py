"""Helpers for the GPU parity tests: device transfer and the error metric.

Tolerances (normwise, per output tensor): max|x - y| / max|y| <= 1e-5 for fp32 storage and
<= 2e-2 for bf16 storage with fp32 accumulation; integer layouts must match bit for bit.
"""
import numpy as np
import pytest
import torch

TOL = {"f32": 1e-5, "bf16": 2e-2}
# bf16 tests with ReLU compare with the plain fp64 definition; biases of +-8 per column (seeded
# signs; the pre-activations' own spread is about 2) keep every pre-activation clear of the kink,
# where the kernel's decision, taken on bf16-rounded intermediates, could legitimately differ.
BF16_RELU_MARGIN = 8.0


def need_gpu():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")


def lib():
    from paper_2608_02168_gb300 import build
    build.build()
    from paper_2608_02168_gb300 import hg
    hg.lib()
    return hg


def dev(a, dtype=None):
    t = torch.from_numpy(np.ascontiguousarray(a))
    return t.to("cuda", dtype) if dtype is not None else t.to("cuda")


def tdtype(dt: str):
    return torch.float32 if dt == "f32" else torch.bfloat16


def host(t) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64) if t.is_floating_point() else t.cpu().numpy()


def relerr(x, y) -> float:
    x = np.asarray(x, np.float64)
    y = np.asarray(y, np.float64)
    return float(np.abs(x - y).max() / max(np.abs(y).max(), 1e-30)) if y.size else 0.0


def layer_params(hg, p: dict, dt: str, act="relu", layernorm=True, ln_eps=1e-5, fused=False):
    td = tdtype(dt)
    return hg.LayerParams(dev(p["W_rel"], td), dev(p["W_agg"], td), dev(p["b_agg"], td), dev(p["ln_gamma"], td),
                          dev(p["ln_beta"], td), act=act, layernorm=layernorm, ln_eps=ln_eps, fused=fused)


def grad_bufs(R, T, d):
    f = dict(dtype=torch.float32, device="cuda")
    return {"W_rel": torch.full((R, d, d), np.nan, **f), "W_agg": torch.full((T, d, d), np.nan, **f),
            "b_agg": torch.full((T, d), np.nan, **f), "ln_gamma": torch.full((T, d), np.nan, **f),
            "ln_beta": torch.full((T, d), np.nan, **f)}
