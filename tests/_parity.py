"""Shared helpers for the GPU parity tests (comparison rules, oracle runs)."""
import numpy as np
import torch

import oracle as O

GRAD_RTOL = 1e-4   # decoded / chunk gradients: ||gpu - ref||_inf / ||ref||_inf
MSE_RTOL = 1e-3    # error measures, relative
COEF_RTOL = 1e-9   # fp64 coefficients (Algorithm 1), relative to ||ref||_inf


def rel_inf(a, b):
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.max(np.abs(b)) if b.size else 0.0
    num = np.max(np.abs(a - b)) if a.size else 0.0
    if den == 0.0:
        return 0.0 if num == 0.0 else np.inf
    return num / den


def assert_grad_close(gpu, ref, what=""):
    r = rel_inf(gpu, ref)
    assert r <= GRAD_RTOL, f"{what}: relative inf-norm error {r:.3e} > {GRAD_RTOL}"


def assert_mse_close(gpu, ref, floor, what=""):
    """Relative 1e-3 above the floor; below it both sides must stay under it
    (exact patterns give rounding-level values)."""
    if ref > floor:
        r = abs(gpu - ref) / ref
        assert r <= MSE_RTOL, f"{what}: mse {gpu:.6e} vs {ref:.6e} (rel {r:.2e})"
    else:
        assert gpu <= floor, f"{what}: mse {gpu:.3e} above floor {floor:.3e} (ref {ref:.3e})"


def to_np(t):
    return t.detach().cpu().numpy()


def dev_tensors(R, order, psi, device="cuda"):
    return (torch.from_numpy(np.ascontiguousarray(R)).to(device),
            torch.from_numpy(np.ascontiguousarray(order, dtype=np.int32)).to(device),
            torch.from_numpy(np.ascontiguousarray(psi, dtype=np.int32)).to(device))


def oracle_decode(R, order, psi, G64, transmit):
    r = O.run_pattern(R, order, psi, G64.shape[0], G64, want_transmit=transmit)
    return r
