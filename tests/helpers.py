"""Test-side conversions between the generator's numpy arrays, torch device tensors and
the oracle's float64 arrays, plus the tolerance checks used by the parity tests."""
import numpy as np
import torch

import oracle as O
from paper_2309_00754_gb300 import synth

# tolerances of the scoring path (bf16-in / fp32-accumulate linear outputs; log-probs and
# KL rewards; fp32 GAE)
TOL_LINEAR = 2e-2
TOL_LOGP = 5e-3
TOL_GAE = 1e-4


def dev_bf16(bits, device="cuda"):
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).to(device)


def dev_f32(a, device="cuda"):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(device)


def dev_i32(a, device="cuda"):
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.int32)).to(device)


def host_f64(t):
    """float64 numpy copy of a device tensor (bf16 widened exactly)."""
    t = t.detach().cpu()
    if t.dtype == torch.bfloat16:
        return O.bf16_to_f64(t.contiguous().view(torch.int16).numpy().view(np.uint16))
    return t.double().numpy()


def f64(bits):
    return O.bf16_to_f64(bits)


def max_rel_err(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.max(np.abs(got - ref) / np.maximum(1.0, np.abs(ref)))) if ref.size else 0.0


def max_abs_err(got, ref):
    got = np.asarray(got, dtype=np.float64)
    ref = np.asarray(ref, dtype=np.float64)
    return float(np.max(np.abs(got - ref))) if ref.size else 0.0


def assert_rel(got, ref, tol, what=""):
    e = max_rel_err(got, ref)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert e <= tol, f"{what}: max |err|/max(1,|ref|) = {e:.3e} > {tol:.1e}"
    return e


def assert_abs(got, ref, tol, what=""):
    e = max_abs_err(got, ref)
    assert np.all(np.isfinite(got)), f"{what}: non-finite output"
    assert e <= tol, f"{what}: max |err| = {e:.3e} > {tol:.1e}"
    return e


__all__ = ["synth", "O"]
