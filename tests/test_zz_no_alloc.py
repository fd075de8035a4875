"""hydra_lora_linear_noalloc: the workspace-free variant of hydra_lora_linear, for callers
that cannot allocate device memory (a plugin whose host framework owns the device memory
pool, or a latency-critical caller that cannot afford cudaMalloc/cudaFree). It keeps the
LoRA down-projection u in the library's static device array instead of a workspace.

The test calls it through the C-ABI twice in a row (the two calls share that array) and
checks both results against the workspace entry point. Both entry points run the same
kernels on the same u, so the outputs must agree bit for bit. The file name makes pytest
collect it last, so a run that stops at the first failure has already run every other
test."""
import numpy as np
import pytest
import torch

from paper_2309_00754_gb300 import build as Bld
from paper_2309_00754_gb300 import hydra as H
from paper_2309_00754_gb300 import synth
from tests.helpers import dev_bf16, host_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    Bld.build()
    H.load()
    H.device_error(clear=True)
    yield
    assert H.device_error(clear=True) == 0


def _problem(M, K, N, r, seed, shared):
    x = dev_bf16(synth.normal_bf16(seed + 1, (M, K)))
    x_on = None if shared else dev_bf16(synth.normal_bf16(seed + 2, (M, K)))
    W = dev_bf16(synth.normal_bf16(seed + 3, (N, K), 0.02))
    A = dev_bf16(synth.normal_bf16(seed + 4, (r, K), 0.02))
    B = dev_bf16(synth.normal_bf16(seed + 5, (N, r), 0.02))
    return x, x_on, W, A, B


def _outputs(M, N):
    return (torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda"),
            torch.full((M, N), float("nan"), dtype=torch.bfloat16, device="cuda"))


def test_noalloc_matches_workspace_entry_point_on_two_calls():
    # call 1: shared input through the tensor-core kernel; call 2: stacked streams through
    # the GEMV kernel, with a different M * r, so it overwrites the array call 1 used
    cases = [(300, 512, 520, 16, 7100, True), (8, 1024, 264, 64, 7200, False)]
    problems = [_problem(M, K, N, r, seed, shared) for M, K, N, r, seed, shared in cases]
    got = []
    for (M, K, N, r, _, _), (x, x_on, W, A, B) in zip(cases, problems):
        y_off, y_on = _outputs(M, N)
        H.hydra_lora_linear_noalloc(x, x_on, W, A, B, 2.0, y_off, y_on)
        got.append((y_off, y_on))
    torch.cuda.synchronize()
    for (M, K, N, r, _, _), (x, x_on, W, A, B), (y_off, y_on) in zip(cases, problems, got):
        ref_off, ref_on = _outputs(M, N)
        ws = torch.empty(H.lora_linear_workspace_size(M, r), dtype=torch.uint8, device="cuda")
        H.hydra_lora_linear(x, x_on, W, A, B, 2.0, ref_off, ref_on, ws)
        assert torch.equal(y_off, ref_off), "y_off differs from the workspace entry point"
        assert torch.equal(y_on, ref_on), "y_on differs from the workspace entry point"
        assert np.all(np.isfinite(host_f64(y_on)))


def test_noalloc_without_lora_matches_and_allocates_nothing():
    # r = 0: no u at all, the plain dual linear; then a warm call with LoRA must leave the
    # device's free memory where it was (the array was reserved when the library loaded)
    M, K, N = 96, 512, 264
    x, x_on, W, A, B = _problem(M, K, N, 16, 7300, False)
    y_off, y_on = _outputs(M, N)
    H.hydra_lora_linear_noalloc(x, x_on, W, None, None, 2.0, y_off, y_on)
    ref_off, ref_on = _outputs(M, N)
    H.hydra_lora_linear(x, x_on, W, None, None, 2.0, ref_off, ref_on, None)
    torch.cuda.synchronize()
    assert torch.equal(y_off, ref_off) and torch.equal(y_on, ref_on)

    H.hydra_lora_linear_noalloc(x, x_on, W, A, B, 2.0, y_off, y_on)  # warm: set-up done
    torch.cuda.synchronize()
    free_before, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        H.hydra_lora_linear_noalloc(x, x_on, W, A, B, 2.0, y_off, y_on)
    torch.cuda.synchronize()
    free_after, _ = torch.cuda.mem_get_info()
    assert free_after == free_before, f"free device memory moved by {free_before - free_after} B"


def test_noalloc_rejects_u_beyond_the_static_array():
    r = 16
    M = (1 << 21) // r + 1
    x = torch.zeros(M, 8, dtype=torch.bfloat16, device="cuda")
    W = torch.zeros(8, 8, dtype=torch.bfloat16, device="cuda")
    A = torch.zeros(r, 8, dtype=torch.bfloat16, device="cuda")
    B = torch.zeros(8, r, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(M, 8, dtype=torch.bfloat16, device="cuda")
    with pytest.raises(H.HydraError) as e:
        H.hydra_lora_linear_noalloc(x, None, W, A, B, 2.0, y, y.clone())
    assert e.value.status == 2  # HYDRA_ERR_SHAPE
