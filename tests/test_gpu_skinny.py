"""GPU parity of the split-K decode linear (hydra_skinny_linear): both streams' rows in one
matrix, y = x W^T with the LoRA term u B^T on the LoRA-on rows (§3 Dynamic LoRA: one frozen
W serves the LoRA-off and LoRA-on streams), against the oracle's dual-output LoRA linear on
the same seeded inputs. Every element is compared; the cases span several tiles, a ragged N
tail, a ragged last k-block, one to eight CTAs splitting K (with ranks that own no columns),
two LoRA k-blocks and partial LoRA row ranges."""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2309_00754_gb300 import build as B
from paper_2309_00754_gb300 import hydra as H
from paper_2309_00754_gb300 import synth
from tests.helpers import TOL_LINEAR, assert_rel, dev_bf16, f64, host_f64

pytestmark = pytest.mark.gpu

S_LORA = 2.0


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    L = H.load()
    H.device_error(clear=True)
    yield L
    assert H.device_error(clear=True) == 0


def _problem(M, K, N, r, seed):
    x = synth.normal_bf16(synth.tensor_seed(seed, 1), (M, K), 1.0)
    W = synth.normal_bf16(synth.tensor_seed(seed, 3), (N, K), 0.02)
    A = synth.normal_bf16(synth.tensor_seed(seed, 4), (max(r, 1), K), 0.02)[:r]
    Bm = synth.normal_bf16(synth.tensor_seed(seed, 5), (N, max(r, 1)), 0.02)[:, :r]
    return x, W, A, Bm


def _reference(x, W, A, Bm, u_row0, u_rows, out_bf16=True):
    """Oracle dual-output linear: rows outside [u_row0, u_row0 + u_rows) are the LoRA-off
    stream, the rows inside the LoRA-on stream (u = s x_on A^T stored as bf16)."""
    xf, Wf = f64(x), f64(W)
    y = xf @ Wf.T
    u = None
    if A.shape[0] > 0:
        x_on = xf[u_row0:u_row0 + u_rows]
        _, y_on = O.dual_lora_linear(x_on, x_on, Wf, f64(A), f64(Bm), S_LORA, out_bf16=False)
        y[u_row0:u_row0 + u_rows] = y_on
        u = O.lora_down(x_on, f64(A), S_LORA)
    return (O.round_bf16(y) if out_bf16 else y), u


def _run(x, W, u, Bm, u_row0, out=torch.bfloat16, tile_n=0, split_k=0):
    M = x.shape[0]
    N = W.shape[0]
    y = torch.full((M, N), float("nan"), dtype=out, device="cuda")
    H.hydra_skinny_linear(x, W, y, u=u, B=Bm, u_row0=u_row0, tile_n=tile_n, split_k=split_k)
    torch.cuda.synchronize()
    return y


@pytest.mark.parametrize("S,K,N,r,tile_n,split_k", [
    (64, 4096, 4096, 16, 0, 0),     # decode o / down shape, library's choice
    (64, 512, 1024, 32, 256, 8),    # one k-block per CTA of the cluster
    (12, 1032, 528, 16, 0, 0),      # ragged last k-block, N tail of 16 columns
    (9, 328, 272, 8, 96, 3),        # everything ragged
    (64, 256, 512, 0, 0, 0),        # no LoRA
    (33, 640, 800, 64, 160, 5),     # five CTAs, LoRA k-block on the last
    (50, 2048, 1024, 72, 128, 6),   # two LoRA k-blocks; ranks 4 and 5 own no columns
    (40, 1024, 1040, 16, 256, 1),   # single CTA per tile
    (64, 4096, 12288, 32, 0, 0),    # decode qkv shape
    (64, 4096, 22016, 32, 0, 0),    # decode gate/up shape
    (64, 11008, 4096, 16, 0, 0),    # decode down shape
    (12, 11008, 4096, 16, 0, 0),    # down shape at 12 sequences
])
def test_skinny_linear_parity(S, K, N, r, tile_n, split_k):
    x, W, A, Bm = _problem(2 * S, K, N, r, seed=S + K + N + r)
    ref, u = _reference(x, W, A, Bm, S, S)
    ud = dev_bf16(O.f64_to_bf16_bits(u)) if r else None
    y = _run(dev_bf16(x), dev_bf16(W), ud, dev_bf16(Bm) if r else None, S, tile_n=tile_n,
             split_k=split_k)
    assert_rel(host_f64(y[:S]), ref[:S], TOL_LINEAR, "off rows")
    assert_rel(host_f64(y[S:]), ref[S:], TOL_LINEAR, "on rows")


@pytest.mark.parametrize("M,u_row0,u_rows", [(1, 0, 1), (128, 64, 64), (50, 10, 20), (17, 0, 17)])
def test_skinny_linear_lora_row_ranges(M, u_row0, u_rows):
    K, N, r = 768, 528, 16
    x, W, A, Bm = _problem(M, K, N, r, seed=100 + M)
    ref, u = _reference(x, W, A, Bm, u_row0, u_rows)
    y = _run(dev_bf16(x), dev_bf16(W), dev_bf16(O.f64_to_bf16_bits(u)), dev_bf16(Bm), u_row0,
             split_k=4)
    assert_rel(host_f64(y), ref, TOL_LINEAR, "y")


@pytest.mark.parametrize("split_k", [1, 3, 8])
def test_skinny_linear_fp32_out(split_k):
    S, K, N, r = 40, 1024, 1040, 16
    x, W, A, Bm = _problem(2 * S, K, N, r, seed=7)
    ref, u = _reference(x, W, A, Bm, S, S, out_bf16=False)
    y = _run(dev_bf16(x), dev_bf16(W), dev_bf16(O.f64_to_bf16_bits(u)), dev_bf16(Bm), S,
             out=torch.float32, split_k=split_k)
    assert_rel(host_f64(y), ref, 1e-4, "y fp32")


def test_skinny_linear_lm_head_shape_fp32():
    # the decode LM head: 4096 -> 32000 with fp32 logits for both streams' 128 rows
    S, K, N = 64, 4096, 32000
    x, W, A, Bm = _problem(2 * S, K, N, 0, seed=17)
    ref, _ = _reference(x, W, A, Bm, S, S, out_bf16=False)
    y = _run(dev_bf16(x), dev_bf16(W), None, None, 0, out=torch.float32)
    assert_rel(host_f64(y), ref, 1e-4, "logits")


def test_skinny_linear_deterministic_and_lora_off_bitwise():
    # a fixed (tile, split) gives the same bits on every call; with B = 0 the LoRA-on rows equal
    # the LoRA-off rows of the same input bit for bit (§3 Dynamic LoRA), as they do with no LoRA
    S, K, N, r = 32, 2048, 1024, 16
    x, W, A, _ = _problem(S, K, N, r, seed=9)
    xx = dev_bf16(np.concatenate([x, x]))
    Wd = dev_bf16(W)
    u = dev_bf16(O.f64_to_bf16_bits(O.lora_down(f64(x), f64(A), S_LORA)))
    Bz = torch.zeros(N, r, dtype=torch.bfloat16, device="cuda")
    y1 = _run(xx, Wd, u, Bz, S, tile_n=128, split_k=6)
    y2 = _run(xx, Wd, u, Bz, S, tile_n=128, split_k=6)
    y0 = _run(xx, Wd, None, None, 0, tile_n=128, split_k=6)
    assert torch.equal(y1, y2)
    assert torch.equal(y1[:S], y1[S:])
    assert torch.equal(y1, y0)
    Bm = dev_bf16(synth.normal_bf16(11, (N, r), 0.02))
    y3 = _run(xx, Wd, u, Bm, S, tile_n=128, split_k=6)
    assert torch.equal(y3[:S], y1[:S]) and not torch.equal(y3[S:], y1[S:])


def test_skinny_linear_split_choices_agree():
    # different cluster sizes associate the fp32 sums differently; all stay within the
    # linear tolerance of the oracle and of one another
    S, K, N, r = 64, 4096, 2048, 32
    x, W, A, Bm = _problem(2 * S, K, N, r, seed=13)
    ref, u = _reference(x, W, A, Bm, S, S)
    ud = dev_bf16(O.f64_to_bf16_bits(u))
    ys = [_run(dev_bf16(x), dev_bf16(W), ud, dev_bf16(Bm), S, tile_n=tn, split_k=ks)
          for tn, ks in ((256, 1), (256, 2), (256, 8), (192, 3), (64, 4))]
    for y in ys:
        assert_rel(host_f64(y), ref, TOL_LINEAR, "y")
        assert_rel(host_f64(y), host_f64(ys[0]), TOL_LINEAR, "y vs single CTA")
