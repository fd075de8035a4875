"""The C-ABI library without a GPU: it builds for sm_103a, loads, exports every function
include/hydra.h declares, and rejects bad arguments on the host before any CUDA call."""
import ctypes

import pytest

from paper_2309_00754_gb300 import build as B
from paper_2309_00754_gb300 import hydra as H


@pytest.fixture(scope="module")
def lib():
    B.build()
    return H.load()


def test_exports_every_declared_function(lib):
    names = H.header_functions()
    assert "hydra_lora_linear" in names and "hydra_token_logprobs_kl" in names and "ppo_gae" in names
    for n in names:
        assert hasattr(lib, n), f"libhydra.so does not export {n}"
    assert set(names) <= set(H._SIGNATURES), "binding lacks a signature for a declared function"


def test_status_strings_and_version(lib):
    assert H.status_string(0) == "HYDRA_OK"
    for code in range(1, 9):
        assert H.status_string(code).startswith("HYDRA_ERR_")
    assert lib.hydra_abi_version() == 1


def test_workspace_size(lib):
    assert H.lora_linear_workspace_size(0, 16) == 0
    assert H.lora_linear_workspace_size(100, 0) == 0
    assert H.lora_linear_workspace_size(2048, 16) == 2048 * 16 * 2
    assert H.lora_linear_workspace_size(3, 8) == 256


FAKE = 1 << 20  # a 16-byte aligned non-null value; never dereferenced on these paths


def _lin(lib, **kw):
    a = dict(x_off=FAKE, x_on=None, M=64, K=64, N=64, W=FAKE, A=None, B=None, r=0, s=2.0,
             y_off=FAKE, y_on=None, dt=0, ws=None, wsb=0, algo=0)
    a.update(kw)
    return lib.hydra_lora_linear_algo(a["x_off"], a["x_on"], a["M"], a["K"], a["N"], a["W"], a["A"],
                                      a["B"], a["r"], a["s"], a["y_off"], a["y_on"], a["dt"],
                                      a["ws"], a["wsb"], a["algo"], None)


def test_lora_linear_argument_errors(lib):
    assert _lin(lib, x_off=None) == 1
    assert _lin(lib, W=None) == 1
    assert _lin(lib, y_off=None, y_on=None) == 1
    assert _lin(lib, K=60) == 3          # K % 8
    assert _lin(lib, N=12) == 3          # N % 8
    assert _lin(lib, K=0) == 2
    assert _lin(lib, M=-1) == 2
    assert _lin(lib, M=1 << 31) == 2
    assert _lin(lib, r=300, A=FAKE, B=FAKE, y_on=FAKE) == 2
    assert _lin(lib, r=12, A=FAKE, B=FAKE, y_on=FAKE) == 3
    assert _lin(lib, r=16, y_on=FAKE) == 1                      # LoRA without A/B
    assert _lin(lib, r=16, A=FAKE, B=FAKE, y_on=FAKE) == 7      # no workspace
    assert _lin(lib, r=16, A=FAKE, B=FAKE, y_on=FAKE, ws=FAKE, wsb=100) == 7
    assert _lin(lib, x_off=FAKE + 8) == 3                       # misaligned pointer
    assert _lin(lib, dt=7) == 4
    assert _lin(lib, algo=4) == 4
    assert _lin(lib, algo=2, M=9, x_on=FAKE * 2) == 2           # GEMV takes <= 16 rows
    assert _lin(lib, M=0) == 0                                  # empty: no launch


def _skinny(lib, **kw):
    a = dict(x=FAKE, M=128, K=4096, N=4096, W=FAKE, u=None, u_row0=0, u_rows=0, B=None, r=0,
             y=FAKE, dt=0, tile_n=0, split_k=0)
    a.update(kw)
    return lib.hydra_skinny_linear(a["x"], a["M"], a["K"], a["N"], a["W"], a["u"], a["u_row0"],
                                   a["u_rows"], a["B"], a["r"], a["y"], a["dt"], a["tile_n"],
                                   a["split_k"], None)


def test_skinny_linear_argument_errors(lib):
    lora = dict(u=FAKE, B=FAKE, r=16, u_row0=64, u_rows=64)
    assert _skinny(lib, x=None) == 1
    assert _skinny(lib, W=None) == 1
    assert _skinny(lib, y=None) == 1
    assert _skinny(lib, r=16, u_row0=64, u_rows=64) == 1        # LoRA without u and B
    assert _skinny(lib, M=129) == 2                             # one tile of at most 128 rows
    assert _skinny(lib, M=-1) == 2
    assert _skinny(lib, N=4104) == 2                            # N % 16
    assert _skinny(lib, K=4100) == 3                            # K % 8
    assert _skinny(lib, **dict(lora, r=12)) == 3
    assert _skinny(lib, **dict(lora, r=264)) == 2
    assert _skinny(lib, **dict(lora, u_row0=100, u_rows=64)) == 2  # LoRA rows past M
    assert _skinny(lib, **dict(lora, u_rows=0)) == 2
    assert _skinny(lib, **dict(lora, u_row0=-1)) == 2
    assert _skinny(lib, x=FAKE + 8) == 3
    assert _skinny(lib, dt=7) == 4
    assert _skinny(lib, tile_n=24) == 4                         # multiple of 16
    assert _skinny(lib, tile_n=272) == 4
    assert _skinny(lib, split_k=9) == 4
    assert _skinny(lib, K=128, split_k=3) == 4                  # more CTAs than k-blocks
    assert _skinny(lib, M=0) == 0                               # empty: no launch


def test_rope_linear_argument_errors(lib):
    f = lib.hydra_dual_linear_rope

    def call(**kw):
        a = dict(M=64, K=64, N=768, P=100, cols=512, hd=128, table=FAKE)
        a.update(kw)
        return f(FAKE, None, a["M"], a["K"], a["N"], FAKE, None, None, 0, FAKE, None, a["P"],
                 a["cols"], a["hd"], a["table"], None)
    assert call(hd=64) == 4          # heads of 128 only
    assert call(table=None) == 1
    assert call(table=FAKE + 8) == 3
    assert call(cols=500) == 2       # whole heads
    assert call(cols=896) == 2       # beyond N
    assert call(P=0) == 2
    assert call(M=0) == 0            # empty: no launch
    t = lib.hydra_rope_table
    assert t(100, 128, 1e4, None, None) == 1
    assert t(100, 127, 1e4, FAKE, None) == 2
    assert t(100, 128, 0.0, FAKE, None) == 4
    assert t(100, 128, 1e4, FAKE + 4, None) == 3
    assert t(0, 128, 1e4, FAKE, None) == 0


def test_logprobs_and_gae_argument_errors(lib):
    f = lib.hydra_token_logprobs_kl
    assert f(FAKE, FAKE, 5, 1, 1, 10, 10, FAKE, None, None, 0.1, FAKE, FAKE, FAKE, None, None, None) == 4
    assert f(FAKE, FAKE, 1, 1, 1, 10, 9, FAKE, None, None, 0.1, FAKE, FAKE, FAKE, None, None, None) == 2
    assert f(FAKE, FAKE, 1, 1, 1, 0, 0, FAKE, None, None, 0.1, FAKE, FAKE, FAKE, None, None, None) == 2
    assert f(None, FAKE, 1, 1, 1, 10, 10, FAKE, None, None, 0.1, FAKE, FAKE, FAKE, None, None, None) == 1
    assert f(FAKE, FAKE, 1, 0, 4, 10, 10, FAKE, None, None, 0.1, FAKE, FAKE, FAKE, None, None, None) == 0
    g = lib.ppo_gae
    assert g(FAKE, FAKE, None, 2, 20000, 1.0, 0.95, FAKE, FAKE, None) == 2
    assert g(FAKE, FAKE, None, -1, 4, 1.0, 0.95, FAKE, FAKE, None) == 2
    assert g(None, FAKE, None, 2, 4, 1.0, 0.95, FAKE, FAKE, None) == 1
    assert g(FAKE, FAKE, None, 0, 4, 1.0, 0.95, FAKE, FAKE, None) == 0
    assert lib.hydra_lora_down(None, 4, 8, FAKE, 8, 1.0, FAKE, None) == 1
    assert lib.hydra_lora_down(FAKE, 4, 8, FAKE, 4, 1.0, FAKE, None) == 3
    code = ctypes.c_int32(0)
    assert lib.hydra_device_error(None, 0) == 1


def test_ppo_loss_argument_errors(lib):
    ws = H.ppo_workspace_size()
    assert ws >= 16 * 512 + 32 * 1024
    f = lib.hydra_ppo_loss
    args = lambda S=4, L=8, eps=0.2, wh=0, stats=FAKE, a=FAKE, wsb=ws, wsp=FAKE: f(
        a, FAKE, FAKE, FAKE, FAKE, None, S, L, eps, wh, None, FAKE, FAKE, stats, wsp, wsb, None)
    assert args(S=-1) == 2
    assert args(S=1 << 16, L=1 << 15) == 2  # S * L >= 2^31
    assert args(eps=-0.1) == 4 and args(eps=1.0) == 4 and args(eps=float("nan")) == 4
    assert args(wh=2) == 4
    assert args(stats=None) == 1
    assert args(a=None) == 1
    assert args(wsb=ws - 8) == 7 and args(wsp=None) == 7 and args(wsp=FAKE + 8) == 7
    m = lib.hydra_ppo_adv_moments
    assert m(FAKE, None, -1, 4, FAKE, FAKE, ws, None) == 2
    assert m(FAKE, None, 2, 4, None, FAKE, ws, None) == 1
    assert m(FAKE, None, 2, 4, FAKE, FAKE, 16, None) == 7


def test_ppo_merge_moments_matches_whole_batch(lib):
    """The host merge of per-shard (n, mean, M2) triples equals the moments of the whole
    batch (numpy mean and population variance), whatever the split, including empty shards."""
    import numpy as np
    import torch
    rng = np.random.default_rng(7)
    x = rng.normal(3.0, 2.0, 1000)
    for cuts in ([0, 1000], [0, 1, 999, 1000], [0, 300, 300, 700, 1000], [0, 0, 1000]):
        tri = []
        for a, b in zip(cuts[:-1], cuts[1:]):
            s = x[a:b]
            m = s.mean() if len(s) else 0.0
            tri.append([len(s), m, ((s - m) ** 2).sum()])
        out = H.ppo_merge_moments(torch.tensor(tri, dtype=torch.float64)).numpy()
        assert out[0] == 1000
        assert abs(out[1] - x.mean()) < 1e-13
        assert abs(out[2] / 1000 - x.var()) < 1e-12
    assert H.ppo_merge_moments(torch.zeros(0, 3, dtype=torch.float64)).tolist() == [0.0, 0.0, 0.0]
    with pytest.raises(H.HydraError):
        H.ppo_merge_moments(torch.tensor([[-1.0, 0.0, 0.0]], dtype=torch.float64))


def test_binding_refuses_other_output_dtypes():
    import torch
    assert H._out_dtype(torch.empty(1, dtype=torch.float32)) == H.HYDRA_F32
    assert H._out_dtype(torch.empty(1, dtype=torch.bfloat16)) == H.HYDRA_BF16
    with pytest.raises(ValueError):
        H._out_dtype(torch.empty(1, dtype=torch.float16))
