"""In-kernel failure detection without a GPU fault: a kernel waits on an mbarrier that nothing
signals, through the bounded wait every kernel of the library uses. The wait expires, the
kernel records its code in the device error word and returns; nothing traps, and the
context stays usable for the next call."""
import time

import numpy as np
import pytest
import torch

import oracle as O
from paper_2309_00754_gb300 import build as B
from paper_2309_00754_gb300 import hydra as H
from paper_2309_00754_gb300 import synth
from tests.helpers import TOL_GAE, assert_rel, dev_f32, dev_i32, host_f64

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def lib():
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    B.build()
    L = H.load()
    H.device_error(clear=True)
    yield L
    assert H.device_error(clear=True) == 0


def test_bounded_wait_expires_reports_and_leaves_the_context_usable():
    H.device_error(clear=True)
    t0 = time.perf_counter()
    H.selftest_wait_timeout()
    code = H.device_error(clear=True)  # synchronises: the kernel has returned
    dt = time.perf_counter() - t0
    assert code == 0x105
    assert 0.1 < dt < 30.0, f"the wait took {dt:.2f} s"
    assert H.status_string(6).startswith("HYDRA_ERR_TIMEOUT")
    # the next call on the same context runs normally and matches the oracle
    S, L = 4, 64
    rw = synth.normal_f32(5101, (S, L))
    vals = synth.normal_f32(5102, (S, L))
    lengths = np.array([64, 1, 37, 0], dtype=np.int32)
    adv = torch.empty(S, L, device="cuda")
    ret = torch.empty(S, L, device="cuda")
    H.ppo_gae(dev_f32(rw), dev_f32(vals), dev_i32(lengths), 1.0, 0.95, adv, ret)
    ref_a, ref_r = O.gae(rw.astype(np.float64), vals.astype(np.float64), lengths, 1.0, 0.95)
    assert_rel(host_f64(adv), ref_a, TOL_GAE, "advantages")
    assert_rel(host_f64(ret), ref_r, TOL_GAE, "returns")
    assert H.device_error(clear=True) == 0
