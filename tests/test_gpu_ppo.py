"""Parity of the PPO update-side kernels (clipped surrogate, value loss, their gradients,
advantage whitening and moments) with the fp64 oracle, through the C-ABI.

Inputs follow the scored batch the losses consume: logp_old are sampled-token log-probs
(-|N(0, 2)| - 0.05), logp_new = logp_old + N(0, 0.15) (about a fifth of the ratios leave
[0.8, 1.2]), advantages N(0.3, 1.5), returns N(0, 1), values = returns + N(0, 0.5), ragged
lengths.

Tolerances, from the fp32 arithmetic: per-token ratios and gradients carry a few fp32
roundings (expf within 2 ulp): 1e-5 relative. The sums are fp32 within a thread (at most a
few hundred terms) and fp64 beyond: 5e-5 of the sum of the terms' magnitudes. The clip
decisions are taken in fp32 by the kernel and in fp64 by the oracle; tokens whose ratio lies
within 1e-5 of a clip boundary may go either way, and both outcomes are accepted there.
"""
import numpy as np
import pytest
import torch

import oracle as O
from paper_2309_00754_gb300 import hydra as H
from paper_2309_00754_gb300 import synth
from tests.helpers import dev_f32, dev_i32

pytestmark = pytest.mark.gpu

STAT_KEYS = H.PPO_STATS


def make_inputs(seed, S, L, ragged=True):
    ts = lambda i: synth.tensor_seed(seed, i)
    lo = (-np.abs(synth.normal_f32(ts(0), (S, L), 2.0)) - 0.05).astype(np.float32)
    ln = (lo + synth.normal_f32(ts(1), (S, L), 0.15)).astype(np.float32)
    adv = (synth.normal_f32(ts(2), (S, L), 1.5) + 0.3).astype(np.float32)
    ret = synth.normal_f32(ts(3), (S, L), 1.0)
    val = (ret + synth.normal_f32(ts(4), (S, L), 0.5)).astype(np.float32)
    if ragged and S > 0 and L > 0:
        lengths = synth.randint(ts(5), (S,), 0, L + 1)
        lengths[0] = L
    else:
        lengths = np.full(S, L, dtype=np.int32)
    return ln, lo, adv, ret, val, lengths


def run_kernel(ln, lo, adv, ret, val, lengths, eps, whiten, moments=None, misalign=False):
    S, L = ln.shape

    def put(a):
        if not misalign:
            return dev_f32(a)
        buf = torch.zeros(a.size + 1, dtype=torch.float32, device="cuda")
        buf[1:] = dev_f32(a.reshape(-1))
        return buf[1:].view(S, L)

    d = [put(a) for a in (ln, lo, adv, ret, val)]
    gl = put(np.zeros((S, L), np.float32))
    gv = put(np.zeros((S, L), np.float32))
    stats = torch.full((7,), float("nan"), dtype=torch.float64, device="cuda")
    ws = torch.empty(H.ppo_workspace_size(), dtype=torch.uint8, device="cuda")
    H.hydra_ppo_loss(*d, dev_i32(lengths), eps, whiten, gl, gv, stats, ws, adv_moments=moments)
    torch.cuda.synchronize()
    assert H.device_error(clear=True) == 0
    return gl.cpu().double().numpy(), gv.cpu().double().numpy(), stats.cpu().numpy()


def check(got, ln, lo, adv, ret, val, lengths, eps, whiten, moments=None):
    gl, gv, st = got
    ref = O.ppo_loss(ln, lo, adv, ret, val, lengths, clip_eps=eps, whiten=whiten, moments=moments)
    S, L = ln.shape
    valid = np.arange(L)[None, :] < lengths.reshape(S, 1)
    n = ref["n"]
    assert st[6] == n
    if n == 0:
        assert np.all(st == 0.0)
        assert not gl.any() and not gv.any()
        return ref
    inv_n = 1.0 / n
    r = np.exp(ln.astype(np.float64) - lo)
    A = adv.astype(np.float64)
    if whiten:
        A = (A - ref["adv_mean"]) / np.sqrt(ref["adv_std"] ** 2 + 1e-8)
    amb = valid & ((np.abs(r - (1 + eps)) <= 1e-5) | (np.abs(r - (1 - eps)) <= 1e-5))
    # gradients
    g_ref = ref["grad_logp"]
    scale = np.abs(g_ref).max() if g_ref.size else 0.0
    ok = np.abs(gl - g_ref) <= 1e-5 * np.abs(g_ref) + 1e-6 * scale
    alt = np.abs(gl - np.where(g_ref == 0.0, -r * A * inv_n, 0.0)) <= 1e-5 * np.abs(r * A * inv_n) + 1e-6 * scale
    assert np.all(ok | (amb & alt)), f"grad_logp: {np.argwhere(~(ok | (amb & alt)))[:5]}"
    gv_ref = ref["grad_values"]
    assert np.all(np.abs(gv - gv_ref) <= 1e-5 * np.abs(gv_ref) + 1e-7 * np.abs(gv_ref).max())
    assert not gl[~valid].any() and not gv[~valid].any()
    # statistics
    sab = lambda x: float(np.abs(x[valid]).sum()) * inv_n
    assert abs(st[0] - ref["loss_clip"]) <= 5e-5 * sab(r * A) + 1e-12, (st[0], ref["loss_clip"])
    assert abs(st[1] - ref["loss_value"]) <= 5e-5 * ref["loss_value"] + 1e-12
    assert abs(st[2] - ref["clip_frac"]) <= amb.sum() * inv_n + 1e-12
    assert abs(st[3] - ref["approx_kl"]) <= 5e-5 * sab(ln.astype(np.float64) - lo) + 1e-12
    assert abs(st[4] - ref["adv_mean"]) <= 5e-5 * sab(adv.astype(np.float64)) + 1e-12
    rms = np.sqrt(float((adv.astype(np.float64)[valid] ** 2).sum()) * inv_n)
    assert abs(st[5] - ref["adv_std"]) <= 1e-4 * rms + 1e-12
    return ref


CASES = [  # S, L, ragged
    (3, 11, True),      # scalar path (L % 4 != 0)
    (5, 128, False),
    (37, 516, True),    # float4 path, ragged rows
    (64, 512, True),
    (9, 1, False),
    (2, 4097, True),    # scalar path, rows longer than a warp pass
    (300, 64, True),    # more rows than one block's warps
]


@pytest.mark.parametrize("S,L,ragged", CASES)
@pytest.mark.parametrize("whiten", [False, True])
def test_ppo_loss_parity(S, L, ragged, whiten):
    x = make_inputs(40 + S, S, L, ragged)
    check(run_kernel(*x, 0.2, whiten), *x, 0.2, whiten)


@pytest.mark.parametrize("eps", [0.0, 0.1, 0.3])
def test_ppo_loss_clip_ranges(eps):
    x = make_inputs(50, 48, 256)
    check(run_kernel(*x, eps, True), *x, eps, True)


def test_ppo_loss_misaligned_pointers_take_scalar_path():
    x = make_inputs(51, 16, 128)
    check(run_kernel(*x, 0.2, True, misalign=True), *x, 0.2, True)


@pytest.mark.parametrize("S,L", [(0, 16), (4, 0), (0, 0)])
def test_ppo_loss_empty(S, L):
    x = make_inputs(52, S, L, ragged=False)
    check(run_kernel(*x, 0.2, True), *x, 0.2, True)


def test_ppo_loss_all_rows_empty():
    ln, lo, adv, ret, val, _ = make_inputs(53, 6, 32)
    lengths = np.zeros(6, dtype=np.int32)
    check(run_kernel(ln, lo, adv, ret, val, lengths, 0.2, True), ln, lo, adv, ret, val, lengths,
          0.2, True)


def test_ppo_loss_is_deterministic():
    x = make_inputs(54, 200, 512)
    a = run_kernel(*x, 0.2, True)
    b = run_kernel(*x, 0.2, True)
    for u, v in zip(a, b):
        assert np.array_equal(u, v)


def test_ppo_adv_moments():
    ln, lo, adv, ret, val, lengths = make_inputs(55, 77, 260)
    ws = torch.empty(H.ppo_workspace_size(), dtype=torch.uint8, device="cuda")
    m = torch.zeros(3, dtype=torch.float64, device="cuda")
    H.hydra_ppo_adv_moments(dev_f32(adv), dev_i32(lengths), m, ws)
    n, mean, m2 = m.cpu().tolist()
    ref = O.ppo_loss(ln, lo, adv, ret, val, lengths)
    assert n == ref["n"]
    assert abs(mean - ref["adv_mean"]) <= 1e-5 * (abs(ref["adv_mean"]) + ref["adv_std"])
    assert abs(np.sqrt(m2 / n) - ref["adv_std"]) <= 1e-5 * ref["adv_std"]


def test_ppo_loss_shards_with_merged_moments():
    """Two shards of one batch, each whitened and normalised with the merged moments (as
    data-parallel replicas would): their losses add up to the whole batch's, and every
    shard matches the oracle run with the same moments."""
    ln, lo, adv, ret, val, lengths = make_inputs(56, 90, 384)
    ws = torch.empty(H.ppo_workspace_size(), dtype=torch.uint8, device="cuda")
    cut = 33
    parts = []
    for rows in (slice(0, cut), slice(cut, 90)):
        m = torch.zeros(3, dtype=torch.float64, device="cuda")
        H.hydra_ppo_adv_moments(dev_f32(adv[rows]), dev_i32(lengths[rows]), m, ws)
        parts.append(m.cpu())
    merged = H.ppo_merge_moments(torch.stack(parts))
    md = merged.cuda()
    whole = run_kernel(ln, lo, adv, ret, val, lengths, 0.2, True)
    sums = np.zeros(4)
    for rows in (slice(0, cut), slice(cut, 90)):
        sh = [a[rows] for a in (ln, lo, adv, ret, val, lengths)]
        got = run_kernel(*sh, 0.2, True, moments=md)
        check(got, *sh, 0.2, True, moments=merged.numpy())
        sums += got[2][:4]
    np.testing.assert_allclose(sums, whole[2][:4], rtol=1e-5, atol=1e-7)


def test_ppo_loss_bad_length_sets_device_error():
    ln, lo, adv, ret, val, lengths = make_inputs(57, 4, 64)
    lengths[2] = 65
    d = [dev_f32(a) for a in (ln, lo, adv, ret, val)]
    gl, gv = torch.empty_like(d[0]), torch.empty_like(d[0])
    stats = torch.zeros(7, dtype=torch.float64, device="cuda")
    ws = torch.empty(H.ppo_workspace_size(), dtype=torch.uint8, device="cuda")
    H.device_error(clear=True)
    H.hydra_ppo_loss(*d, dev_i32(lengths), 0.2, False, gl, gv, stats, ws)
    torch.cuda.synchronize()
    assert H.device_error(clear=True) == 0x202
    # the bad row is clamped to L tokens
    lengths[2] = 64
    check((gl.cpu().double().numpy(), gv.cpu().double().numpy(), stats.cpu().numpy()),
          ln, lo, adv, ret, val, lengths, 0.2, False)


def test_ppo_loss_full_size_65536x512():
    """The kernel-sweep launch: 65536 sequences x 512 tokens, lengths U[64, 512], whitened.
    Statistics against the oracle over the whole batch; gradients on 64 sampled rows."""
    S, L = 65536, 512
    g = torch.Generator(device="cuda").manual_seed(2309)
    lo = -torch.randn(S, L, device="cuda", generator=g).abs() * 2.0 - 0.05
    ln = lo + 0.15 * torch.randn(S, L, device="cuda", generator=g)
    adv = 1.5 * torch.randn(S, L, device="cuda", generator=g) + 0.3
    ret = torch.randn(S, L, device="cuda", generator=g)
    val = ret + 0.5 * torch.randn(S, L, device="cuda", generator=g)
    lengths = torch.randint(64, 513, (S,), device="cuda", generator=g, dtype=torch.int32)
    gl, gv = torch.empty_like(ln), torch.empty_like(ln)
    stats = torch.zeros(7, dtype=torch.float64, device="cuda")
    ws = torch.empty(H.ppo_workspace_size(), dtype=torch.uint8, device="cuda")
    H.hydra_ppo_loss(ln, lo, adv, ret, val, lengths, 0.2, True, gl, gv, stats, ws)
    torch.cuda.synchronize()
    assert H.device_error(clear=True) == 0
    host = [t.cpu().numpy() for t in (ln, lo, adv, ret, val)]
    lens = lengths.cpu().numpy()
    ref = O.ppo_loss(*host, lens, clip_eps=0.2, whiten=True)
    st = stats.cpu().numpy()
    assert st[6] == ref["n"]
    for i, k in enumerate(("loss_clip", "loss_value", "clip_frac", "approx_kl", "adv_mean", "adv_std")):
        assert abs(st[i] - ref[k]) <= 5e-5 * max(1.0, abs(ref[k])), (k, st[i], ref[k])
    rows = np.random.default_rng(0).choice(S, 64, replace=False)
    sub = [a[rows] for a in host]
    moments = (ref["n"], ref["adv_mean"], ref["adv_std"] ** 2 * ref["n"])
    got = (gl[rows].cpu().double().numpy(), gv[rows].cpu().double().numpy(),
           np.array([0.0] * 6 + [ref["n"]]))
    rs = O.ppo_loss(*sub, lens[rows], clip_eps=0.2, whiten=True, moments=moments)
    r = np.exp(sub[0].astype(np.float64) - sub[1])
    valid = np.arange(L)[None, :] < lens[rows][:, None]
    amb = valid & ((np.abs(r - 1.2) <= 1e-5) | (np.abs(r - 0.8) <= 1e-5))
    scale = np.abs(rs["grad_logp"]).max()
    ok = np.abs(got[0] - rs["grad_logp"]) <= 1e-5 * np.abs(rs["grad_logp"]) + 1e-6 * scale
    assert np.all(ok | amb)
    np.testing.assert_allclose(got[1], rs["grad_values"], rtol=1e-5, atol=1e-7 * np.abs(rs["grad_values"]).max())
