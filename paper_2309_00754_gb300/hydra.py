"""ctypes binding of libhydra (include/hydra.h): same entry-point names, argument
marshalling only. Tensors are torch CUDA tensors (PyTorch provides device memory and
streams); every computation runs in the library's kernels. There is no fallback: if the
library is missing or a call fails, an exception is raised."""
from __future__ import annotations

import ctypes
import os
import re

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libhydra.so")
HEADER = os.path.join(os.path.dirname(_PKG), "include", "hydra.h")

HYDRA_BF16 = 0
HYDRA_F32 = 1

_c_i64 = ctypes.c_int64
_vp = ctypes.c_void_p

_SIGNATURES = {
    "hydra_status_string": (ctypes.c_char_p, [ctypes.c_int]),
    "hydra_abi_version": (ctypes.c_int, []),
    "hydra_device_error": (ctypes.c_int, [ctypes.POINTER(ctypes.c_int32), ctypes.c_int]),
    "hydra_lora_down": (ctypes.c_int, [_vp, _c_i64, _c_i64, _vp, _c_i64, ctypes.c_float, _vp, _vp]),
    "hydra_lora_linear_workspace_size": (ctypes.c_size_t, [_c_i64, _c_i64]),
    "hydra_lora_linear": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp, _c_i64,
                                         ctypes.c_float, _vp, _vp, ctypes.c_int, _vp,
                                         ctypes.c_size_t, _vp]),
    "hydra_lora_linear_algo": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp,
                                              _c_i64, ctypes.c_float, _vp, _vp, ctypes.c_int, _vp,
                                              ctypes.c_size_t, ctypes.c_int, _vp]),
    "hydra_dual_linear": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp, _c_i64,
                                         _vp, _vp, ctypes.c_int, ctypes.c_int, _vp]),
    "hydra_lora_linear_noalloc": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp,
                                                 _c_i64, ctypes.c_float, _vp, _vp, ctypes.c_int,
                                                 _vp]),
    "hydra_token_logprobs_kl": (ctypes.c_int, [_vp, _vp, ctypes.c_int, _c_i64, _c_i64, _c_i64,
                                               _c_i64, _vp, _vp, _vp, ctypes.c_float, _vp, _vp,
                                               _vp, _vp, _vp, _vp]),
    "ppo_gae": (ctypes.c_int, [_vp, _vp, _vp, _c_i64, _c_i64, ctypes.c_float, ctypes.c_float, _vp,
                               _vp, _vp]),
}

_lib = None


class HydraError(RuntimeError):
    def __init__(self, fn, status):
        self.status = status
        super().__init__(f"{fn} failed: {status_string(status)}")


def load():
    """Load libhydra.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with __graft_entry__.build() "
                               "or python -m paper_2309_00754_gb300.build")
        lib = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in _SIGNATURES.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
    return _lib


def header_functions():
    """Names of the functions declared in include/hydra.h."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b([a-z_][a-z0-9_]*)\s*\(", text)) -
                  {"if", "sizeof", "defined"})


def status_string(status: int) -> str:
    return load().hydra_status_string(int(status)).decode()


def _check(fn, status):
    if status != 0:
        raise HydraError(fn, status)


def _p(t):
    return None if t is None else t.data_ptr()


def _stream(stream):
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def _req(t, dtype, name):
    if t is None:
        return
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")


def device_error(clear: bool = True) -> int:
    code = ctypes.c_int32(0)
    _check("hydra_device_error", load().hydra_device_error(ctypes.byref(code), int(clear)))
    return code.value


def lora_linear_workspace_size(M: int, r: int) -> int:
    return int(load().hydra_lora_linear_workspace_size(M, r))


def hydra_lora_down(x_on, A, s, u, stream=None):
    _req(x_on, torch.bfloat16, "x_on")
    _req(A, torch.bfloat16, "A")
    _req(u, torch.bfloat16, "u")
    M, K = x_on.shape
    r = A.shape[0]
    _check("hydra_lora_down", load().hydra_lora_down(_p(x_on), M, K, _p(A), r, float(s), _p(u),
                                                     _stream(stream)))


def hydra_lora_linear(x_off, x_on, W, A, B, s, y_off, y_on, workspace=None, algo=0, stream=None):
    """y_off = x_off W^T, y_on = x_on W^T + s (x_on A^T) B^T (x_on None/x_off: shared input).
    Outputs are preallocated [M, N] bf16 or fp32 tensors (either may be None)."""
    for t, n in ((x_off, "x_off"), (x_on, "x_on"), (W, "W"), (A, "A"), (B, "B")):
        _req(t, torch.bfloat16, n)
    out = y_off if y_off is not None else y_on
    out_dtype = HYDRA_F32 if out.dtype == torch.float32 else HYDRA_BF16
    for t, n in ((y_off, "y_off"), (y_on, "y_on")):
        _req(t, out.dtype, n)
    M, K = x_off.shape
    N = W.shape[0]
    r = 0 if A is None else A.shape[0]
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check("hydra_lora_linear", load().hydra_lora_linear_algo(
        _p(x_off), _p(x_on), M, K, N, _p(W), _p(A), _p(B), r, float(s), _p(y_off), _p(y_on),
        out_dtype, _p(workspace), ws_bytes, int(algo), _stream(stream)))


def hydra_dual_linear(x_off, x_on, W, u, B, y_off, y_on, algo=0, stream=None):
    """y_off = x_off W^T, y_on = x_on W^T + u B^T with u from hydra_lora_down (None: no LoRA)."""
    for t, n in ((x_off, "x_off"), (x_on, "x_on"), (W, "W"), (u, "u"), (B, "B")):
        _req(t, torch.bfloat16, n)
    out = y_off if y_off is not None else y_on
    out_dtype = HYDRA_F32 if out.dtype == torch.float32 else HYDRA_BF16
    for t, n in ((y_off, "y_off"), (y_on, "y_on")):
        _req(t, out.dtype, n)
    M, K = x_off.shape
    N = W.shape[0]
    r = 0 if u is None else u.shape[1]
    _check("hydra_dual_linear", load().hydra_dual_linear(
        _p(x_off), _p(x_on), M, K, N, _p(W), _p(u), _p(B), r, _p(y_off), _p(y_on), out_dtype,
        int(algo), _stream(stream)))


def hydra_lora_linear_noalloc(x_off, x_on, W, A, B, s, y_off, y_on, stream=None):
    """hydra_lora_linear without a workspace: u lives in the library's static device array
    (M * r <= HYDRA_NOALLOC_MAX_U_ELEMS), for callers that cannot allocate device memory."""
    for t, n in ((x_off, "x_off"), (x_on, "x_on"), (W, "W"), (A, "A"), (B, "B")):
        _req(t, torch.bfloat16, n)
    out = y_off if y_off is not None else y_on
    out_dtype = HYDRA_F32 if out.dtype == torch.float32 else HYDRA_BF16
    for t, n in ((y_off, "y_off"), (y_on, "y_on")):
        _req(t, out.dtype, n)
    M, K = x_off.shape
    N = W.shape[0]
    r = 0 if A is None else A.shape[0]
    _check("hydra_lora_linear_noalloc", load().hydra_lora_linear_noalloc(
        _p(x_off), _p(x_on), M, K, N, _p(W), _p(A), _p(B), r, float(s), _p(y_off), _p(y_on),
        out_dtype, _stream(stream)))


def hydra_token_logprobs_kl(logits_actor, logits_ref, ids, lengths, seq_score, beta, S, L,
                            logp_actor, logp_ref, reward_tok, lse_actor=None, lse_ref=None,
                            stream=None):
    """Sampled-token log-probabilities under both heads and the KL-penalised reward.
    logits_*: [S*L, V] (row stride may exceed V), fp32 or bf16; outputs fp32 [S*L]."""
    dt = logits_actor.dtype
    if dt not in (torch.float32, torch.bfloat16) or logits_ref.dtype != dt:
        raise ValueError("logits must both be float32 or both bfloat16")
    if logits_actor.stride(1) != 1 or logits_ref.stride(1) != 1 or \
            logits_actor.stride(0) != logits_ref.stride(0):
        raise ValueError("logit rows must be unit-stride with one common row stride")
    _req(ids, torch.int32, "ids")
    _req(lengths, torch.int32, "lengths")
    _req(seq_score, torch.float32, "seq_score")
    for t, n in ((logp_actor, "logp_actor"), (logp_ref, "logp_ref"), (reward_tok, "reward_tok"),
                 (lse_actor, "lse_actor"), (lse_ref, "lse_ref")):
        _req(t, torch.float32, n)
    V = logits_actor.shape[1]
    ld = logits_actor.stride(0)
    _check("hydra_token_logprobs_kl", load().hydra_token_logprobs_kl(
        _p(logits_actor), _p(logits_ref), HYDRA_F32 if dt == torch.float32 else HYDRA_BF16, S, L,
        V, ld, _p(ids), _p(lengths), _p(seq_score), float(beta), _p(logp_actor), _p(logp_ref),
        _p(reward_tok), _p(lse_actor), _p(lse_ref), _stream(stream)))


def ppo_gae(rewards, values, lengths, gamma, lam, advantages, returns, stream=None):
    """GAE advantages and returns over [S, L] fp32 rewards/values (lengths int32 [S] or None)."""
    for t, n in ((rewards, "rewards"), (values, "values"), (advantages, "advantages"),
                 (returns, "returns")):
        _req(t, torch.float32, n)
    _req(lengths, torch.int32, "lengths")
    S, L = rewards.shape
    _check("ppo_gae", load().ppo_gae(_p(rewards), _p(values), _p(lengths), S, L, float(gamma),
                                     float(lam), _p(advantages), _p(returns), _stream(stream)))
