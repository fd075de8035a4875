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
    "hydra_selftest_wait_timeout": (ctypes.c_int, [_vp]),
    "hydra_skinny_linear": (ctypes.c_int, [_vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _c_i64, _c_i64,
                                           _vp, _c_i64, _vp, ctypes.c_int, ctypes.c_int,
                                           ctypes.c_int, _vp]),
    "hydra_dual_linear": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp, _c_i64,
                                         _vp, _vp, ctypes.c_int, ctypes.c_int, _vp]),
    "hydra_dual_linear_ex": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp,
                                            _c_i64, _vp, _vp, ctypes.c_int, ctypes.c_int, _vp]),
    "hydra_dual_linear_rope": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp,
                                              _c_i64, _vp, _vp, _c_i64, _c_i64, _c_i64, _vp,
                                              _vp]),
    "hydra_rope_table": (ctypes.c_int, [_c_i64, _c_i64, ctypes.c_float, _vp, _vp]),
    "hydra_lora_linear_tri_workspace_size": (ctypes.c_size_t, [_c_i64, _c_i64]),
    "hydra_lora_linear_tri": (ctypes.c_int, [_vp, _vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp,
                                             _vp, _vp, _c_i64, ctypes.c_float, _vp, _vp, _vp,
                                             ctypes.c_int, _vp, ctypes.c_size_t, _vp]),
    "hydra_lm_head_logprobs_workspace_size": (ctypes.c_size_t, [_c_i64, _c_i64, _c_i64, _c_i64]),
    "hydra_lm_head_logprobs": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _c_i64, _vp, _vp,
                                              _vp, _c_i64, ctypes.c_float, _vp, _vp, _vp,
                                              ctypes.c_float, _vp, _vp, _vp, _vp, _vp, _vp,
                                              ctypes.c_size_t, _vp]),
    "hydra_lora_linear_noalloc": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _c_i64, _vp, _vp, _vp,
                                                 _c_i64, ctypes.c_float, _vp, _vp, ctypes.c_int,
                                                 _vp]),
    "hydra_token_logprobs_kl": (ctypes.c_int, [_vp, _vp, ctypes.c_int, _c_i64, _c_i64, _c_i64,
                                               _c_i64, _vp, _vp, _vp, ctypes.c_float, _vp, _vp,
                                               _vp, _vp, _vp, _vp]),
    "ppo_gae": (ctypes.c_int, [_vp, _vp, _vp, _c_i64, _c_i64, ctypes.c_float, ctypes.c_float, _vp,
                               _vp, _vp]),
    "hydra_ppo_workspace_size": (ctypes.c_size_t, []),
    "hydra_ppo_loss": (ctypes.c_int, [_vp, _vp, _vp, _vp, _vp, _vp, _c_i64, _c_i64, ctypes.c_float,
                                      ctypes.c_int, _vp, _vp, _vp, _vp, _vp, ctypes.c_size_t, _vp]),
    "hydra_ppo_adv_moments": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, _vp, _vp, ctypes.c_size_t,
                                             _vp]),
    "hydra_ppo_merge_moments": (ctypes.c_int, [_vp, _c_i64, _vp]),
}


class LlamaConfigC(ctypes.Structure):
    _fields_ = [("n_layers", _c_i64), ("d_model", _c_i64), ("n_heads", _c_i64),
                ("head_dim", _c_i64), ("ffn", _c_i64), ("vocab", _c_i64),
                ("prompt_len", _c_i64), ("response_len", _c_i64), ("lora_rank", _c_i64),
                ("lora_scale", ctypes.c_float), ("rms_eps", ctypes.c_float),
                ("rope_theta", ctypes.c_float), ("beta", ctypes.c_float),
                ("gamma", ctypes.c_float), ("lam", ctypes.c_float)]


class LlamaLayerC(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("w_qkv", "a_qv", "b_qkv", "w_o", "w_gu", "a_gu", "b_gu",
                                   "w_down", "a_down", "b_down", "norm_attn", "norm_ffn")]


class LlamaLoraC(ctypes.Structure):
    _fields_ = [(n, _vp) for n in ("a_qv", "b_qkv", "a_gu", "b_gu", "a_down", "b_down")]


class LlamaWeightsC(ctypes.Structure):
    _fields_ = [("embed", _vp), ("layers", ctypes.POINTER(LlamaLayerC)), ("final_norm", _vp),
                ("lm_head", _vp), ("w_rm", _vp)]


_SIGNATURES.update({
    "hydra_embed": (ctypes.c_int, [_vp, _c_i64, _c_i64, _vp, _c_i64, ctypes.c_int, _vp, _vp]),
    "hydra_rmsnorm": (ctypes.c_int, [_vp, _vp, _c_i64, _c_i64, ctypes.c_float, _c_i64, _c_i64,
                                     _c_i64, _vp, _vp]),
    "hydra_rope": (ctypes.c_int, [_vp, _c_i64, _c_i64, _c_i64, _c_i64, _c_i64, ctypes.c_float,
                                  _vp]),
    "hydra_causal_attention": (ctypes.c_int, [_vp, _c_i64, _c_i64, _c_i64, _c_i64, _c_i64, _vp,
                                              _c_i64, _vp]),
    "hydra_swiglu": (ctypes.c_int, [_vp, _c_i64, _c_i64, _vp, _vp]),
    "hydra_residual_add": (ctypes.c_int, [_vp, _vp, _c_i64, _vp]),
    "hydra_head_dot": (ctypes.c_int, [_vp, _c_i64, _vp, _c_i64, _c_i64, _c_i64, _c_i64, _vp,
                                      _vp]),
    "hydra_profile_enable": (ctypes.c_int, [ctypes.c_int]),
    "hydra_profile_collect": (ctypes.c_int, [ctypes.POINTER(ctypes.c_float),
                                             ctypes.POINTER(ctypes.c_int64), ctypes.c_int]),
    "hydra_generate_llama_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(LlamaConfigC),
                                                              _c_i64]),
    "hydra_generate_llama": (ctypes.c_int, [ctypes.POINTER(LlamaConfigC),
                                            ctypes.POINTER(LlamaWeightsC), _vp, _c_i64, _c_i64,
                                            _vp, _vp, ctypes.c_size_t, _vp, _vp, _vp, _vp, _vp,
                                            _vp]),
    "hydra_score_llama_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(LlamaConfigC),
                                                           _c_i64]),
    "hydra_score_llama": (ctypes.c_int, [ctypes.POINTER(LlamaConfigC),
                                         ctypes.POINTER(LlamaWeightsC), _vp, _vp, _c_i64, _vp,
                                         ctypes.c_size_t, _vp, _vp, _vp, _vp, _vp, _vp, _vp,
                                         _vp]),
    "hydra_score_llama_hydra_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(LlamaConfigC),
                                                                 _c_i64]),
    "hydra_score_llama_hydra": (ctypes.c_int, [ctypes.POINTER(LlamaConfigC),
                                               ctypes.POINTER(LlamaWeightsC),
                                               ctypes.POINTER(LlamaLoraC), _vp, _vp, _c_i64,
                                               _vp, ctypes.c_size_t, _vp, _vp, _vp, _vp, _vp,
                                               _vp, _vp, _vp]),
})

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


def _out_dtype(t, name="output"):
    """HYDRA_BF16 or HYDRA_F32 for an output tensor; any other dtype is refused."""
    if t.dtype == torch.float32:
        return HYDRA_F32
    if t.dtype == torch.bfloat16:
        return HYDRA_BF16
    raise ValueError(f"{name} must be torch.bfloat16 or torch.float32, got {t.dtype}")


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


def selftest_wait_timeout(stream=None):
    """Launch the bounded-wait self-test: about 1 s later the device error word holds 0x105."""
    _check("hydra_selftest_wait_timeout", load().hydra_selftest_wait_timeout(_stream(stream)))


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
    out_dtype = _out_dtype(out)
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
    out_dtype = _out_dtype(out)
    for t, n in ((y_off, "y_off"), (y_on, "y_on")):
        _req(t, out.dtype, n)
    M, K = x_off.shape
    N = W.shape[0]
    r = 0 if u is None else u.shape[1]
    _check("hydra_dual_linear", load().hydra_dual_linear(
        _p(x_off), _p(x_on), M, K, N, _p(W), _p(u), _p(B), r, _p(y_off), _p(y_on), out_dtype,
        int(algo), _stream(stream)))


def hydra_skinny_linear(x, W, y, u=None, B=None, u_row0=0, tile_n=0, split_k=0, stream=None):
    """Decode-step linear over both streams' rows stacked in x (at most 128): y = x W^T, plus
    u B^T on rows [u_row0, u_row0 + len(u)) (u None: no LoRA). tile_n / split_k 0: chosen by
    the library."""
    for t, n in ((x, "x"), (W, "W"), (u, "u"), (B, "B")):
        _req(t, torch.bfloat16, n)
    out_dtype = _out_dtype(y)
    _req(y, y.dtype, "y")
    M, K = x.shape
    N = W.shape[0]
    r = 0 if u is None else u.shape[1]
    u_rows = 0 if u is None else u.shape[0]
    _check("hydra_skinny_linear", load().hydra_skinny_linear(
        _p(x), M, K, N, _p(W), _p(u), int(u_row0), u_rows, _p(B), r, _p(y), out_dtype,
        int(tile_n), int(split_k), _stream(stream)))


def hydra_lora_linear_noalloc(x_off, x_on, W, A, B, s, y_off, y_on, stream=None):
    """hydra_lora_linear without a workspace: u lives in the library's static device array
    (M * r <= HYDRA_NOALLOC_MAX_U_ELEMS), for callers that cannot allocate device memory."""
    for t, n in ((x_off, "x_off"), (x_on, "x_on"), (W, "W"), (A, "A"), (B, "B")):
        _req(t, torch.bfloat16, n)
    out = y_off if y_off is not None else y_on
    out_dtype = _out_dtype(out)
    for t, n in ((y_off, "y_off"), (y_on, "y_on")):
        _req(t, out.dtype, n)
    M, K = x_off.shape
    N = W.shape[0]
    r = 0 if A is None else A.shape[0]
    _check("hydra_lora_linear_noalloc", load().hydra_lora_linear_noalloc(
        _p(x_off), _p(x_on), M, K, N, _p(W), _p(A), _p(B), r, float(s), _p(y_off), _p(y_on),
        out_dtype, _stream(stream)))


EPI_STORE, EPI_SWIGLU, EPI_RESIDUAL = 0, 1, 2


def hydra_dual_linear_ex(x_off, x_on, W, u, B, y_off, y_on, epilogue, stream=None):
    """tcgen05 dual linear with a fused epilogue (EPI_STORE, EPI_SWIGLU: bf16 [M, N/2] from
    128-row-interleaved gate/up weights, EPI_RESIDUAL: fp32 [M, N] += bf16 result)."""
    for t, n in ((x_off, "x_off"), (x_on, "x_on"), (W, "W"), (u, "u"), (B, "B")):
        _req(t, torch.bfloat16, n)
    out = y_off if y_off is not None else y_on
    out_dtype = _out_dtype(out)
    for t, n in ((y_off, "y_off"), (y_on, "y_on")):
        _req(t, out.dtype, n)
    M, K = x_off.shape
    N = W.shape[0]
    r = 0 if u is None else u.shape[1]
    _check("hydra_dual_linear_ex", load().hydra_dual_linear_ex(
        _p(x_off), _p(x_on), M, K, N, _p(W), _p(u), _p(B), r, _p(y_off), _p(y_on), out_dtype,
        int(epilogue), _stream(stream)))


def hydra_rope_table(P, head_dim, theta, table, stream=None):
    """(cos, sin) of the rotary angles: table fp32 [P, head_dim // 2, 2]."""
    _req(table, torch.float32, "table")
    _check("hydra_rope_table", load().hydra_rope_table(int(P), int(head_dim), float(theta),
                                                       _p(table), _stream(stream)))


def hydra_dual_linear_rope(x_off, x_on, W, u, B, y_off, y_on, P, rope_cols, head_dim, table,
                           stream=None):
    """tcgen05 dual linear (bf16 outputs) with the rotary embedding of columns
    [0, rope_cols) fused into the epilogue, angles from hydra_rope_table; equal to
    hydra_dual_linear + hydra_rope."""
    _req(table, torch.float32, "table")
    for t, n in ((x_off, "x_off"), (x_on, "x_on"), (W, "W"), (u, "u"), (B, "B"),
                 (y_off, "y_off"), (y_on, "y_on")):
        _req(t, torch.bfloat16, n)
    M, K = x_off.shape
    N = W.shape[0]
    r = 0 if u is None else u.shape[1]
    _check("hydra_dual_linear_rope", load().hydra_dual_linear_rope(
        _p(x_off), _p(x_on), M, K, N, _p(W), _p(u), _p(B), r, _p(y_off), _p(y_on), int(P),
        int(rope_cols), int(head_dim), _p(table), _stream(stream)))


def lora_linear_tri_workspace_size(M, r):
    return int(load().hydra_lora_linear_tri_workspace_size(M, r))


def hydra_lora_linear_tri(x_off, x_act, x_crit, W, A_act, B_act, A_crit, B_crit, s, y_off, y_act,
                          y_crit, workspace=None, stream=None):
    """Hydra-PPO's off / actor / critic streams through one W (two LoRA sets)."""
    for t, n in ((x_off, "x_off"), (x_act, "x_act"), (x_crit, "x_crit"), (W, "W"),
                 (A_act, "A_act"), (B_act, "B_act"), (A_crit, "A_crit"), (B_crit, "B_crit")):
        _req(t, torch.bfloat16, n)
    out = next(t for t in (y_off, y_act, y_crit) if t is not None)
    out_dtype = _out_dtype(out)
    for t, n in ((y_off, "y_off"), (y_act, "y_act"), (y_crit, "y_crit")):
        _req(t, out.dtype, n)
    M, K = x_off.shape
    N = W.shape[0]
    A = A_act if A_act is not None else A_crit
    r = 0 if A is None else A.shape[0]
    wsb = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check("hydra_lora_linear_tri", load().hydra_lora_linear_tri(
        _p(x_off), _p(x_act), _p(x_crit), M, K, N, _p(W), _p(A_act), _p(B_act), _p(A_crit),
        _p(B_crit), r, float(s), _p(y_off), _p(y_act), _p(y_crit), out_dtype, _p(workspace), wsb,
        _stream(stream)))


def lm_head_logprobs_workspace_size(S, L, V, r):
    return int(load().hydra_lm_head_logprobs_workspace_size(S, L, V, r))


def hydra_lm_head_logprobs(h_off, h_on, W, A, B, s, ids, lengths, seq_score, beta, S, L,
                           logp_actor, logp_ref, reward_tok, workspace, lse_actor=None,
                           lse_ref=None, stream=None):
    """Dual LM head + log-probabilities/KL without materialised logits. h_*: bf16 [S*L, d]
    (h_on None: shared input); W bf16 [V, d]; A/B the actor head's LoRA (None: none)."""
    for t, n in ((h_off, "h_off"), (h_on, "h_on"), (W, "W"), (A, "A"), (B, "B")):
        _req(t, torch.bfloat16, n)
    _req(ids, torch.int32, "ids")
    _req(lengths, torch.int32, "lengths")
    for t, n in ((seq_score, "seq_score"), (logp_actor, "logp_actor"), (logp_ref, "logp_ref"),
                 (reward_tok, "reward_tok"), (lse_actor, "lse_actor"), (lse_ref, "lse_ref")):
        _req(t, torch.float32, n)
    d = h_off.shape[1]
    V = W.shape[0]
    r = 0 if A is None else A.shape[0]
    _check("hydra_lm_head_logprobs", load().hydra_lm_head_logprobs(
        _p(h_off), _p(h_on), S, L, d, V, _p(W), _p(A), _p(B), r, float(s), _p(ids), _p(lengths),
        _p(seq_score), float(beta), _p(logp_actor), _p(logp_ref), _p(reward_tok), _p(lse_actor),
        _p(lse_ref), _p(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))


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


PPO_STATS = ("loss_clip", "loss_value", "clip_frac", "approx_kl", "adv_mean", "adv_std", "n")


def ppo_workspace_size():
    return int(load().hydra_ppo_workspace_size())


def hydra_ppo_loss(logp_new, logp_old, advantages, returns, values, lengths, clip_eps, whiten,
                   grad_logp, grad_values, stats, workspace, adv_moments=None, stream=None):
    """Clipped surrogate, value loss and their gradients over [S, L] fp32 tensors; stats is a
    device fp64 [7] tensor (order PPO_STATS); adv_moments an optional device fp64 [3]."""
    for t, n in ((logp_new, "logp_new"), (logp_old, "logp_old"), (advantages, "advantages"),
                 (returns, "returns"), (values, "values"), (grad_logp, "grad_logp"),
                 (grad_values, "grad_values")):
        _req(t, torch.float32, n)
    _req(lengths, torch.int32, "lengths")
    _req(stats, torch.float64, "stats")
    _req(adv_moments, torch.float64, "adv_moments")
    S, L = logp_new.shape
    _check("hydra_ppo_loss", load().hydra_ppo_loss(
        _p(logp_new), _p(logp_old), _p(advantages), _p(returns), _p(values), _p(lengths), S, L,
        float(clip_eps), int(bool(whiten)), _p(adv_moments), _p(grad_logp), _p(grad_values),
        _p(stats), _p(workspace), workspace.numel() * workspace.element_size(), _stream(stream)))


def hydra_ppo_adv_moments(advantages, lengths, moments, workspace, stream=None):
    """(n, mean, M2) of the valid advantages into the device fp64 [3] tensor moments."""
    _req(advantages, torch.float32, "advantages")
    _req(lengths, torch.int32, "lengths")
    _req(moments, torch.float64, "moments")
    S, L = advantages.shape
    _check("hydra_ppo_adv_moments", load().hydra_ppo_adv_moments(
        _p(advantages), _p(lengths), S, L, _p(moments), _p(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)))


def ppo_merge_moments(triples):
    """Merge host (n, mean, M2) triples (a [k, 3] fp64 CPU tensor, rank order) in the library."""
    t = torch.as_tensor(triples, dtype=torch.float64).contiguous().reshape(-1, 3)
    out = torch.zeros(3, dtype=torch.float64)
    _check("hydra_ppo_merge_moments", load().hydra_ppo_merge_moments(
        t.data_ptr() if t.numel() else None, t.shape[0], out.data_ptr()))
    return out


def all_reduce_adv_moments(moments, group=None):
    """Replace each rank's (n, mean, M2) by the merge over all ranks (all_gather of three
    doubles, merged in rank order on the host, so every rank gets the same bits)."""
    import torch.distributed as dist
    host = moments.detach().to("cpu", torch.float64).reshape(3)
    world = dist.get_world_size(group)
    parts = [torch.zeros(3, dtype=torch.float64) for _ in range(world)]
    if dist.get_backend(group) == "nccl":
        dev = moments.device
        gathered = [torch.zeros(3, dtype=torch.float64, device=dev) for _ in range(world)]
        dist.all_gather(gathered, host.to(dev), group=group)
        parts = [g.cpu() for g in gathered]
    else:
        dist.all_gather(parts, host, group=group)
    merged = ppo_merge_moments(torch.stack(parts))
    moments.copy_(merged.to(moments.device))
    return moments


# ----------------------------------------------------------------------------- Llama pieces


def hydra_embed(table, ids, copies, h, stream=None):
    _req(table, torch.bfloat16, "table")
    _req(ids, torch.int32, "ids")
    _req(h, torch.float32, "h")
    V, d = table.shape
    _check("hydra_embed", load().hydra_embed(_p(table), V, d, _p(ids), ids.numel(), int(copies),
                                             _p(h), _stream(stream)))


def hydra_rmsnorm(x, w, eps, y, rows=None, g_out=None, g_in=None, off=0, stream=None):
    """y[i] = bf16(RMSNorm(x[j]) * w), j = (i // g_out) * g_in + off + i % g_out."""
    _req(x, torch.float32, "x")
    _req(w, torch.bfloat16, "w")
    _req(y, torch.bfloat16, "y")
    d = x.shape[-1]
    rows = y.shape[0] if rows is None else rows
    g_out = rows if g_out is None else g_out
    g_in = g_out if g_in is None else g_in
    _check("hydra_rmsnorm", load().hydra_rmsnorm(_p(x), _p(w), rows, d, float(eps), g_out, g_in,
                                                 off, _p(y), _stream(stream)))


def hydra_rope(qkv, d, head_dim, P, theta, stream=None):
    _req(qkv, torch.bfloat16, "qkv")
    R, ld = qkv.shape
    _check("hydra_rope", load().hydra_rope(_p(qkv), R, ld, d, head_dim, P, float(theta),
                                           _stream(stream)))


def hydra_causal_attention(qkv, nseq, P, n_heads, head_dim, out, stream=None):
    _req(qkv, torch.bfloat16, "qkv")
    _req(out, torch.bfloat16, "out")
    _check("hydra_causal_attention", load().hydra_causal_attention(
        _p(qkv), nseq, P, qkv.shape[1], n_heads, head_dim, _p(out), out.shape[1],
        _stream(stream)))


def hydra_swiglu(gu, m, stream=None):
    _req(gu, torch.bfloat16, "gu")
    _req(m, torch.bfloat16, "m")
    _check("hydra_swiglu", load().hydra_swiglu(_p(gu), gu.shape[0], m.shape[1], _p(m),
                                               _stream(stream)))


def hydra_residual_add(h, y, stream=None):
    _req(h, torch.float32, "h")
    _req(y, torch.bfloat16, "y")
    _check("hydra_residual_add", load().hydra_residual_add(_p(h), _p(y), h.numel(),
                                                           _stream(stream)))


def hydra_head_dot(x, w, out, g_out=None, g_in=None, off=0, stream=None):
    _req(x, torch.bfloat16, "x")
    _req(w, torch.bfloat16, "w")
    _req(out, torch.float32, "out")
    n = out.numel()
    g_out = n if g_out is None else g_out
    g_in = g_out if g_in is None else g_in
    _check("hydra_head_dot", load().hydra_head_dot(_p(x), x.shape[-1], _p(w), n, g_out, g_in, off,
                                                   _p(out), _stream(stream)))


def llama_config_c(cfg):
    """hydra_llama_config from a dict with the keys of LlamaConfigC."""
    return LlamaConfigC(**{k: cfg[k] for k, _ in LlamaConfigC._fields_})


def score_llama_workspace_size(cfg, S):
    c = llama_config_c(cfg)
    return int(load().hydra_score_llama_workspace_size(ctypes.byref(c), S))


def score_llama_hydra_workspace_size(cfg, S):
    c = llama_config_c(cfg)
    return int(load().hydra_score_llama_hydra_workspace_size(ctypes.byref(c), S))


def _weights_c(cfg, weights):
    n = cfg["n_layers"]
    layers = (LlamaLayerC * n)()
    for l in range(n):
        for name, _ in LlamaLayerC._fields_:
            t = weights[name][l]
            _req(t, torch.bfloat16, name)
            setattr(layers[l], name, t.data_ptr())
    for name in ("embed", "final_norm", "lm_head", "w_rm"):
        _req(weights[name], torch.bfloat16, name)
    w = LlamaWeightsC(weights["embed"].data_ptr(), layers, weights["final_norm"].data_ptr(),
                      weights["lm_head"].data_ptr(), weights["w_rm"].data_ptr())
    return w, layers


def hydra_score_llama_hydra(cfg, weights, critic, ids, lengths, workspace, outputs, stream=None):
    """Hydra-PPO scoring pass: as hydra_score_llama with the critic's LoRA set critic (dict of
    per-layer lists a_qv, b_qkv, a_gu, b_gu, a_down, b_down in the fused layouts) as a third
    stream whose final hidden states give the values."""
    c = llama_config_c(cfg)
    w, _layers = _weights_c(cfg, weights)
    n = cfg["n_layers"]
    crit = (LlamaLoraC * n)()
    for l in range(n):
        for name, _ in LlamaLoraC._fields_:
            t = critic[name][l]
            _req(t, torch.bfloat16, name)
            setattr(crit[l], name, t.data_ptr())
    _req(ids, torch.int32, "ids")
    _req(lengths, torch.int32, "lengths")
    names = ("logp_actor", "logp_ref", "reward", "values", "advantages", "returns", "score")
    for k in names:
        _req(outputs[k], torch.float32, k)
    ws_bytes = workspace.numel() * workspace.element_size()
    _check("hydra_score_llama_hydra", load().hydra_score_llama_hydra(
        ctypes.byref(c), ctypes.byref(w), crit, _p(ids), _p(lengths), ids.shape[0], _p(workspace),
        ws_bytes, *[_p(outputs[k]) for k in names], _stream(stream)))


def hydra_score_llama(cfg, weights, ids, lengths, workspace, outputs, stream=None):
    """Full J-Hydra scoring pass. cfg: dict (LlamaConfigC keys); weights: dict of device
    tensors in the fused layouts (see include/hydra.h: embed, final_norm, lm_head, w_rm and
    per-layer lists w_qkv, a_qv, b_qkv, w_o, w_gu, a_gu, b_gu, w_down, a_down, b_down,
    norm_attn, norm_ffn); ids int32 [S, P0 + L]; lengths int32 [S] or None; outputs: dict
    with fp32 logp_actor, logp_ref, reward, values, advantages, returns [S, L], score [S]."""
    c = llama_config_c(cfg)
    n = cfg["n_layers"]
    layers = (LlamaLayerC * n)()
    for l in range(n):
        for name, _ in LlamaLayerC._fields_:
            t = weights[name][l]
            _req(t, torch.bfloat16, name)
            setattr(layers[l], name, t.data_ptr())
    for name in ("embed", "final_norm", "lm_head", "w_rm"):
        _req(weights[name], torch.bfloat16, name)
    w = LlamaWeightsC(weights["embed"].data_ptr(), layers, weights["final_norm"].data_ptr(),
                      weights["lm_head"].data_ptr(), weights["w_rm"].data_ptr())
    _req(ids, torch.int32, "ids")
    _req(lengths, torch.int32, "lengths")
    names = ("logp_actor", "logp_ref", "reward", "values", "advantages", "returns", "score")
    for k in names:
        _req(outputs[k], torch.float32, k)
    S = ids.shape[0]
    ws_bytes = workspace.numel() * workspace.element_size()
    _check("hydra_score_llama", load().hydra_score_llama(
        ctypes.byref(c), ctypes.byref(w), _p(ids), _p(lengths), S, _p(workspace), ws_bytes,
        *[_p(outputs[k]) for k in names], _stream(stream)))


def generate_llama_workspace_size(cfg, S):
    c = llama_config_c(cfg)
    return int(load().hydra_generate_llama_workspace_size(ctypes.byref(c), S))


def hydra_generate_llama(cfg, weights, prompt_ids, n_steps, gumbel, workspace, outputs,
                         stream=None):
    """KV-cached generation with the actor plus the LoRA-off stream. prompt_ids int32
    [S, P0]; gumbel fp32 [n_steps, S, V] or None (greedy); outputs: dict with int32 tokens
    and fp32 logp_actor, logp_ref, values [S, n_steps], and fp32 score [S] or None."""
    c = llama_config_c(cfg)
    w, _layers = _weights_c(cfg, weights)
    _req(prompt_ids, torch.int32, "prompt_ids")
    _req(gumbel, torch.float32, "gumbel")
    _req(outputs["tokens"], torch.int32, "tokens")
    for k in ("logp_actor", "logp_ref", "values"):
        _req(outputs[k], torch.float32, k)
    _req(outputs.get("score"), torch.float32, "score")
    S = prompt_ids.shape[0]
    ws_bytes = workspace.numel() * workspace.element_size()
    _check("hydra_generate_llama", load().hydra_generate_llama(
        ctypes.byref(c), ctypes.byref(w), _p(prompt_ids), S, int(n_steps), _p(gumbel),
        _p(workspace), ws_bytes, _p(outputs["tokens"]), _p(outputs["logp_actor"]),
        _p(outputs["logp_ref"]), _p(outputs["values"]), _p(outputs.get("score")),
        _stream(stream)))


PROF_CLASSES = ("gemm_qkv", "gemm_o", "gemm_gu", "gemm_down", "gemm_lmhead", "lora_down",
                "attention", "elementwise", "logprobs", "gae", "heads")
GEMM_CLASSES = PROF_CLASSES[:5]


def profile_enable(on=True):
    _check("hydra_profile_enable", load().hydra_profile_enable(int(bool(on))))


def profile_collect(reset=True):
    """{class: (ms, launches)} summed since the last reset."""
    n = len(PROF_CLASSES)
    ms = (ctypes.c_float * n)()
    cnt = (ctypes.c_int64 * n)()
    _check("hydra_profile_collect", load().hydra_profile_collect(ms, cnt, int(reset)))
    return {k: (float(ms[i]), int(cnt[i])) for i, k in enumerate(PROF_CLASSES)}
