"""Thin Python binding of the C ABI in ``include/rl_loss.h``.

Argument marshalling only: each function checks the tensors it is handed
(device, dtype, size, contiguity), passes their device pointers and the
current CUDA stream to the library function of the same name, and raises
``RLError`` on a non-OK status. Every step of the computation runs in the
library's CUDA kernels; there is no fallback path. PyTorch only owns memory
and streams.
"""

from __future__ import annotations

import ctypes
import os

import numpy as np
import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "librl_loss.so")

RL_OK = 0
STATUS_NAMES = {0: "RL_OK", 1: "RL_ERR_INVALID_ARG", 2: "RL_ERR_UNSUPPORTED", 3: "RL_ERR_ALIGNMENT",
                4: "RL_ERR_WORKSPACE_TOO_SMALL", 5: "RL_ERR_CUDA", 6: "RL_ERR_DEVICE_CHECK", 7: "RL_ERR_TIMEOUT"}
RL_BF16, RL_F32 = 0, 1
RL_DEV_BAD_TOKEN, RL_DEV_BAD_TRAJ, RL_DEV_BAD_OFFSETS, RL_DEV_TIMEOUT, RL_DEV_BAD_VALUE = 1, 2, 4, 8, 16
AGG_SEQ_MEAN_TOKEN_MEAN, AGG_TOKEN_MEAN, AGG_TOKEN_SUM = 0, 1, 2

# C function name -> (restype, argtypes)
_P = ctypes.c_void_p
_I32, _I64, _SZ, _F = ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_float
EXPORTS = {
    "rl_version": (_I32, []),
    "rl_last_error_message": (ctypes.c_char_p, []),
    "rl_workspace_size": (_SZ, [_I64, _I64, _I64]),
    "rl_workspace_init": (_I32, [_P, _SZ, _P]),
    "rl_fused_head_workspace_size": (_SZ, [_I64, _I64, _I64, _I64]),
    "rl_query_status": (_I32, [_P, _P, ctypes.POINTER(_I32)]),
    "rl_selftest_bounded_wait": (_I32, [_P, _SZ, _I64, _P, _P]),
    "rl_group_advantages": (_I32, [_I32, _I32, _P, _P, _P, _I64, _P, _P, _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "rl_token_logprobs": (_I32, [_P, _I32, _I64, _I64, _I64, _P, _P, _P, _P, _P, _SZ, _P]),
    "rl_policy_loss_fwd_bwd": (_I32, [_P, _I32, _I64, _I64, _I64, _P, _P, _P, _I32, _P, _P, _P, _P, _P, _P,
                                      _P, _P, _P, _P, _SZ, _P]),
    "rl_policy_loss_fwd_bwd_noalloc": (_I32, [_P, _I32, _I64, _I64, _I64, _P, _P, _P, _I32, _P, _P, _P, _P, _P,
                                              _P, _P, _P, _P, _P, _P]),
    "rl_sequence_is_weights": (_I32, [_I32, _I64, _P, _P, _P, _P, _F, _P, _P, _P, _P, _P, _SZ, _P]),
    "rl_prefix_tree_build_batch": (_I32, [_I32, _P, _P, _P, _P, _P, _P, _P, _P, _I32, _I32, _I64, _P, _P, _P, _P,
                                          _P, _P, _P, _P, _P, _P, _P, _P]),
    "rl_group_advantages_by_owner": (_I32, [_I32, _I32, _P, _P, _P, _I64, _P, _P, _P, _P, _P, _P, _P, _SZ, _P]),
    "rl_rollout_value_advantages": (_I32, [_I64, _P, _P, _P, _P, _I32, _P, _P, _P, _SZ, _P]),
    "rl_token_stats_summary": (_I32, [_I64, _P, _P, _P, _I32, _P, _P, _P, _SZ, _P]),
    "rl_masked_gae": (_I32, [_I32, _P, _I64, _P, _P, _P, _P, _F, _F, _I32, _P, _P, _P, _SZ, _P]),
    "rl_value_loss_fwd_bwd": (_I32, [_I64, _P, _P, _P, _P, _I32, _P, _P, _P, _P, _SZ, _P]),
    "rl_fused_head_token_logprobs": (_I32, [_P, _P, _I64, _I64, _I64, _P, _P, _P, _P, _P, _SZ, _P]),
    "rl_fused_head_loss_fwd_bwd": (_I32, [_P, _P, _I64, _I64, _I64, _P, _P, _P, _I32, _P, _P, _P, _P, _P, _P, _P,
                                          _I32, _P, _P, _P, _P, _SZ, _P]),
}


class rl_loss_params(ctypes.Structure):
    _fields_ = [("clip_eps_low", _F), ("clip_eps_high", _F), ("kl_coef", _F), ("kl_estimator", _I32),
                ("entropy_coef", _F), ("tis_cap", _F), ("adv_eps", _F), ("loss_agg", _I32),
                ("token_level_adv", _I32)]


def make_params(clip_eps_low=0.2, clip_eps_high=0.28, kl_coef=0.0, kl_estimator=0, entropy_coef=0.0,
                tis_cap=0.0, adv_eps=1e-6, loss_agg=AGG_SEQ_MEAN_TOKEN_MEAN, token_level_adv=0) -> rl_loss_params:
    return rl_loss_params(clip_eps_low, clip_eps_high, kl_coef, kl_estimator, entropy_coef, tis_cap, adv_eps,
                          loss_agg, int(token_level_adv))


class rl_tree_stats(ctypes.Structure):
    _fields_ = [("valid", _I32), ("n_leaves", _I32), ("n_kept_leaves", _I32), ("n_unplaced", _I32),
                ("n_tokens", _I64), ("n_trainable", _I64)]


class RLError(RuntimeError):
    def __init__(self, fn, status, message):
        super().__init__(f"{fn}: {STATUS_NAMES.get(status, status)}: {message}")
        self.status = status


_lib = None


def lib() -> ctypes.CDLL:
    """Load ``librl_loss.so`` (built by ``build.py``); raises if it is missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: build it with paper_2608_16798_gb300.build.build()")
        handle = ctypes.CDLL(LIB_PATH)
        for name, (res, args) in EXPORTS.items():
            f = getattr(handle, name)
            f.restype = res
            f.argtypes = args
        _lib = handle
    return _lib


def _check(fn, st):
    if st != RL_OK:
        msg = lib().rl_last_error_message()
        raise RLError(fn, st, msg.decode() if msg else "")


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _need(t, name, dtype, numel=None, device=None):
    if t is None:
        raise ValueError(f"{name} is required")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() < numel:
        raise ValueError(f"{name} has {t.numel()} elements, needs {numel}")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")
    return t


def _opt(t, name, dtype, numel=None, device=None):
    return None if t is None else _need(t, name, dtype, numel, device)


def _logits_dtype(t):
    if t.dtype == torch.bfloat16:
        return RL_BF16
    if t.dtype == torch.float32:
        return RL_F32
    raise ValueError(f"logits must be bfloat16 or float32, got {t.dtype}")


def _rows_view(logits):
    if logits.dim() != 2 or logits.stride(1) != 1:
        raise ValueError("logits must be a 2-D tensor with unit stride along the vocabulary")
    return logits.shape[0], logits.shape[1], logits.stride(0)


# ----------------------------------------------------------------------------- ABI functions

def rl_version() -> int:
    return int(lib().rl_version())


def rl_last_error_message() -> str:
    m = lib().rl_last_error_message()
    return m.decode() if m else ""


def rl_workspace_size(max_rows: int, V: int, D: int = 0) -> int:
    return int(lib().rl_workspace_size(max_rows, V, D))


def rl_fused_head_workspace_size(T: int, V: int, D: int, group_tokens: int) -> int:
    return int(lib().rl_fused_head_workspace_size(T, V, D, group_tokens))


def rl_workspace_init(ws: torch.Tensor, stream=None):
    _need(ws, "ws", torch.uint8)
    _check("rl_workspace_init", lib().rl_workspace_init(_ptr(ws), ws.numel(), _stream(stream)))


def rl_selftest_bounded_wait(ws: torch.Tensor, limit_ns: int, waited_ns: torch.Tensor | None = None, stream=None):
    """Run one bounded wait that runs out (the failure path of every kernel wait); afterwards
    rl_query_status reports RL_ERR_TIMEOUT. waited_ns: optional int64 [1] on the device."""
    _need(ws, "ws", torch.uint8)
    _opt(waited_ns, "waited_ns", torch.int64, 1, device=ws.device)
    _check("rl_selftest_bounded_wait",
           lib().rl_selftest_bounded_wait(_ptr(ws), ws.numel(), int(limit_ns), _ptr(waited_ns), _stream(stream)))


def new_workspace(max_rows: int, V: int, D: int = 0, device=None, stream=None, group_tokens: int = 0) -> torch.Tensor:
    """Allocate (with torch) and initialise a workspace for calls of up to max_rows rows
    (with group_tokens > 0: the fused head's grouped workspace, rl_fused_head_workspace_size)."""
    nbytes = rl_fused_head_workspace_size(max_rows, V, D, group_tokens) if group_tokens > 0 and D > 0 \
        else rl_workspace_size(max_rows, V, D)
    ws = torch.empty(nbytes, dtype=torch.uint8, device=device or "cuda")
    rl_workspace_init(ws, stream)
    return ws


def rl_query_status(ws: torch.Tensor, stream=None):
    """Synchronise the stream and return (status, device_status_word)."""
    word = ctypes.c_int32(0)
    st = lib().rl_query_status(_ptr(ws), _stream(stream), ctypes.byref(word))
    if st not in (RL_OK, 6, 7):
        _check("rl_query_status", st)
    return st, int(word.value)


def rl_group_advantages(group_offsets, rewards, traj_offsets, mask, params: rl_loss_params, ws,
                        traj_valid=None, adv_out=None, coef_out=None, n_tok_out=None, token_traj_out=None,
                        want_token_traj=True, stream=None):
    """Advantages A_i, coefficients c_i, counts L_i (and token owners) for a packed batch."""
    dev = rewards.device
    n_traj = rewards.numel()
    n_groups = group_offsets.numel() - 1
    n_tokens = mask.numel()
    _need(rewards, "rewards", torch.float32, device=dev)
    _need(group_offsets, "group_offsets", torch.int32, device=dev)
    _need(traj_offsets, "traj_offsets", torch.int64, n_traj + 1, device=dev)
    _need(mask, "mask", torch.uint8, device=dev)
    _opt(traj_valid, "traj_valid", torch.uint8, n_traj, device=dev)
    adv_out = torch.empty(n_traj, dtype=torch.float32, device=dev) if adv_out is None else adv_out
    coef_out = torch.empty(n_traj, dtype=torch.float32, device=dev) if coef_out is None else coef_out
    n_tok_out = torch.empty(n_traj, dtype=torch.int32, device=dev) if n_tok_out is None else n_tok_out
    if want_token_traj and token_traj_out is None:
        token_traj_out = torch.empty(n_tokens, dtype=torch.int32, device=dev)
    _need(adv_out, "adv_out", torch.float32, n_traj, device=dev)
    _need(coef_out, "coef_out", torch.float32, n_traj, device=dev)
    _need(n_tok_out, "n_tok_out", torch.int32, n_traj, device=dev)
    _opt(token_traj_out, "token_traj_out", torch.int32, n_tokens, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_group_advantages(n_traj, n_groups, _ptr(group_offsets), _ptr(rewards), _ptr(traj_valid),
                                   n_tokens, _ptr(traj_offsets), _ptr(mask), ctypes.byref(params), _ptr(adv_out),
                                   _ptr(coef_out), _ptr(n_tok_out), _ptr(token_traj_out), _ptr(ws), ws.numel(),
                                   _stream(stream))
    _check("rl_group_advantages", st)
    return adv_out, coef_out, n_tok_out, token_traj_out


def rl_token_logprobs(logits, token_ids, ws, logp_out=None, entropy_out=None, lse_out=None,
                      want_entropy=False, want_lse=False, stream=None):
    """logp of the sampled ids (and optionally entropy, lse) for every logits row."""
    rows, V, ld = _rows_view(logits)
    dt = _logits_dtype(logits)
    dev = logits.device
    _need(token_ids, "token_ids", torch.int32, rows, device=dev)
    logp_out = torch.empty(rows, dtype=torch.float32, device=dev) if logp_out is None else logp_out
    if want_entropy and entropy_out is None:
        entropy_out = torch.empty(rows, dtype=torch.float32, device=dev)
    if want_lse and lse_out is None:
        lse_out = torch.empty(rows, dtype=torch.float32, device=dev)
    _need(logp_out, "logp_out", torch.float32, rows, device=dev)
    _opt(entropy_out, "entropy_out", torch.float32, rows, device=dev)
    _opt(lse_out, "lse_out", torch.float32, rows, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_token_logprobs(_ptr(logits), dt, rows, V, ld, _ptr(token_ids), _ptr(logp_out), _ptr(entropy_out),
                                 _ptr(lse_out), _ptr(ws), ws.numel(), _stream(stream))
    _check("rl_token_logprobs", st)
    return logp_out, entropy_out, lse_out


def rl_policy_loss_fwd_bwd(logits, token_ids, mask, token_traj, adv, coef, old_logp, params: rl_loss_params, ws,
                           loss_accum, grad_out=None, ref_logp=None, rollout_logp=None, token_stats=None,
                           stream=None):
    """Adds the microbatch loss to ``loss_accum`` (float64 [1]) and writes d loss / d logits.

    ``grad_out`` defaults to a new tensor shaped like ``logits``; pass ``logits`` itself
    for an in-place gradient. Returns grad_out.
    """
    rows, V, ld = _rows_view(logits)
    dt = _logits_dtype(logits)
    dev = logits.device
    n_traj = coef.numel()
    _need(token_ids, "token_ids", torch.int32, rows, device=dev)
    _need(mask, "mask", torch.uint8, rows, device=dev)
    _need(token_traj, "token_traj", torch.int32, rows, device=dev)
    _need(coef, "coef", torch.float32, n_traj, device=dev)
    _need(adv, "adv", torch.float32, rows if params.token_level_adv else n_traj, device=dev)
    _need(old_logp, "old_logp", torch.float32, rows, device=dev)
    _opt(ref_logp, "ref_logp", torch.float32, rows, device=dev)
    _opt(rollout_logp, "rollout_logp", torch.float32, rows, device=dev)
    _need(loss_accum, "loss_accum", torch.float64, 1, device=dev)
    _opt(token_stats, "token_stats", torch.float32, rows * 5, device=dev)
    if grad_out is None:
        grad_out = torch.empty_strided(logits.shape, logits.stride(), dtype=logits.dtype, device=dev)
    if grad_out.dtype != logits.dtype or grad_out.shape != logits.shape or grad_out.stride() != logits.stride():
        raise ValueError("grad_out must match logits in dtype, shape and strides")
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_policy_loss_fwd_bwd(_ptr(logits), dt, rows, V, ld, _ptr(token_ids), _ptr(mask), _ptr(token_traj),
                                      n_traj, _ptr(adv), _ptr(coef), _ptr(old_logp), _ptr(ref_logp),
                                      _ptr(rollout_logp), ctypes.byref(params), _ptr(grad_out), _ptr(loss_accum),
                                      _ptr(token_stats), _ptr(ws), ws.numel(), _stream(stream))
    _check("rl_policy_loss_fwd_bwd", st)
    return grad_out


def rl_policy_loss_fwd_bwd_noalloc(logits, token_ids, mask, token_traj, adv, coef, old_logp,
                                   params: rl_loss_params, loss_accum, grad_out, ref_logp=None, rollout_logp=None,
                                   token_stats=None, device_status=None, stream=None):
    """rl_policy_loss_fwd_bwd without a caller workspace, for callers that cannot allocate.

    ``grad_out`` must be provided (this form allocates nothing, not even through torch).
    ``device_status`` (int32 [1] on the device, optional) receives the call's status word.
    """
    rows, V, ld = _rows_view(logits)
    dt = _logits_dtype(logits)
    dev = logits.device
    n_traj = coef.numel()
    _need(token_ids, "token_ids", torch.int32, rows, device=dev)
    _need(mask, "mask", torch.uint8, rows, device=dev)
    _need(token_traj, "token_traj", torch.int32, rows, device=dev)
    _need(coef, "coef", torch.float32, n_traj, device=dev)
    _need(adv, "adv", torch.float32, rows if params.token_level_adv else n_traj, device=dev)
    _need(old_logp, "old_logp", torch.float32, rows, device=dev)
    _opt(ref_logp, "ref_logp", torch.float32, rows, device=dev)
    _opt(rollout_logp, "rollout_logp", torch.float32, rows, device=dev)
    _need(loss_accum, "loss_accum", torch.float64, 1, device=dev)
    _opt(token_stats, "token_stats", torch.float32, rows * 5, device=dev)
    _opt(device_status, "device_status", torch.int32, 1, device=dev)
    if grad_out is None or grad_out.dtype != logits.dtype or grad_out.shape != logits.shape or \
            grad_out.stride() != logits.stride():
        raise ValueError("grad_out must be given and match logits in dtype, shape and strides")
    st = lib().rl_policy_loss_fwd_bwd_noalloc(_ptr(logits), dt, rows, V, ld, _ptr(token_ids), _ptr(mask),
                                              _ptr(token_traj), n_traj, _ptr(adv), _ptr(coef), _ptr(old_logp),
                                              _ptr(ref_logp), _ptr(rollout_logp), ctypes.byref(params),
                                              _ptr(grad_out), _ptr(loss_accum), _ptr(token_stats),
                                              _ptr(device_status), _stream(stream))
    _check("rl_policy_loss_fwd_bwd_noalloc", st)
    return grad_out


def rl_fused_head_loss_fwd_bwd(hidden, weight, token_ids, mask, token_traj, adv, coef, old_logp,
                               params: rl_loss_params, ws, loss_accum, d_weight, d_hidden=None,
                               d_hidden_dtype=torch.bfloat16, ref_logp=None, rollout_logp=None, token_stats=None,
                               stream=None):
    """Loss of the LM head hidden @ weight^T without materialising the logits; returns d_hidden
    (overwritten) and adds d loss / d weight into ``d_weight`` (float32 [V, D])."""
    if hidden.dim() != 2 or weight.dim() != 2 or hidden.shape[1] != weight.shape[1]:
        raise ValueError("hidden [T, D] and weight [V, D] must share D")
    T, D = hidden.shape
    V = weight.shape[0]
    dev = hidden.device
    n_traj = coef.numel()
    _need(hidden, "hidden", torch.bfloat16, device=dev)
    _need(weight, "weight", torch.bfloat16, device=dev)
    _need(token_ids, "token_ids", torch.int32, T, device=dev)
    _need(mask, "mask", torch.uint8, T, device=dev)
    _need(token_traj, "token_traj", torch.int32, T, device=dev)
    _need(coef, "coef", torch.float32, n_traj, device=dev)
    _need(adv, "adv", torch.float32, T if params.token_level_adv else n_traj, device=dev)
    _need(old_logp, "old_logp", torch.float32, T, device=dev)
    _opt(ref_logp, "ref_logp", torch.float32, T, device=dev)
    _opt(rollout_logp, "rollout_logp", torch.float32, T, device=dev)
    _need(loss_accum, "loss_accum", torch.float64, 1, device=dev)
    _opt(token_stats, "token_stats", torch.float32, T * 5, device=dev)
    _need(d_weight, "d_weight", torch.float32, V * D, device=dev)
    if d_hidden is None:
        d_hidden = torch.empty((T, D), dtype=d_hidden_dtype, device=dev)
    _need(d_hidden, "d_hidden", d_hidden.dtype, T * D, device=dev)
    dt = _logits_dtype(d_hidden)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_fused_head_loss_fwd_bwd(_ptr(hidden), _ptr(weight), T, D, V, _ptr(token_ids), _ptr(mask),
                                          _ptr(token_traj), n_traj, _ptr(adv), _ptr(coef), _ptr(old_logp),
                                          _ptr(ref_logp), _ptr(rollout_logp), ctypes.byref(params), _ptr(d_hidden),
                                          dt, _ptr(d_weight), _ptr(loss_accum), _ptr(token_stats), _ptr(ws),
                                          ws.numel(), _stream(stream))
    _check("rl_fused_head_loss_fwd_bwd", st)
    return d_hidden


def rl_fused_head_token_logprobs(hidden, weight, token_ids, ws, logp_out=None, entropy_out=None, lse_out=None,
                                 want_entropy=False, want_lse=False, stream=None):
    """logp of the sampled ids (and optionally entropy, lse) under logits hidden @ weight^T,
    without materialising the logits."""
    if hidden.dim() != 2 or weight.dim() != 2 or hidden.shape[1] != weight.shape[1]:
        raise ValueError("hidden [T, D] and weight [V, D] must share D")
    T, D = hidden.shape
    V = weight.shape[0]
    dev = hidden.device
    _need(hidden, "hidden", torch.bfloat16, device=dev)
    _need(weight, "weight", torch.bfloat16, device=dev)
    _need(token_ids, "token_ids", torch.int32, T, device=dev)
    logp_out = torch.empty(T, dtype=torch.float32, device=dev) if logp_out is None else logp_out
    if want_entropy and entropy_out is None:
        entropy_out = torch.empty(T, dtype=torch.float32, device=dev)
    if want_lse and lse_out is None:
        lse_out = torch.empty(T, dtype=torch.float32, device=dev)
    _need(logp_out, "logp_out", torch.float32, T, device=dev)
    _opt(entropy_out, "entropy_out", torch.float32, T, device=dev)
    _opt(lse_out, "lse_out", torch.float32, T, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_fused_head_token_logprobs(_ptr(hidden), _ptr(weight), T, D, V, _ptr(token_ids), _ptr(logp_out),
                                            _ptr(entropy_out), _ptr(lse_out), _ptr(ws), ws.numel(), _stream(stream))
    _check("rl_fused_head_token_logprobs", st)
    return logp_out, entropy_out, lse_out


def rl_masked_gae(traj_offsets, mask, values, ws, gamma=1.0, gae_lambda=1.0, skip_masked=True, token_rewards=None,
                  traj_rewards=None, adv_out=None, returns_out=None, want_returns=True, stream=None):
    """Masked GAE per trajectory (Sec. 2.3.1): returns (adv, returns) float32 [T], zero at masked tokens.
    traj_rewards [n] places R_i at trajectory i's last trainable token (Sec. 2.3.4)."""
    n_traj = traj_offsets.numel() - 1
    T = mask.numel()
    dev = mask.device
    _need(traj_offsets, "traj_offsets", torch.int64, n_traj + 1, device=dev)
    _need(mask, "mask", torch.uint8, T, device=dev)
    _need(values, "values", torch.float32, T, device=dev)
    _opt(token_rewards, "token_rewards", torch.float32, T, device=dev)
    _opt(traj_rewards, "traj_rewards", torch.float32, n_traj, device=dev)
    adv_out = torch.empty(T, dtype=torch.float32, device=dev) if adv_out is None else adv_out
    if want_returns and returns_out is None:
        returns_out = torch.empty(T, dtype=torch.float32, device=dev)
    _need(adv_out, "adv_out", torch.float32, T, device=dev)
    _opt(returns_out, "returns_out", torch.float32, T, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_masked_gae(n_traj, _ptr(traj_offsets), T, _ptr(mask), _ptr(values), _ptr(token_rewards),
                             _ptr(traj_rewards), float(gamma), float(gae_lambda), 1 if skip_masked else 0,
                             _ptr(adv_out), _ptr(returns_out), _ptr(ws), ws.numel(), _stream(stream))
    _check("rl_masked_gae", st)
    return adv_out, returns_out


def rl_value_loss_fwd_bwd(values, returns, mask, token_traj, coef, ws, loss_accum, d_values=None, stream=None):
    """Adds sum_t c M (V - G)^2 to ``loss_accum`` (float64 [1]); returns d loss / d values (float32)."""
    rows = values.numel()
    dev = values.device
    n_traj = coef.numel()
    _need(values, "values", torch.float32, rows, device=dev)
    _need(returns, "returns", torch.float32, rows, device=dev)
    _need(mask, "mask", torch.uint8, rows, device=dev)
    _need(token_traj, "token_traj", torch.int32, rows, device=dev)
    _need(coef, "coef", torch.float32, n_traj, device=dev)
    _need(loss_accum, "loss_accum", torch.float64, 1, device=dev)
    d_values = torch.empty(rows, dtype=torch.float32, device=dev) if d_values is None else d_values
    _need(d_values, "d_values", torch.float32, rows, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_value_loss_fwd_bwd(rows, _ptr(values), _ptr(returns), _ptr(mask), _ptr(token_traj), n_traj,
                                     _ptr(coef), _ptr(d_values), _ptr(loss_accum), _ptr(ws), ws.numel(),
                                     _stream(stream))
    _check("rl_value_loss_fwd_bwd", st)
    return d_values


def rl_sequence_is_weights(token_traj, mask, old_logp, rollout_logp, n_traj, ws, cap=0.0, weight_out=None,
                           log_ratio_out=None, want_log_ratio=False, traj_adv_inout=None, token_adv_inout=None,
                           stream=None):
    """Sequence-level importance weights w_i = min(exp(sum_t M (old - rollout)), cap) over the
    tokens each unit owns (Sec. 3.2.4); optionally scales advantages in place. Returns
    (weight, log_ratio)."""
    T = mask.numel()
    dev = mask.device
    _need(token_traj, "token_traj", torch.int32, T, device=dev)
    _need(mask, "mask", torch.uint8, T, device=dev)
    _need(old_logp, "old_logp", torch.float32, T, device=dev)
    _need(rollout_logp, "rollout_logp", torch.float32, T, device=dev)
    weight_out = torch.empty(n_traj, dtype=torch.float32, device=dev) if weight_out is None else weight_out
    if want_log_ratio and log_ratio_out is None:
        log_ratio_out = torch.empty(n_traj, dtype=torch.float32, device=dev)
    _need(weight_out, "weight_out", torch.float32, n_traj, device=dev)
    _opt(log_ratio_out, "log_ratio_out", torch.float32, n_traj, device=dev)
    _opt(traj_adv_inout, "traj_adv_inout", torch.float32, n_traj, device=dev)
    _opt(token_adv_inout, "token_adv_inout", torch.float32, T, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_sequence_is_weights(n_traj, T, _ptr(token_traj), _ptr(mask), _ptr(old_logp), _ptr(rollout_logp),
                                      float(cap), _ptr(weight_out), _ptr(log_ratio_out), _ptr(traj_adv_inout),
                                      _ptr(token_adv_inout), _ptr(ws), ws.numel(), _stream(stream))
    _check("rl_sequence_is_weights", st)
    return weight_out, log_ratio_out


def _np_ptr(a):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _csr(seqs, dtype, off_dtype=np.int64):
    lens = np.fromiter((len(q) for q in seqs), dtype=np.int64, count=len(seqs))
    offs = np.zeros(len(seqs) + 1, dtype=off_dtype)
    np.cumsum(lens, out=offs[1:])
    flat = np.concatenate([np.asarray(q, dtype=dtype) for q in seqs]) if len(seqs) and offs[-1] else \
        np.zeros(1, dtype=dtype)
    return offs, np.ascontiguousarray(flat)


def rl_prefix_tree_build_batch(prompts, calls, aux=None, max_leaves=0, n_threads=None):
    """Prefix trees of a batch of rollouts, packed (host arrays in, numpy arrays out).

    prompts: one token sequence per rollout; calls: per rollout, a list of (x, y) token
    sequences in capture order; aux: per rollout, a list of flags (or None). Returns a dict of
    the packed per-token arrays (tokens, mask, parent, depth, owner, node_call), the kept
    leaves (leaf_call, leaf_end, leaf_offsets), rollout_offsets and per-rollout stats."""
    n = len(prompts)
    if len(calls) != n:
        raise ValueError("one list of calls per rollout")
    p_off, p_tok = _csr(prompts, np.int32)
    c_off = np.zeros(n + 1, dtype=np.int32)
    np.cumsum([len(c) for c in calls], out=c_off[1:])
    flat = [c for rc in calls for c in rc]
    x_off, x_tok = _csr([c[0] for c in flat], np.int32)
    y_off, y_tok = _csr([c[1] for c in flat], np.int32)
    aux_arr = None
    if aux is not None:
        aux_arr = np.concatenate([np.asarray(a if a is not None else [0] * len(rc), dtype=np.uint8)
                                  for a, rc in zip(aux, calls)]) if flat else np.zeros(1, np.uint8)
    n_calls = len(flat)
    threads = n_threads if n_threads is not None else min(16, os.cpu_count() or 1)
    stats = (rl_tree_stats * max(n, 1))()
    r_off = np.zeros(n + 1, dtype=np.int64)
    l_off = np.zeros(n + 1, dtype=np.int64)
    n_tok = ctypes.c_int64(0)
    L = lib()
    args = (n, _np_ptr(p_off), _np_ptr(p_tok), _np_ptr(c_off), _np_ptr(x_off), _np_ptr(x_tok), _np_ptr(y_off),
            _np_ptr(y_tok), _np_ptr(aux_arr), int(max_leaves), int(threads))
    st = L.rl_prefix_tree_build_batch(*args, 0, None, None, None, None, None, None, None, None, None, stats,
                                      _np_ptr(r_off), ctypes.byref(n_tok))
    if st not in (RL_OK, 4):
        _check("rl_prefix_tree_build_batch", st)
    T = n_tok.value
    out = dict(tokens=np.empty(T, np.int32), mask=np.empty(T, np.uint8), parent=np.empty(T, np.int64),
               depth=np.empty(T, np.int32), owner=np.empty(T, np.int32), node_call=np.empty(T, np.int32),
               leaf_call=np.empty(max(n_calls, 1), np.int32), leaf_end=np.empty(max(n_calls, 1), np.int64))
    st = L.rl_prefix_tree_build_batch(*args, T, *(_np_ptr(out[k]) for k in ("tokens", "mask", "parent", "depth",
                                                                              "owner", "node_call", "leaf_call",
                                                                              "leaf_end")),
                                      _np_ptr(l_off), stats, _np_ptr(r_off), ctypes.byref(n_tok))
    _check("rl_prefix_tree_build_batch", st)
    out["leaf_call"] = out["leaf_call"][:l_off[-1]]
    out["leaf_end"] = out["leaf_end"][:l_off[-1]]
    out.update(leaf_offsets=l_off, rollout_offsets=r_off,
               stats=[dict(valid=stats[r].valid, n_leaves=stats[r].n_leaves, n_kept_leaves=stats[r].n_kept_leaves,
                           n_unplaced=stats[r].n_unplaced, n_tokens=stats[r].n_tokens,
                           n_trainable=stats[r].n_trainable) for r in range(n)])
    return out


def rl_group_advantages_by_owner(group_offsets, rewards, token_traj, mask, params: rl_loss_params, ws,
                                 traj_valid=None, adv_out=None, coef_out=None, n_tok_out=None, stream=None):
    """rl_group_advantages with the owner of every token given (any token order)."""
    n_traj = rewards.numel()
    n_groups = group_offsets.numel() - 1
    T = mask.numel()
    dev = rewards.device
    _need(group_offsets, "group_offsets", torch.int32, n_groups + 1, device=dev)
    _need(rewards, "rewards", torch.float32, n_traj, device=dev)
    _opt(traj_valid, "traj_valid", torch.uint8, n_traj, device=dev)
    _need(token_traj, "token_traj", torch.int32, T, device=dev)
    _need(mask, "mask", torch.uint8, T, device=dev)
    adv_out = torch.empty(n_traj, dtype=torch.float32, device=dev) if adv_out is None else adv_out
    coef_out = torch.empty(n_traj, dtype=torch.float32, device=dev) if coef_out is None else coef_out
    n_tok_out = torch.empty(n_traj, dtype=torch.int32, device=dev) if n_tok_out is None else n_tok_out
    _need(adv_out, "adv_out", torch.float32, n_traj, device=dev)
    _need(coef_out, "coef_out", torch.float32, n_traj, device=dev)
    _need(n_tok_out, "n_tok_out", torch.int32, n_traj, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_group_advantages_by_owner(n_traj, n_groups, _ptr(group_offsets), _ptr(rewards), _ptr(traj_valid), T,
                                            _ptr(token_traj), _ptr(mask), ctypes.byref(params), _ptr(adv_out),
                                            _ptr(coef_out), _ptr(n_tok_out), _ptr(ws), ws.numel(), _stream(stream))
    _check("rl_group_advantages_by_owner", st)
    return adv_out, coef_out, n_tok_out


def rl_rollout_value_advantages(token_traj, mask, values, rewards, ws, adv_out=None, returns_out=None,
                                want_returns=True, stream=None):
    """A_t = R_i - V_t, G_t = R_i on trainable tokens (Sec. 2.3.4), tokens in any order."""
    T = mask.numel()
    n_traj = rewards.numel()
    dev = mask.device
    _need(token_traj, "token_traj", torch.int32, T, device=dev)
    _need(mask, "mask", torch.uint8, T, device=dev)
    _need(values, "values", torch.float32, T, device=dev)
    _need(rewards, "rewards", torch.float32, n_traj, device=dev)
    adv_out = torch.empty(T, dtype=torch.float32, device=dev) if adv_out is None else adv_out
    if want_returns and returns_out is None:
        returns_out = torch.empty(T, dtype=torch.float32, device=dev)
    _need(adv_out, "adv_out", torch.float32, T, device=dev)
    _opt(returns_out, "returns_out", torch.float32, T, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_rollout_value_advantages(T, _ptr(token_traj), _ptr(mask), _ptr(values), _ptr(rewards), n_traj,
                                           _ptr(adv_out), _ptr(returns_out), _ptr(ws), ws.numel(), _stream(stream))
    _check("rl_rollout_value_advantages", st)
    return adv_out, returns_out


def rl_token_stats_summary(token_stats, mask, token_traj, coef, ws, summary_accum=None, stream=None):
    """Adds (trained tokens, clipped, sum H, sum KL, sum rho) over the trained tokens to
    ``summary_accum`` (float64 [5], created if None) and returns it."""
    rows = mask.numel()
    n_traj = coef.numel()
    dev = mask.device
    _need(token_stats, "token_stats", torch.float32, rows * 5, device=dev)
    _need(mask, "mask", torch.uint8, rows, device=dev)
    _need(token_traj, "token_traj", torch.int32, rows, device=dev)
    _need(coef, "coef", torch.float32, n_traj, device=dev)
    if summary_accum is None:
        summary_accum = torch.zeros(5, dtype=torch.float64, device=dev)
    _need(summary_accum, "summary_accum", torch.float64, 5, device=dev)
    _need(ws, "ws", torch.uint8, device=dev)
    st = lib().rl_token_stats_summary(rows, _ptr(token_stats), _ptr(mask), _ptr(token_traj), n_traj, _ptr(coef),
                                      _ptr(summary_accum), _ptr(ws), ws.numel(), _stream(stream))
    _check("rl_token_stats_summary", st)
    return summary_accum
