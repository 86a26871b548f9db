"""Thin Python binding of libsao (include/sao.h), argument marshalling only.

Every function here has the name of the C entry point it calls, takes torch
tensors that already live on the current CUDA device, checks their dtypes and
shapes, and passes raw device pointers and the current CUDA stream to the
library. All arithmetic happens in libsao's CUDA kernels; if the library is
missing the import of this module's functions raises, there is no fallback.
"""
from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libsao.so")

SAO_F32, SAO_BF16 = 0, 1
SAO_STEP_AVERAGE, SAO_STEP_LAST = 0, 1
SAO_NORM_TOKEN, SAO_NORM_SEQUENCE = 0, 1
STATUS = {0: "SAO_OK", 1: "SAO_ERR_INVALID_ARG", 2: "SAO_ERR_SHAPE", 3: "SAO_ERR_WORKSPACE",
          4: "SAO_ERR_UNSUPPORTED", 5: "SAO_ERR_CUDA", 6: "SAO_ERR_DEVICE_CHECK"}
FLAG_IN, FLAG_LOW, FLAG_HIGH, FLAG_NONFINITE, FLAG_NOT_ACTION = 0, 1, 2, 3, 4
FLAG_MISMATCH_LOW, FLAG_MISMATCH_HIGH = 5, 6

EXPORTS = ("sao_version", "sao_last_error_string", "sao_set_checked", "sao_get_checked",
           "sao_set_dz_budget_bytes", "sao_get_dz_budget_bytes", "sao_set_cta_pairs", "sao_get_cta_pairs",
           "sao_debug_set_scan_hooks", "sao_workspace_bytes", "sao_token_logprobs_fwd",
           "sao_token_logprobs_bwd", "sao_advantages", "sao_advantages_noalloc", "sao_step_advantages",
           "sao_policy_loss_fwd", "sao_policy_loss_bwd", "sao_clip_loss_fwd", "sao_clip_loss_bwd",
           "sao_group_advantages", "sao_running_mean_advantages", "sao_decoupled_loss_fwd",
           "sao_decoupled_loss_bwd", "sao_logprob_cache_bytes", "sao_token_logprobs_fwd_cached",
           "sao_token_logprobs_bwd_cached",
           "sao_value_loss", "sao_profile_enable", "sao_profile_reset", "sao_profile_read")


class SaoError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


_lib = None


def load(path: Optional[str] = None):
    """Load libsao.so (building it first if absent) and declare its signatures."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        from . import build as _build
        _build.build()
    L = ctypes.CDLL(path)
    P, I64, I32, F, SZ = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float, ctypes.c_size_t
    sig = {
        "sao_version": (ctypes.c_int, []),
        "sao_last_error_string": (ctypes.c_char_p, []),
        "sao_set_checked": (None, [ctypes.c_int]),
        "sao_get_checked": (ctypes.c_int, []),
        "sao_set_dz_budget_bytes": (None, [SZ]),
        "sao_get_dz_budget_bytes": (SZ, []),
        "sao_set_cta_pairs": (None, [ctypes.c_int]),
        "sao_get_cta_pairs": (ctypes.c_int, []),
        "sao_debug_set_scan_hooks": (None, [ctypes.c_uint64, I32]),
        "sao_workspace_bytes": (SZ, [I64, I32, I32, ctypes.c_int]),
        "sao_logprob_cache_bytes": (SZ, [I64, I32]),
        "sao_token_logprobs_fwd_cached": (ctypes.c_int, [P, P, ctypes.c_int, P, P, I64, I32, I32, P, P, P, SZ, P,
                                                         SZ, P]),
        "sao_token_logprobs_bwd_cached": (ctypes.c_int, [P, P, ctypes.c_int, P, P, P, I64, I32, I32, P, P,
                                                         ctypes.c_int, P, SZ, P, SZ, P]),
        "sao_token_logprobs_fwd": (ctypes.c_int, [P, P, ctypes.c_int, P, P, I64, I32, I32, P, P, P, SZ, P]),
        "sao_token_logprobs_bwd": (ctypes.c_int, [P, P, ctypes.c_int, P, P, P, I64, I32, I32, P, P,
                                                  ctypes.c_int, P, SZ, P]),
        "sao_advantages": (ctypes.c_int, [P, P, P, P, I32, I64, F, F, F, F, P, P, P, SZ, P]),
        "sao_advantages_noalloc": (ctypes.c_int, [P, P, P, P, I32, I64, F, F, F, F, P, P, P]),
        "sao_step_advantages": (ctypes.c_int, [P, P, P, P, I32, I64, F, F, F, F, ctypes.c_int, P, P, P, P, SZ, P]),
        "sao_policy_loss_fwd": (ctypes.c_int, [P, P, P, P, I64, F, F, I64, P, P, P, P, P, SZ, P]),
        "sao_policy_loss_bwd": (ctypes.c_int, [P, P, P, P, I64, F, F, I64, P, P, P, SZ, P]),
        "sao_decoupled_loss_fwd": (ctypes.c_int, [P, P, P, P, P, I64, F, F, F, F, I64, P, P, P, P, P, SZ, P]),
        "sao_decoupled_loss_bwd": (ctypes.c_int, [P, P, P, P, P, I64, F, F, F, F, I64, P, P, P, SZ, P]),
        "sao_value_loss": (ctypes.c_int, [P, P, P, I64, I64, P, P, P, P, SZ, P]),
        "sao_clip_loss_fwd": (ctypes.c_int, [P, P, P, P, P, I32, I64, F, F, ctypes.c_int, P, P, P, P, P, SZ, P]),
        "sao_clip_loss_bwd": (ctypes.c_int, [P, P, P, P, P, I32, I64, F, F, ctypes.c_int, P, P, P, SZ, P]),
        "sao_group_advantages": (ctypes.c_int, [P, P, I32, P, P, I64, F, P, P, SZ, P]),
        "sao_running_mean_advantages": (ctypes.c_int, [P, P, I32, I32, P, P, I32, P, P, I64, P, P, SZ, P]),
        "sao_profile_enable": (None, [ctypes.c_int]),
        "sao_profile_reset": (None, []),
        "sao_profile_read": (ctypes.c_int, [P, P, P, ctypes.c_int]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def _check(status: int):
    if status != 0:
        raise SaoError(status, load().sao_last_error_string().decode())


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("libsao takes CUDA tensors")
    if not t.is_contiguous():
        raise ValueError("libsao takes contiguous tensors")
    return ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    if stream is None:
        stream = torch.cuda.current_stream()
    return ctypes.c_void_p(stream.cuda_stream)


def _dtype_code(t: torch.Tensor) -> int:
    if t.dtype == torch.bfloat16:
        return SAO_BF16
    if t.dtype == torch.float32:
        return SAO_F32
    raise ValueError(f"H and W must be bf16 or fp32, got {t.dtype}")


def _expect(t, dtype, n, name):
    if t is None:
        return
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if t.numel() != n:
        raise ValueError(f"{name} must have {n} elements, got {t.numel()}")


# ---------------------------------------------------------------------------
# process settings
# ---------------------------------------------------------------------------

def sao_version() -> int:
    return load().sao_version()


def sao_set_checked(on: bool):
    load().sao_set_checked(1 if on else 0)


def sao_get_checked() -> bool:
    return bool(load().sao_get_checked())


def sao_set_dz_budget_bytes(nbytes: int):
    load().sao_set_dz_budget_bytes(int(nbytes))


def sao_get_dz_budget_bytes() -> int:
    return int(load().sao_get_dz_budget_bytes())


def sao_set_cta_pairs(on: bool):
    load().sao_set_cta_pairs(1 if on else 0)


def sao_get_cta_pairs() -> bool:
    return bool(load().sao_get_cta_pairs())


def sao_debug_set_scan_hooks(wait_ns: int = 0, skip_chunks: int = 0):
    """Test hooks of the advantage scan; (0, 0) restores the defaults."""
    load().sao_debug_set_scan_hooks(int(wait_ns), int(skip_chunks))


def sao_workspace_bytes(N: int, h: int = 0, V: int = 0, dtype=torch.bfloat16) -> int:
    code = SAO_BF16 if dtype == torch.bfloat16 else SAO_F32
    return int(load().sao_workspace_bytes(int(N), int(h), int(V), code))


def workspace(N: int, h: int = 0, V: int = 0, dtype=torch.bfloat16, device=None) -> torch.Tensor:
    """Allocate a workspace tensor (torch owns the memory; 256-byte aligned)."""
    n = sao_workspace_bytes(N, h, V, dtype)
    return torch.empty(max(n, 256), dtype=torch.uint8, device=device or "cuda")


# ---------------------------------------------------------------------------
# entry points
# ---------------------------------------------------------------------------

def sao_token_logprobs_fwd(H, W, y, logp, lse, ws, row_mask=None, stream=None):
    N, h = H.shape
    V = W.shape[0]
    if W.shape[1] != h or W.dtype != H.dtype:
        raise ValueError("W must be [V, h] with the dtype of H")
    _expect(y, torch.int32, N, "y")
    _expect(logp, torch.float32, N, "logp")
    _expect(lse, torch.float32, N, "lse")
    _expect(row_mask, torch.uint8, N, "row_mask")
    _check(load().sao_token_logprobs_fwd(_ptr(H), _ptr(W), _dtype_code(H), _ptr(y), _ptr(row_mask), N, h, V,
                                         _ptr(logp), _ptr(lse), _ptr(ws), ws.numel(), _stream(stream)))


def sao_token_logprobs_bwd(H, W, y, lse, grad_logp, dH, dW, ws, accumulate_dW=False, stream=None):
    N, h = H.shape
    V = W.shape[0]
    if W.shape[1] != h or W.dtype != H.dtype or dH.dtype != H.dtype or tuple(dH.shape) != (N, h):
        raise ValueError("W [V,h] and dH [N,h] must share the dtype of H")
    if dW.dtype != torch.float32 or tuple(dW.shape) != (V, h):
        raise ValueError("dW must be fp32 [V, h]")
    _expect(y, torch.int32, N, "y")
    _expect(lse, torch.float32, N, "lse")
    _expect(grad_logp, torch.float32, N, "grad_logp")
    _check(load().sao_token_logprobs_bwd(_ptr(H), _ptr(W), _dtype_code(H), _ptr(y), _ptr(lse), _ptr(grad_logp),
                                         N, h, V, _ptr(dH), _ptr(dW), 1 if accumulate_dW else 0, _ptr(ws),
                                         ws.numel(), _stream(stream)))


def sao_logprob_cache_bytes(N: int, V: int) -> int:
    return int(load().sao_logprob_cache_bytes(int(N), int(V)))


def logprob_cache(N: int, V: int, device=None) -> torch.Tensor:
    """Allocate the forward's probability cache (about 2*N*V bytes)."""
    return torch.empty(max(sao_logprob_cache_bytes(N, V), 256), dtype=torch.uint8, device=device or "cuda")


def sao_token_logprobs_fwd_cached(H, W, y, logp, lse, cache, ws, row_mask=None, stream=None):
    N, h = H.shape
    V = W.shape[0]
    if W.shape[1] != h or W.dtype != H.dtype:
        raise ValueError("W must be [V, h] with the dtype of H")
    _expect(y, torch.int32, N, "y")
    _expect(logp, torch.float32, N, "logp")
    _expect(lse, torch.float32, N, "lse")
    _expect(row_mask, torch.uint8, N, "row_mask")
    _check(load().sao_token_logprobs_fwd_cached(_ptr(H), _ptr(W), _dtype_code(H), _ptr(y), _ptr(row_mask), N, h, V,
                                                _ptr(logp), _ptr(lse), _ptr(cache), cache.numel(), _ptr(ws),
                                                ws.numel(), _stream(stream)))


def sao_token_logprobs_bwd_cached(H, W, y, lse, grad_logp, dH, dW, cache, ws, accumulate_dW=False, stream=None):
    N, h = H.shape
    V = W.shape[0]
    if W.shape[1] != h or W.dtype != H.dtype or dH.dtype != H.dtype or tuple(dH.shape) != (N, h):
        raise ValueError("W [V,h] and dH [N,h] must share the dtype of H")
    if dW.dtype != torch.float32 or tuple(dW.shape) != (V, h):
        raise ValueError("dW must be fp32 [V, h]")
    _expect(y, torch.int32, N, "y")
    _expect(lse, torch.float32, N, "lse")
    _expect(grad_logp, torch.float32, N, "grad_logp")
    _check(load().sao_token_logprobs_bwd_cached(_ptr(H), _ptr(W), _dtype_code(H), _ptr(y), _ptr(lse),
                                                _ptr(grad_logp), N, h, V, _ptr(dH), _ptr(dW),
                                                1 if accumulate_dW else 0, _ptr(cache), cache.numel(), _ptr(ws),
                                                ws.numel(), _stream(stream)))


def sao_advantages(values, rewards, loss_mask, cu_seqlens, gamma, lambda_policy, lambda_critic,
                   len_adaptive_alpha, adv, ret, ws, stream=None):
    N = values.numel()
    B = cu_seqlens.numel() - 1
    _expect(values, torch.float32, N, "values")
    _expect(rewards, torch.float32, B, "rewards")
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(cu_seqlens, torch.int32, B + 1, "cu_seqlens")
    _expect(adv, torch.float32, N, "adv")
    _expect(ret, torch.float32, N, "ret")
    _check(load().sao_advantages(_ptr(values), _ptr(rewards), _ptr(loss_mask), _ptr(cu_seqlens), B, N,
                                 float(gamma), float(lambda_policy), float(lambda_critic),
                                 float(len_adaptive_alpha), _ptr(adv), _ptr(ret), _ptr(ws), ws.numel(),
                                 _stream(stream)))


def sao_step_advantages(values, rewards, loss_mask, cu_seqlens, gamma, lambda_policy, lambda_critic,
                        len_adaptive_alpha, mode, adv, ret, ws, value_mask=None, stream=None):
    N = values.numel()
    B = cu_seqlens.numel() - 1
    _expect(values, torch.float32, N, "values")
    _expect(rewards, torch.float32, B, "rewards")
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(cu_seqlens, torch.int32, B + 1, "cu_seqlens")
    _expect(adv, torch.float32, N, "adv")
    _expect(ret, torch.float32, N, "ret")
    _expect(value_mask, torch.uint8, N, "value_mask")
    _check(load().sao_step_advantages(_ptr(values), _ptr(rewards), _ptr(loss_mask), _ptr(cu_seqlens), B, N,
                                      float(gamma), float(lambda_policy), float(lambda_critic),
                                      float(len_adaptive_alpha), int(mode), _ptr(adv), _ptr(ret), _ptr(value_mask),
                                      _ptr(ws), ws.numel(), _stream(stream)))


def sao_advantages_noalloc(values, rewards, loss_mask, cu_seqlens, gamma, lambda_policy, lambda_critic,
                           len_adaptive_alpha, adv, ret, stream=None):
    """sao_advantages with the library's fixed device scratch instead of a
    workspace, for callers that cannot allocate device memory."""
    N = values.numel()
    B = cu_seqlens.numel() - 1
    _expect(values, torch.float32, N, "values")
    _expect(rewards, torch.float32, B, "rewards")
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(cu_seqlens, torch.int32, B + 1, "cu_seqlens")
    _expect(adv, torch.float32, N, "adv")
    _expect(ret, torch.float32, N, "ret")
    _check(load().sao_advantages_noalloc(_ptr(values), _ptr(rewards), _ptr(loss_mask), _ptr(cu_seqlens), B, N,
                                         float(gamma), float(lambda_policy), float(lambda_critic),
                                         float(len_adaptive_alpha), _ptr(adv), _ptr(ret), _stream(stream)))


def sao_policy_loss_fwd(logp, old_logp, adv, loss_mask, eps_low, eps_high, loss, counts, ws, coef=None,
                        flags=None, n_norm=0, stream=None):
    N = logp.numel()
    for t, name in ((logp, "logp"), (old_logp, "old_logp"), (adv, "adv")):
        _expect(t, torch.float32, N, name)
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(coef, torch.float32, N, "coef")
    _expect(flags, torch.uint8, N, "flags")
    _expect(loss, torch.float32, 1, "loss")
    _expect(counts, torch.int64, 4, "counts")
    _check(load().sao_policy_loss_fwd(_ptr(logp), _ptr(old_logp), _ptr(adv), _ptr(loss_mask), N, float(eps_low),
                                      float(eps_high), int(n_norm), _ptr(loss), _ptr(coef), _ptr(flags),
                                      _ptr(counts), _ptr(ws), ws.numel(), _stream(stream)))


def sao_policy_loss_bwd(logp, old_logp, adv, loss_mask, eps_low, eps_high, grad_loss, grad_logp, ws, n_norm=0,
                        stream=None):
    N = logp.numel()
    for t, name in ((logp, "logp"), (old_logp, "old_logp"), (adv, "adv"), (grad_logp, "grad_logp")):
        _expect(t, torch.float32, N, name)
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(grad_loss, torch.float32, 1, "grad_loss")
    _check(load().sao_policy_loss_bwd(_ptr(logp), _ptr(old_logp), _ptr(adv), _ptr(loss_mask), N, float(eps_low),
                                      float(eps_high), int(n_norm), _ptr(grad_loss), _ptr(grad_logp), _ptr(ws),
                                      ws.numel(), _stream(stream)))


def sao_decoupled_loss_fwd(logp, prox_logp, rollout_logp, adv, loss_mask, eps_low, eps_high, w_low, w_high, loss,
                           counts, ws, coef=None, flags=None, n_norm=0, stream=None):
    N = logp.numel()
    for t, name in ((logp, "logp"), (prox_logp, "prox_logp"), (rollout_logp, "rollout_logp"), (adv, "adv")):
        _expect(t, torch.float32, N, name)
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(coef, torch.float32, N, "coef")
    _expect(flags, torch.uint8, N, "flags")
    _expect(loss, torch.float32, 1, "loss")
    _expect(counts, torch.int64, 6, "counts")
    _check(load().sao_decoupled_loss_fwd(_ptr(logp), _ptr(prox_logp), _ptr(rollout_logp), _ptr(adv),
                                         _ptr(loss_mask), N, float(eps_low), float(eps_high), float(w_low),
                                         float(w_high), int(n_norm), _ptr(loss), _ptr(coef), _ptr(flags),
                                         _ptr(counts), _ptr(ws), ws.numel(), _stream(stream)))


def sao_decoupled_loss_bwd(logp, prox_logp, rollout_logp, adv, loss_mask, eps_low, eps_high, w_low, w_high,
                           grad_loss, grad_logp, ws, n_norm=0, stream=None):
    N = logp.numel()
    for t, name in ((logp, "logp"), (prox_logp, "prox_logp"), (rollout_logp, "rollout_logp"), (adv, "adv"),
                    (grad_logp, "grad_logp")):
        _expect(t, torch.float32, N, name)
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(grad_loss, torch.float32, 1, "grad_loss")
    _check(load().sao_decoupled_loss_bwd(_ptr(logp), _ptr(prox_logp), _ptr(rollout_logp), _ptr(adv),
                                         _ptr(loss_mask), N, float(eps_low), float(eps_high), float(w_low),
                                         float(w_high), int(n_norm), _ptr(grad_loss), _ptr(grad_logp), _ptr(ws),
                                         ws.numel(), _stream(stream)))


def sao_value_loss(values, ret, loss_mask, loss, grad_values, ws, ev_sums=None, n_norm=0, stream=None):
    N = values.numel()
    _expect(values, torch.float32, N, "values")
    _expect(ret, torch.float32, N, "ret")
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(grad_values, torch.float32, N, "grad_values")
    _expect(loss, torch.float32, 1, "loss")
    _expect(ev_sums, torch.float64, 4, "ev_sums")
    _check(load().sao_value_loss(_ptr(values), _ptr(ret), _ptr(loss_mask), N, int(n_norm), _ptr(loss),
                                 _ptr(grad_values), _ptr(ev_sums), _ptr(ws), ws.numel(), _stream(stream)))


def sao_clip_loss_fwd(logp, old_logp, adv, loss_mask, cu_seqlens, eps_low, eps_high, norm, loss, counts, ws,
                      coef=None, flags=None, stream=None):
    N = logp.numel()
    B = cu_seqlens.numel() - 1
    for t, name in ((logp, "logp"), (old_logp, "old_logp"), (adv, "adv")):
        _expect(t, torch.float32, N, name)
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(cu_seqlens, torch.int32, B + 1, "cu_seqlens")
    _expect(coef, torch.float32, N, "coef")
    _expect(flags, torch.uint8, N, "flags")
    _expect(loss, torch.float32, 1, "loss")
    _expect(counts, torch.int64, 4, "counts")
    _check(load().sao_clip_loss_fwd(_ptr(logp), _ptr(old_logp), _ptr(adv), _ptr(loss_mask), _ptr(cu_seqlens), B, N,
                                    float(eps_low), float(eps_high), int(norm), _ptr(loss), _ptr(coef), _ptr(flags),
                                    _ptr(counts), _ptr(ws), ws.numel(), _stream(stream)))


def sao_clip_loss_bwd(logp, old_logp, adv, loss_mask, cu_seqlens, eps_low, eps_high, norm, grad_loss, grad_logp, ws,
                      stream=None):
    N = logp.numel()
    B = cu_seqlens.numel() - 1
    for t, name in ((logp, "logp"), (old_logp, "old_logp"), (adv, "adv"), (grad_logp, "grad_logp")):
        _expect(t, torch.float32, N, name)
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(cu_seqlens, torch.int32, B + 1, "cu_seqlens")
    _expect(grad_loss, torch.float32, 1, "grad_loss")
    _check(load().sao_clip_loss_bwd(_ptr(logp), _ptr(old_logp), _ptr(adv), _ptr(loss_mask), _ptr(cu_seqlens), B, N,
                                    float(eps_low), float(eps_high), int(norm), _ptr(grad_loss), _ptr(grad_logp),
                                    _ptr(ws), ws.numel(), _stream(stream)))


def sao_group_advantages(rewards, group_ids, loss_mask, cu_seqlens, eps_stab, adv, ws, stream=None):
    N = loss_mask.numel()
    B = cu_seqlens.numel() - 1
    _expect(rewards, torch.float32, B, "rewards")
    _expect(group_ids, torch.int32, B, "group_ids")
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(cu_seqlens, torch.int32, B + 1, "cu_seqlens")
    _expect(adv, torch.float32, N, "adv")
    _check(load().sao_group_advantages(_ptr(rewards), _ptr(group_ids), B, _ptr(loss_mask), _ptr(cu_seqlens), N,
                                       float(eps_stab), _ptr(adv), _ptr(ws), ws.numel(), _stream(stream)))


def sao_running_mean_advantages(rewards, prompt_ids, history, seen, loss_mask, cu_seqlens, adv, ws, stream=None):
    """history [P, window] fp32 and seen [P] int64 are updated in place."""
    N = loss_mask.numel()
    B = cu_seqlens.numel() - 1
    P, window = history.shape
    _expect(rewards, torch.float32, B, "rewards")
    _expect(prompt_ids, torch.int32, B, "prompt_ids")
    _expect(seen, torch.int64, P, "seen")
    _expect(loss_mask, torch.uint8, N, "loss_mask")
    _expect(cu_seqlens, torch.int32, B + 1, "cu_seqlens")
    _expect(adv, torch.float32, N, "adv")
    if history.dtype != torch.float32:
        raise ValueError("history must be fp32")
    _check(load().sao_running_mean_advantages(_ptr(rewards), _ptr(prompt_ids), B, P, _ptr(history), _ptr(seen),
                                              window, _ptr(loss_mask), _ptr(cu_seqlens), N, _ptr(adv), _ptr(ws),
                                              ws.numel(), _stream(stream)))


# ---------------------------------------------------------------------------
# kernel timing
# ---------------------------------------------------------------------------

def sao_profile_enable(on: bool):
    load().sao_profile_enable(1 if on else 0)


def sao_profile_reset():
    load().sao_profile_reset()


def sao_profile_read(cap: int = 64):
    """{kernel name: (launches, total ms)} since the last reset."""
    names = (ctypes.c_char_p * cap)()
    launches = (ctypes.c_int64 * cap)()
    ms = (ctypes.c_double * cap)()
    n = load().sao_profile_read(ctypes.cast(names, ctypes.c_void_p), ctypes.cast(launches, ctypes.c_void_p),
                                ctypes.cast(ms, ctypes.c_void_p), cap)
    return {names[i].decode(): (int(launches[i]), float(ms[i])) for i in range(n)}
