"""Python binding of libmc (include/mc.h): argument marshalling only.

Every function here checks tensor devices/dtypes/shapes, allocates outputs and
workspace with PyTorch (device memory is PyTorch's job), passes raw pointers
and the current CUDA stream to the C ABI, and raises on a non-OK status. All
arithmetic runs in libmc's kernels. If ``libmc.so`` has not been built the
first call raises: there is no fallback of any kind.
"""

from __future__ import annotations

import ctypes
import os
from typing import Optional

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libmc.so")
_lib = None

MC_OK = 0
STATUS_NAMES = {
    0: "MC_OK",
    1: "MC_ERR_INVALID_ARG",
    2: "MC_ERR_UNSUPPORTED",
    3: "MC_ERR_CUDA",
    4: "MC_ERR_TIMEOUT",
    5: "MC_ERR_WORKSPACE",
    6: "MC_ERR_TARGET_RANGE",
    7: "MC_ERR_SCRATCH_LIMIT",
}
MC_DEV_TIMEOUT = 0x1
MC_DEV_TARGET_RANGE = 0x2

# name -> (restype, argtypes); mirrors include/mc.h
_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_I32 = ctypes.c_int32
_F = ctypes.c_float
_SZ = ctypes.c_size_t
SIGNATURES = {
    "mc_status_string": (ctypes.c_char_p, [_I32]),
    "mc_last_cuda_error": (ctypes.c_char_p, []),
    "mc_version": (_I32, []),
    "mc_kernel_launches": (ctypes.c_uint64, []),
    "mc_token_logprobs_workspace_size": (_SZ, [_I64, _I32, _I32]),
    "mc_token_logprobs": (_I32, [_P, _P, _P, _I64, _I32, _I32, _F, _P, _P, _P, _P, _SZ, _P, _P]),
    "mc_token_logprobs_noalloc": (_I32, [_P, _P, _P, _I64, _I32, _I32, _F, _P, _P, _P, _P, _P]),
    "mc_token_logprob_state": (_I32, [_P, _P, _P, _I64, _I32, _I32, _I32, _F, _P, _P, _SZ, _P, _P]),
    "mc_merge_logprob_states": (_I32, [_P, _I32, _I64, _P, _P, _P, _P, _P]),
    "mc_token_logprobs_bwd_workspace_size": (_SZ, [_I64, _I32, _I32, _I64]),
    "mc_token_logprobs_bwd": (_I32, [_P, _P, _P, _P, _P, _P, _P, _P, _I64, _I32, _I32, _F, _P, _P, _I32, _P,
                                     _SZ, _P, _P]),
    "mc_seq_ratio_filter": (_I32, [_P, _P, _P, _P, _I32, _I64, _F, _F, _P, _P, _P, _P, _P, _P, _P, _P]),
    "mc_grpo_masked_loss_workspace_size": (_SZ, [_I32]),
    "mc_grpo_masked_loss": (_I32, [_P, _P, _P, _P, _P, _P, _P, _I32, _I64, _F, _F, _P, _F, _P, _P, _P, _P, _P, _P,
                                   _SZ, _P]),
    "mc_prime_echo_advantages": (_I32, [_P, _P, _P, _I32, _I32, _I32, _F, _F, _F, _F, _P, _P, _P]),
    "mc_selftest_bounded_wait": (_I32, [_P, _I64, _P]),
}


class McError(RuntimeError):
    def __init__(self, fn: str, status: int):
        detail = ""
        if status == 3 and _lib is not None:
            detail = ": " + _lib.mc_last_cuda_error().decode()
        super().__init__(f"{fn} -> {STATUS_NAMES.get(status, status)}{detail}")
        self.status = status


def lib_path() -> str:
    return _LIB_PATH


def lib() -> ctypes.CDLL:
    """Load libmc.so (once). Raises if it is missing: build it first."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError(f"libmc.so not found at {_LIB_PATH}; run __graft_entry__.build() "
                               "(python -m paper_2606_04847_gb300.build)")
        L = ctypes.CDLL(_LIB_PATH)
        for name, (res, args) in SIGNATURES.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


def _ptr(t: Optional[torch.Tensor]):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(stream) -> ctypes.c_void_p:
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def _check(fn: str, status: int):
    if status != MC_OK:
        raise McError(fn, status)


def _need(t: torch.Tensor, name: str, dtype, ndim: int):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if t.dim() != ndim or not t.is_contiguous():
        raise ValueError(f"{name} must be a contiguous {ndim}-d tensor")


def _shaped(t: Optional[torch.Tensor], name: str, dtype, shape, device) -> Optional[torch.Tensor]:
    """Checks a caller-supplied tensor (None passes): dtype, device, contiguity
    and exact shape, so that no kernel writes or reads past its end."""
    if t is None:
        return None
    _need(t, name, dtype, len(shape))
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")
    if t.device != device:
        raise ValueError(f"{name} must be on {device}, got {t.device}")
    return t


def _ws(t: torch.Tensor, device) -> torch.Tensor:
    """A caller-supplied workspace: uint8, 1-d, contiguous, on `device` (its
    size is checked by the library against the call's requirement)."""
    _need(t, "workspace", torch.uint8, 1)
    if t.device != device:
        raise ValueError(f"workspace must be on {device}, got {t.device}")
    return t


def version() -> tuple:
    v = lib().mc_version()
    return (v >> 16, v & 0xFFFF)


def kernel_launches() -> int:
    """Kernels libmc has enqueued in this process so far (mc_kernel_launches)."""
    return int(lib().mc_kernel_launches())


def forward_workspace_size(N: int, d: int, V: int) -> int:
    return int(lib().mc_token_logprobs_workspace_size(N, d, V))


def backward_workspace_size(N: int, d: int, V: int, rows_per_chunk: Optional[int] = None) -> int:
    return int(lib().mc_token_logprobs_bwd_workspace_size(N, d, V, N if rows_per_chunk is None else rows_per_chunk))


def token_logprobs(hidden: torch.Tensor, w_vocab: torch.Tensor, targets: torch.Tensor,
                   inv_temperature: float = 1.0, *, out: Optional[dict] = None,
                   workspace: Optional[torch.Tensor] = None, dev_status: Optional[torch.Tensor] = None,
                   stream=None) -> dict:
    """mc_token_logprobs: returns {"logp", "entropy", "lse"} (fp32 [N])."""
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(w_vocab, "w_vocab", torch.bfloat16, 2)
    _need(targets, "targets", torch.int32, 1)
    N, d = hidden.shape
    V = w_vocab.shape[0]
    if w_vocab.shape[1] != d or targets.shape[0] != N:
        raise ValueError("shape mismatch")
    dev = hidden.device
    _shaped(w_vocab, "w_vocab", torch.bfloat16, (V, d), dev)
    _shaped(targets, "targets", torch.int32, (N,), dev)
    if out is None:
        out = {k: torch.empty(N, dtype=torch.float32, device=dev) for k in ("logp", "entropy", "lse")}
    _shaped(out["logp"], "out['logp']", torch.float32, (N,), dev)
    for k in ("entropy", "lse"):
        _shaped(out.get(k), f"out['{k}']", torch.float32, (N,), dev)
    need = forward_workspace_size(N, d, V)
    if workspace is None:
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
    _ws(workspace, dev)
    st = lib().mc_token_logprobs(_ptr(hidden), _ptr(w_vocab), _ptr(targets), N, d, V, float(inv_temperature),
                                 _ptr(out["logp"]), _ptr(out.get("entropy")), _ptr(out.get("lse")),
                                 _ptr(workspace), workspace.numel(), _ptr(dev_status), _stream(stream))
    _check("mc_token_logprobs", st)
    return out


def token_logprob_state(hidden: torch.Tensor, w_shard: torch.Tensor, targets: torch.Tensor, v_begin: int,
                        inv_temperature: float = 1.0, *, state: Optional[torch.Tensor] = None,
                        workspace: Optional[torch.Tensor] = None, dev_status: Optional[torch.Tensor] = None,
                        stream=None) -> torch.Tensor:
    """mc_token_logprob_state: the [N, 4] softmax state (m, s, u, z_y) of one vocabulary slice."""
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(w_shard, "w_shard", torch.bfloat16, 2)
    _need(targets, "targets", torch.int32, 1)
    N, d = hidden.shape
    Vs = w_shard.shape[0]
    dev = hidden.device
    _shaped(w_shard, "w_shard", torch.bfloat16, (Vs, d), dev)
    _shaped(targets, "targets", torch.int32, (N,), dev)
    if state is None:
        state = torch.empty((N, 4), dtype=torch.float32, device=dev)
    _shaped(state, "state", torch.float32, (N, 4), dev)
    if workspace is None:
        workspace = torch.empty(max(forward_workspace_size(N, d, Vs), 256), dtype=torch.uint8, device=dev)
    _ws(workspace, dev)
    st = lib().mc_token_logprob_state(_ptr(hidden), _ptr(w_shard), _ptr(targets), N, d, Vs, int(v_begin),
                                      float(inv_temperature), _ptr(state), _ptr(workspace), workspace.numel(),
                                      _ptr(dev_status), _stream(stream))
    _check("mc_token_logprob_state", st)
    return state


def merge_logprob_states(states: torch.Tensor, *, out: Optional[dict] = None,
                         dev_status: Optional[torch.Tensor] = None, stream=None) -> dict:
    """mc_merge_logprob_states: {"logp", "entropy", "lse"} from slice states [P, N, 4]."""
    _need(states, "states", torch.float32, 3)
    P, N, four = states.shape
    if four != 4:
        raise ValueError("states must be [P, N, 4]")
    if out is None:
        out = {k: torch.empty(N, dtype=torch.float32, device=states.device) for k in ("logp", "entropy", "lse")}
    _shaped(out["logp"], "out['logp']", torch.float32, (N,), states.device)
    for k in ("entropy", "lse"):
        _shaped(out.get(k), f"out['{k}']", torch.float32, (N,), states.device)
    st = lib().mc_merge_logprob_states(_ptr(states), P, N, _ptr(out["logp"]), _ptr(out.get("entropy")),
                                       _ptr(out.get("lse")), _ptr(dev_status), _stream(stream))
    _check("mc_merge_logprob_states", st)
    return out


def token_logprobs_noalloc(hidden: torch.Tensor, w_vocab: torch.Tensor, targets: torch.Tensor,
                           inv_temperature: float = 1.0, *, out: dict, dev_status: Optional[torch.Tensor] = None,
                           stream=None) -> dict:
    """mc_token_logprobs_noalloc: the forward with the library's fixed scratch.

    For callers that must not allocate device memory: the caller supplies the
    output tensors in ``out`` ("logp", optional "entropy"/"lse") and nothing is
    allocated here or in the library. Raises McError(MC_ERR_SCRATCH_LIMIT) when
    the problem needs more than the fixed scratch.
    """
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(w_vocab, "w_vocab", torch.bfloat16, 2)
    _need(targets, "targets", torch.int32, 1)
    N, d = hidden.shape
    V = w_vocab.shape[0]
    dev = hidden.device
    _shaped(w_vocab, "w_vocab", torch.bfloat16, (V, d), dev)
    _shaped(targets, "targets", torch.int32, (N,), dev)
    _shaped(out["logp"], "out['logp']", torch.float32, (N,), dev)
    for k in ("entropy", "lse"):
        _shaped(out.get(k), f"out['{k}']", torch.float32, (N,), dev)
    st = lib().mc_token_logprobs_noalloc(_ptr(hidden), _ptr(w_vocab), _ptr(targets), N, d, V,
                                         float(inv_temperature), _ptr(out["logp"]), _ptr(out.get("entropy")),
                                         _ptr(out.get("lse")), _ptr(dev_status), _stream(stream))
    _check("mc_token_logprobs_noalloc", st)
    return out


def token_logprobs_bwd(hidden: torch.Tensor, w_vocab: torch.Tensor, targets: torch.Tensor, lse: torch.Tensor,
                       entropy: Optional[torch.Tensor], grad_logp: torch.Tensor,
                       grad_entropy: Optional[torch.Tensor] = None, inv_temperature: float = 1.0, *,
                       row_keep: Optional[torch.Tensor] = None,
                       grad_hidden: Optional[torch.Tensor] = None, grad_w: Optional[torch.Tensor] = None,
                       accumulate: bool = False, workspace: Optional[torch.Tensor] = None,
                       rows_per_chunk: Optional[int] = None, dev_status: Optional[torch.Tensor] = None,
                       stream=None) -> dict:
    """mc_token_logprobs_bwd: returns {"grad_hidden" (bf16 [N,d]), "grad_w" (fp32 [V,d])}."""
    _need(hidden, "hidden", torch.bfloat16, 2)
    _need(w_vocab, "w_vocab", torch.bfloat16, 2)
    _need(targets, "targets", torch.int32, 1)
    _need(lse, "lse", torch.float32, 1)
    _need(grad_logp, "grad_logp", torch.float32, 1)
    if row_keep is not None:
        _need(row_keep, "row_keep", torch.uint8, 1)
    N, d = hidden.shape
    V = w_vocab.shape[0]
    dev = hidden.device
    _shaped(w_vocab, "w_vocab", torch.bfloat16, (V, d), dev)
    _shaped(targets, "targets", torch.int32, (N,), dev)
    _shaped(lse, "lse", torch.float32, (N,), dev)
    _shaped(entropy, "entropy", torch.float32, (N,), dev)
    _shaped(grad_logp, "grad_logp", torch.float32, (N,), dev)
    _shaped(grad_entropy, "grad_entropy", torch.float32, (N,), dev)
    _shaped(row_keep, "row_keep", torch.uint8, (N,), dev)
    if grad_hidden is None:
        grad_hidden = torch.empty((N, d), dtype=torch.bfloat16, device=dev)
    if grad_w is None:
        grad_w = torch.empty((V, d), dtype=torch.float32, device=dev)
    _shaped(grad_hidden, "grad_hidden", torch.bfloat16, (N, d), dev)
    _shaped(grad_w, "grad_w", torch.float32, (V, d), dev)
    if workspace is None:
        need = backward_workspace_size(N, d, V, rows_per_chunk)
        workspace = torch.empty(max(need, 256), dtype=torch.uint8, device=dev)
    _ws(workspace, dev)
    st = lib().mc_token_logprobs_bwd(_ptr(hidden), _ptr(w_vocab), _ptr(targets), _ptr(lse), _ptr(entropy),
                                     _ptr(grad_logp), _ptr(grad_entropy), _ptr(row_keep), N, d, V,
                                     float(inv_temperature),
                                     _ptr(grad_hidden), _ptr(grad_w), int(bool(accumulate)), _ptr(workspace),
                                     workspace.numel(), _ptr(dev_status), _stream(stream))
    _check("mc_token_logprobs_bwd", st)
    return {"grad_hidden": grad_hidden, "grad_w": grad_w}


def seq_ratio_filter(logp_policy: torch.Tensor, logp_behaviour: torch.Tensor, loss_mask: Optional[torch.Tensor],
                     cu_seqlens: torch.Tensor, delta: float, delta_vanilla: float = -1.0, *,
                     token_outputs: bool = True, out: Optional[dict] = None, stream=None) -> dict:
    """mc_seq_ratio_filter: per-sequence signed/absolute mean log-ratio, counts, masks; per-token ratio/keep."""
    _need(logp_policy, "logp_policy", torch.float32, 1)
    _need(logp_behaviour, "logp_behaviour", torch.float32, 1)
    _need(cu_seqlens, "cu_seqlens", torch.int64, 1)
    if loss_mask is not None:
        _need(loss_mask, "loss_mask", torch.uint8, 1)
    N = logp_policy.shape[0]
    B = cu_seqlens.shape[0] - 1
    dev = logp_policy.device
    if out is None:
        out = {
            "signed_mean": torch.empty(B, dtype=torch.float32, device=dev),
            "abs_mean": torch.empty(B, dtype=torch.float32, device=dev),
            "n_tokens": torch.empty(B, dtype=torch.int32, device=dev),
            "keep": torch.empty(B, dtype=torch.uint8, device=dev),
            "keep_vanilla": torch.empty(B, dtype=torch.uint8, device=dev),
        }
        if token_outputs:
            out["token_ratio"] = torch.empty(N, dtype=torch.float32, device=dev)
            out["token_keep"] = torch.empty(N, dtype=torch.uint8, device=dev)
    _shaped(logp_behaviour, "logp_behaviour", torch.float32, (N,), dev)
    _shaped(loss_mask, "loss_mask", torch.uint8, (N,), dev)
    _shaped(cu_seqlens, "cu_seqlens", torch.int64, (B + 1,), dev)
    for k, dt, n in (("signed_mean", torch.float32, B), ("abs_mean", torch.float32, B), ("n_tokens", torch.int32, B),
                     ("keep", torch.uint8, B), ("keep_vanilla", torch.uint8, B), ("token_ratio", torch.float32, N),
                     ("token_keep", torch.uint8, N)):
        if k in ("signed_mean", "abs_mean", "n_tokens", "keep") and out.get(k) is None:
            raise ValueError(f"out['{k}'] is required")
        _shaped(out.get(k), f"out['{k}']", dt, (n,), dev)
    st = lib().mc_seq_ratio_filter(_ptr(logp_policy), _ptr(logp_behaviour), _ptr(loss_mask), _ptr(cu_seqlens),
                                   B, N, float(delta), float(delta_vanilla), _ptr(out["signed_mean"]),
                                   _ptr(out["abs_mean"]), _ptr(out["n_tokens"]), _ptr(out["keep"]),
                                   _ptr(out.get("keep_vanilla")), _ptr(out.get("token_ratio")),
                                   _ptr(out.get("token_keep")), _stream(stream))
    _check("mc_seq_ratio_filter", st)
    return out


def grpo_masked_loss(logp_policy: torch.Tensor, logp_behaviour: torch.Tensor, loss_mask: Optional[torch.Tensor],
                     cu_seqlens: torch.Tensor, advantages: torch.Tensor, keep: torch.Tensor, n_tokens: torch.Tensor,
                     eps_low: float, eps_high: float, *, logp_ref: Optional[torch.Tensor] = None,
                     beta: float = 0.0, out: Optional[dict] = None, workspace: Optional[torch.Tensor] = None,
                     stream=None) -> dict:
    """mc_grpo_masked_loss: {"loss" [1], "grad_logp" [N], "seq_loss" [B], "n_clipped" [1], "kl" [1]}."""
    if logp_ref is not None:
        _need(logp_ref, "logp_ref", torch.float32, 1)
    _need(logp_policy, "logp_policy", torch.float32, 1)
    _need(logp_behaviour, "logp_behaviour", torch.float32, 1)
    _need(cu_seqlens, "cu_seqlens", torch.int64, 1)
    _need(advantages, "advantages", torch.float32, 1)
    _need(keep, "keep", torch.uint8, 1)
    _need(n_tokens, "n_tokens", torch.int32, 1)
    if loss_mask is not None:
        _need(loss_mask, "loss_mask", torch.uint8, 1)
    N = logp_policy.shape[0]
    B = cu_seqlens.shape[0] - 1
    dev = logp_policy.device
    if out is None:
        out = {"loss": torch.empty(1, dtype=torch.float32, device=dev),
               "grad_logp": torch.empty(N, dtype=torch.float32, device=dev),
               "seq_loss": torch.empty(B, dtype=torch.float32, device=dev),
               "n_clipped": torch.empty(1, dtype=torch.int32, device=dev),
               "kl": torch.empty(1, dtype=torch.float32, device=dev)}
    _shaped(logp_behaviour, "logp_behaviour", torch.float32, (N,), dev)
    _shaped(logp_ref, "logp_ref", torch.float32, (N,), dev)
    _shaped(loss_mask, "loss_mask", torch.uint8, (N,), dev)
    _shaped(cu_seqlens, "cu_seqlens", torch.int64, (B + 1,), dev)
    _shaped(advantages, "advantages", torch.float32, (B,), dev)
    _shaped(keep, "keep", torch.uint8, (B,), dev)
    _shaped(n_tokens, "n_tokens", torch.int32, (B,), dev)
    for k, dt, n in (("loss", torch.float32, 1), ("grad_logp", torch.float32, N), ("seq_loss", torch.float32, B),
                     ("n_clipped", torch.int32, 1), ("kl", torch.float32, 1)):
        if k in ("loss", "grad_logp") and out.get(k) is None:
            raise ValueError(f"out['{k}'] is required")
        _shaped(out.get(k), f"out['{k}']", dt, (n,), dev)
    if workspace is None:
        workspace = torch.empty(lib().mc_grpo_masked_loss_workspace_size(B), dtype=torch.uint8, device=dev)
    _ws(workspace, dev)
    st = lib().mc_grpo_masked_loss(_ptr(logp_policy), _ptr(logp_behaviour), _ptr(loss_mask), _ptr(cu_seqlens),
                                   _ptr(advantages), _ptr(keep), _ptr(n_tokens), B, N, float(eps_low),
                                   float(eps_high), _ptr(logp_ref), float(beta), _ptr(out["loss"]),
                                   _ptr(out["grad_logp"]), _ptr(out.get("seq_loss")), _ptr(out.get("n_clipped")),
                                   _ptr(out.get("kl")), _ptr(workspace), workspace.numel(), _stream(stream))
    _check("mc_grpo_masked_loss", st)
    return out


def prime_echo_advantages(scores: torch.Tensor, success: torch.Tensor, n_turns: torch.Tensor, group_size: int,
                          alpha: float = 0.75, beta1: float = 0.0, beta2: float = 0.0, eps: float = 1e-6, *,
                          stream=None) -> dict:
    """mc_prime_echo_advantages: {"reward" [T], "advantage" [T]} from per-turn scores [T, K]."""
    _need(scores, "scores", torch.float32, 2)
    _need(success, "success", torch.uint8, 2)
    _need(n_turns, "n_turns", torch.int32, 1)
    T, K = scores.shape
    _shaped(success, "success", torch.uint8, (T, K), scores.device)
    _shaped(n_turns, "n_turns", torch.int32, (T,), scores.device)
    out = {"reward": torch.empty(T, dtype=torch.float32, device=scores.device),
           "advantage": torch.empty(T, dtype=torch.float32, device=scores.device)}
    st = lib().mc_prime_echo_advantages(_ptr(scores), _ptr(success), _ptr(n_turns), T, K, int(group_size),
                                        float(alpha), float(beta1), float(beta2), float(eps), _ptr(out["reward"]),
                                        _ptr(out["advantage"]), _stream(stream))
    _check("mc_prime_echo_advantages", st)
    return out


def selftest_bounded_wait(dev_status: torch.Tensor, timeout_ns: int, stream=None) -> None:
    _need(dev_status, "dev_status", torch.int32, 1)
    _check("mc_selftest_bounded_wait", lib().mc_selftest_bounded_wait(_ptr(dev_status), int(timeout_ns),
                                                                      _stream(stream)))
