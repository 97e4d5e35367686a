"""Python binding of ``libgrpo_gb300.so`` (argument marshalling only).

The functions carry the C ABI's names (include/grpo.h) and take torch tensors that already live
on the GPU; they check shapes/dtypes, allocate outputs with torch when the caller passes none, and
call the library on the current torch stream. All arithmetic runs in the library's CUDA kernels:
there is no fallback, and importing this module fails loudly if the library is missing.
"""
from __future__ import annotations

import ctypes
import os
import re
from dataclasses import dataclass
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libgrpo_gb300.so")
HEADER_PATH = os.path.join(os.path.dirname(_HERE), "include", "grpo.h")

GRPO_F32, GRPO_BF16 = 0, 1
STATIC_SCRATCH_BYTES = 64 << 20      # GRPO_STATIC_SCRATCH_BYTES of include/grpo.h
GEMM_WINDOW_DEFAULT = (256, 1)       # GRPO_GEMM_WINDOW_DEFAULT_{CHECK,LAG} of include/grpo.h
STD_MODES = {"unbiased": 0, "population": 1}
AGG_MODES = {"seq_mean": 0, "token_mean": 1}
STATUS_NAMES = {0: "GRPO_OK", -1: "GRPO_ERR_INVALID_ARG", -2: "GRPO_ERR_UNSUPPORTED",
                -3: "GRPO_ERR_CUDA", -4: "GRPO_ERR_WORKSPACE", -5: "GRPO_ERR_TOKEN_RANGE",
                -6: "GRPO_ERR_TIMEOUT", -7: "GRPO_ERR_GROUPS"}
KERNEL_NAMES = ["mask_scan", "pack_tokens", "group_adv", "fwd_gemm_tc", "fwd_merge", "loss_tokens",
                "loss_final", "bwd_dz_gemm_tc", "bwd_dh_gemm_tc", "bwd_dw_gemm_tc",
                "dh_zero_unscored", "f32_fwd", "f32_dh", "f32_dw", "rewards", "shard_stats",
                "merge_shards", "gather_rows"]


class GrpoError(RuntimeError):
    def __init__(self, status: int, what: str):
        self.status = status
        super().__init__(f"{what}: {STATUS_NAMES.get(status, status)} "
                         f"({_lib().grpo_status_string(status).decode()})")


_LIB = None
_p, _i32, _i64, _f32, _f64, _sz = (ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64,
                                   ctypes.c_float, ctypes.c_double, ctypes.c_size_t)


def _declare(lib):
    sig = {
        "grpo_workspace_bytes": (_sz, [_i32, _i32, _i32, _i32, _i32, _i32]),
        "grpo_workspace_bytes_kl": (_sz, [_i32, _i32, _i32, _i32, _i32, _i32]),
        "grpo_workspace_init": (ctypes.c_int, [_p, _sz, _p]),
        "group_advantages": (ctypes.c_int, [_p, _p, _i32, _i32, _i32, _f32, _p, _p, _sz, _p]),
        "grpo_score_fwd": (ctypes.c_int, [_p, _p, _i32, _p, _p, _i32, _i32, _i32, _i32, _p, _p,
                                          _p, _p, _p, _p, _sz, _p]),
        "grpo_loss_bwd": (ctypes.c_int, [_p, _p, _i32, _p, _p, _i32, _i32, _i32, _i32, _p, _p,
                                         _p, _p, _p, _p, _f32, _f32, _f32, _i32, _f64, _p, _p,
                                         _p, _p, _sz, _p]),
        "grpo_last_device_error": (ctypes.c_int, [_p, ctypes.POINTER(_i32), _p]),
        "grpo_status_string": (ctypes.c_char_p, [ctypes.c_int]),
        "grpo_kernel_name": (ctypes.c_char_p, [_i32]),
        "grpo_timing_enable": (ctypes.c_int, [_i32]),
        "grpo_timing_reset": (ctypes.c_int, []),
        "grpo_timing_read": (ctypes.c_int, [_i32, ctypes.POINTER(_i64), ctypes.POINTER(_f64)]),
        "grpo_debug_inject_stall": (ctypes.c_int, [_i32]),
        "grpo_set_cta_pair": (ctypes.c_int, [_i32]),
        "grpo_set_tile_mode": (ctypes.c_int, [_i32]),
        "grpo_get_tile_mode": (ctypes.c_int, []),
        "grpo_set_role_tile_mode": (ctypes.c_int, [_i32, _i32]),
        "grpo_get_role_tile_mode": (ctypes.c_int, [_i32]),
        "grpo_set_gemm_window": (ctypes.c_int, [_i32, _i32]),
        "grpo_sft_loss_bwd": (ctypes.c_int, [_p, _p, _i32, _p, _p, _i32, _i32, _i32, _i32, _p,
                                             _p, _p, _i32, _f64, _p, _p, _p, _p, _sz, _p]),
        "grpo_rewards": (ctypes.c_int, [_p, _p, _p, _p, _p, _i32, _f32, _p, _p]),
        "grpo_score_fwd_kl": (ctypes.c_int, [_p, _p, _p, _p, _i32, _p, _p, _i32, _i32, _i32, _i32,
                                             _p, _p, _p, _p, _p, _p, _p, _p, _sz, _p]),
        "grpo_loss_bwd_kl": (ctypes.c_int, [_p, _p, _p, _p, _i32, _p, _p, _i32, _i32, _i32, _i32,
                                            _p, _p, _p, _p, _p, _p, _p, _f32, _f32, _f32, _i32,
                                            _f64, _p, _p, _p, _p, _sz, _p]),
        "grpo_score_fwd_shard": (ctypes.c_int, [_p, _p, _i32, _p, _p, _i32, _i32, _i32, _i32,
                                                _i32, _i32, _p, _p, _p, _sz, _p]),
        "grpo_merge_shard_stats": (ctypes.c_int, [_p, _p, _i32, _p, _p, _i32, _i32, _i32, _p, _p,
                                                  _p, _p, _p, _p, _sz, _p]),
        "grpo_loss_bwd_shard": (ctypes.c_int, [_p, _p, _i32, _p, _p, _i32, _i32, _i32, _i32,
                                               _i32, _i32, _p, _p, _p, _p, _p, _p, _f32, _f32,
                                               _f32, _i32, _f64, _p, _p, _p, _p, _sz, _p]),
        "grpo_score_fwd_static": (ctypes.c_int, [_p, _p, _i32, _p, _p, _i32, _i32, _i32, _i32, _p,
                                                 _p, _p, _p, _p, _p, _p]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    return lib


def _lib():
    global _LIB
    if _LIB is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with "
                              "`python -c 'import __graft_entry__ as g; g.build()'` "
                              "(the GRPO path has no fallback)")
        _LIB = _declare(ctypes.CDLL(LIB_PATH))
    return _LIB


def header_functions(path: str = HEADER_PATH):
    """Names of the functions declared in include/grpo.h."""
    text = open(path).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b([a-z_][a-z0-9_]*)\s*\([^;{]*\)\s*;", text)))


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t: Optional[torch.Tensor]):
    return ctypes.c_void_p(0 if t is None else t.data_ptr())


def _check(status: int, what: str):
    if status != 0:
        raise GrpoError(status, what)


def _need(t: torch.Tensor, name: str, dtype, shape=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if not t.is_cuda:
        raise ValueError(f"{name} must live on a CUDA device")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} must have shape {tuple(shape)}, got {tuple(t.shape)}")


def _dtype_code(H: torch.Tensor) -> int:
    if H.dtype == torch.bfloat16:
        return GRPO_BF16
    if H.dtype == torch.float32:
        return GRPO_F32
    raise ValueError(f"H must be bf16 or f32, got {H.dtype}")


# ---------------------------------------------------------------------------------------------
def grpo_workspace_bytes(S: int, T: int, d: int, V: int, dtype, vocab_chunk: int = 0) -> int:
    code = dtype if isinstance(dtype, int) else (GRPO_BF16 if dtype == torch.bfloat16 else GRPO_F32)
    return int(_lib().grpo_workspace_bytes(S, T, d, V, code, vocab_chunk))


def grpo_workspace_bytes_kl(S: int, T: int, d: int, V: int, dtype, vocab_chunk: int = 0) -> int:
    """Workspace of the exact-KL entry points (also serves every other entry point)."""
    code = dtype if isinstance(dtype, int) else (GRPO_BF16 if dtype == torch.bfloat16 else GRPO_F32)
    return int(_lib().grpo_workspace_bytes_kl(S, T, d, V, code, vocab_chunk))


@dataclass
class Workspace:
    """A device workspace (torch-owned bytes) plus its size; initialised on creation."""
    buf: torch.Tensor
    nbytes: int

    @classmethod
    def create(cls, nbytes: int, device="cuda") -> "Workspace":
        nbytes = max(int(nbytes), 256)
        buf = torch.empty(nbytes + 256, dtype=torch.uint8, device=device)
        off = (-buf.data_ptr()) % 256
        view = buf[off: off + nbytes]
        ws = cls(view, nbytes)
        _check(_lib().grpo_workspace_init(_ptr(view), nbytes, _stream()), "grpo_workspace_init")
        return ws

    @classmethod
    def for_problem(cls, S, T, d, V, dtype, vocab_chunk=0, device="cuda",
                    kl=False) -> "Workspace":
        """Workspace for this shape; `kl=True` sizes it for the exact-KL entry points."""
        n = (grpo_workspace_bytes_kl if kl else grpo_workspace_bytes)(S, T, d, V, dtype,
                                                                      vocab_chunk)
        if n == 0:
            raise ValueError("invalid problem shape")
        return cls.create(n, device)

    @property
    def ptr(self):
        return _ptr(self.buf)


def grpo_workspace_init(ws: Workspace, stream=None):
    _check(_lib().grpo_workspace_init(ws.ptr, ws.nbytes, _stream(stream)), "grpo_workspace_init")


def group_advantages(rewards: torch.Tensor, group_offsets: torch.Tensor, ws: Workspace,
                     std_mode: str = "unbiased", std_eps: float = 1e-4,
                     adv_out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    S = rewards.numel()
    _need(rewards, "rewards", torch.float32, (S,))
    _need(group_offsets, "group_offsets", torch.int32)
    if adv_out is None:
        adv_out = torch.empty_like(rewards)
    _need(adv_out, "adv_out", torch.float32, (S,))
    st = _lib().group_advantages(_ptr(rewards), _ptr(group_offsets), group_offsets.numel() - 1, S,
                                 STD_MODES[std_mode], float(std_eps), _ptr(adv_out), ws.ptr,
                                 ws.nbytes, _stream(stream))
    _check(st, "group_advantages")
    return adv_out


def grpo_score_fwd(H: torch.Tensor, W: torch.Tensor, tokens: torch.Tensor, mask: torch.Tensor,
                   ws: Workspace, out: Optional[dict] = None, stream=None) -> dict:
    """Returns dict(logp, lse, entropy [S,T] f32, argmax [S,T] int32, valid_count [S] int32)."""
    if H.dim() != 3:
        raise ValueError("H must be [S, T, d]")
    S, T, d = H.shape
    V = W.shape[0]
    code = _dtype_code(H)
    _need(H, "H", H.dtype)
    _need(W, "W", H.dtype, (V, d))
    _need(tokens, "tokens", torch.int32, (S, T))
    _need(mask, "mask", torch.uint8, (S, T))
    if out is None:
        f = dict(dtype=torch.float32, device=H.device)
        out = {"logp": torch.empty((S, T), **f), "lse": torch.empty((S, T), **f),
               "entropy": torch.empty((S, T), **f),
               "argmax": torch.empty((S, T), dtype=torch.int32, device=H.device),
               "valid_count": torch.empty((S,), dtype=torch.int32, device=H.device)}
    for k in ("logp", "lse", "entropy"):
        _need(out[k], k, torch.float32, (S, T))
    _need(out["argmax"], "argmax", torch.int32, (S, T))
    _need(out["valid_count"], "valid_count", torch.int32, (S,))
    st = _lib().grpo_score_fwd(_ptr(H), _ptr(W), code, _ptr(tokens), _ptr(mask), S, T, d, V,
                               _ptr(out["logp"]), _ptr(out["lse"]), _ptr(out["entropy"]),
                               _ptr(out["argmax"]), _ptr(out["valid_count"]), ws.ptr, ws.nbytes,
                               _stream(stream))
    _check(st, "grpo_score_fwd")
    return out


def grpo_loss_bwd(H, W, tokens, mask, logp, lse, old_logp, ref_logp, adv, valid_count,
                  ws: Workspace, eps_low=0.2, eps_high=0.2, beta=0.04, agg="seq_mean", norm=0.0,
                  out: Optional[dict] = None, stream=None) -> dict:
    """Returns dict(loss [1] f32 device, dH [S,T,d] H.dtype, dW [V,d] f32)."""
    S, T, d = H.shape
    V = W.shape[0]
    code = _dtype_code(H)
    _need(H, "H", H.dtype)
    _need(W, "W", H.dtype, (V, d))
    _need(tokens, "tokens", torch.int32, (S, T))
    _need(mask, "mask", torch.uint8, (S, T))
    for name, t in (("logp", logp), ("lse", lse), ("old_logp", old_logp)):
        _need(t, name, torch.float32, (S, T))
    if ref_logp is not None:
        _need(ref_logp, "ref_logp", torch.float32, (S, T))
    _need(adv, "adv", torch.float32, (S,))
    _need(valid_count, "valid_count", torch.int32, (S,))
    if out is None:
        out = {"loss": torch.empty((1,), dtype=torch.float32, device=H.device),
               "dH": torch.empty_like(H),
               "dW": torch.empty((V, d), dtype=torch.float32, device=H.device)}
    _need(out["loss"], "loss", torch.float32, (1,))
    _need(out["dH"], "dH", H.dtype, (S, T, d))
    _need(out["dW"], "dW", torch.float32, (V, d))
    st = _lib().grpo_loss_bwd(_ptr(H), _ptr(W), code, _ptr(tokens), _ptr(mask), S, T, d, V,
                              _ptr(logp), _ptr(lse), _ptr(old_logp), _ptr(ref_logp), _ptr(adv),
                              _ptr(valid_count), float(eps_low), float(eps_high), float(beta),
                              AGG_MODES[agg], float(norm), _ptr(out["loss"]), _ptr(out["dH"]),
                              _ptr(out["dW"]), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "grpo_loss_bwd")
    return out


def grpo_score_fwd_static(H: torch.Tensor, W: torch.Tensor, tokens: torch.Tensor,
                          mask: torch.Tensor, out: Optional[dict] = None, stream=None) -> dict:
    """grpo_score_fwd with the library's fixed device scratch instead of a workspace (for callers
    that cannot allocate device memory). Adds out["status"], a device int32 status word."""
    S, T, d = H.shape
    V = W.shape[0]
    code = _dtype_code(H)
    _need(H, "H", H.dtype)
    _need(W, "W", H.dtype, (V, d))
    _need(tokens, "tokens", torch.int32, (S, T))
    _need(mask, "mask", torch.uint8, (S, T))
    if out is None:
        f = dict(dtype=torch.float32, device=H.device)
        out = {"logp": torch.empty((S, T), **f), "lse": torch.empty((S, T), **f),
               "entropy": torch.empty((S, T), **f),
               "argmax": torch.empty((S, T), dtype=torch.int32, device=H.device),
               "valid_count": torch.empty((S,), dtype=torch.int32, device=H.device),
               "status": torch.empty((1,), dtype=torch.int32, device=H.device)}
    st = _lib().grpo_score_fwd_static(_ptr(H), _ptr(W), code, _ptr(tokens), _ptr(mask), S, T, d,
                                      V, _ptr(out["logp"]), _ptr(out["lse"]),
                                      _ptr(out["entropy"]), _ptr(out["argmax"]),
                                      _ptr(out["valid_count"]), _ptr(out.get("status")),
                                      _stream(stream))
    _check(st, "grpo_score_fwd_static")
    return out


def grpo_sft_loss_bwd(H, W, tokens, mask, logp, lse, valid_count, ws: Workspace,
                      agg="token_mean", norm=0.0, out: Optional[dict] = None, stream=None) -> dict:
    """Distillation (token cross-entropy) loss and gradients; dict(loss, dH, dW)."""
    S, T, d = H.shape
    V = W.shape[0]
    code = _dtype_code(H)
    _need(H, "H", H.dtype)
    _need(W, "W", H.dtype, (V, d))
    _need(tokens, "tokens", torch.int32, (S, T))
    _need(mask, "mask", torch.uint8, (S, T))
    _need(logp, "logp", torch.float32, (S, T))
    _need(lse, "lse", torch.float32, (S, T))
    _need(valid_count, "valid_count", torch.int32, (S,))
    if out is None:
        out = {"loss": torch.empty((1,), dtype=torch.float32, device=H.device),
               "dH": torch.empty_like(H),
               "dW": torch.empty((V, d), dtype=torch.float32, device=H.device)}
    st = _lib().grpo_sft_loss_bwd(_ptr(H), _ptr(W), code, _ptr(tokens), _ptr(mask), S, T, d, V,
                                  _ptr(logp), _ptr(lse), _ptr(valid_count), AGG_MODES[agg],
                                  float(norm), _ptr(out["loss"]), _ptr(out["dH"]),
                                  _ptr(out["dW"]), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "grpo_sft_loss_bwd")
    return out


def grpo_rewards(correct, t_base, t_new, tools_used, tools_avail, lambda_tools=0.5,
                 r_out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Eq. 2-4 rewards of n completions (device tensors)."""
    n = correct.numel()
    _need(correct, "correct", torch.uint8, (n,))
    _need(t_base, "t_base", torch.float32, (n,))
    _need(t_new, "t_new", torch.float32, (n,))
    _need(tools_used, "tools_used", torch.int32, (n,))
    _need(tools_avail, "tools_avail", torch.int32, (n,))
    if r_out is None:
        r_out = torch.empty((n,), dtype=torch.float32, device=correct.device)
    st = _lib().grpo_rewards(_ptr(correct), _ptr(t_base), _ptr(t_new), _ptr(tools_used),
                             _ptr(tools_avail), n, float(lambda_tools), _ptr(r_out),
                             _stream(stream))
    _check(st, "grpo_rewards")
    return r_out


def grpo_score_fwd_kl(H, W, H_ref, W_ref, tokens, mask, ws: Workspace, out: Optional[dict] = None,
                      stream=None) -> dict:
    """Forward with the exact per-token KL to the reference model: grpo_score_fwd's outputs plus
    lse_ref and kl."""
    S, T, d = H.shape
    V = W.shape[0]
    for name, t, shape in (("H", H, (S, T, d)), ("W", W, (V, d)), ("H_ref", H_ref, (S, T, d)),
                           ("W_ref", W_ref, (V, d))):
        _need(t, name, torch.bfloat16, shape)
    _need(tokens, "tokens", torch.int32, (S, T))
    _need(mask, "mask", torch.uint8, (S, T))
    if out is None:
        f = dict(dtype=torch.float32, device=H.device)
        out = {k: torch.empty((S, T), **f) for k in ("logp", "lse", "entropy", "lse_ref", "kl")}
        out["argmax"] = torch.empty((S, T), dtype=torch.int32, device=H.device)
        out["valid_count"] = torch.empty((S,), dtype=torch.int32, device=H.device)
    st = _lib().grpo_score_fwd_kl(_ptr(H), _ptr(W), _ptr(H_ref), _ptr(W_ref), GRPO_BF16,
                                  _ptr(tokens), _ptr(mask), S, T, d, V, _ptr(out["logp"]),
                                  _ptr(out["lse"]), _ptr(out["entropy"]), _ptr(out["argmax"]),
                                  _ptr(out["valid_count"]), _ptr(out["lse_ref"]), _ptr(out["kl"]),
                                  ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "grpo_score_fwd_kl")
    return out


def grpo_loss_bwd_kl(H, W, H_ref, W_ref, tokens, mask, fwd: dict, old_logp, adv,
                     ws: Workspace, eps_low=0.2, eps_high=0.2, beta=0.04, agg="seq_mean",
                     norm=0.0, out: Optional[dict] = None, stream=None) -> dict:
    """GRPO loss with the exact KL and its gradients; `fwd` is grpo_score_fwd_kl's output."""
    S, T, d = H.shape
    V = W.shape[0]
    if out is None:
        out = {"loss": torch.empty((1,), dtype=torch.float32, device=H.device),
               "dH": torch.empty_like(H),
               "dW": torch.empty((V, d), dtype=torch.float32, device=H.device)}
    st = _lib().grpo_loss_bwd_kl(_ptr(H), _ptr(W), _ptr(H_ref), _ptr(W_ref), GRPO_BF16,
                                 _ptr(tokens), _ptr(mask), S, T, d, V, _ptr(fwd["logp"]),
                                 _ptr(fwd["lse"]), _ptr(fwd["lse_ref"]), _ptr(fwd["kl"]),
                                 _ptr(old_logp), _ptr(adv), _ptr(fwd["valid_count"]),
                                 float(eps_low), float(eps_high), float(beta), AGG_MODES[agg],
                                 float(norm), _ptr(out["loss"]), _ptr(out["dH"]), _ptr(out["dW"]),
                                 ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "grpo_loss_bwd_kl")
    return out


def grpo_score_fwd_shard(H, W_shard, tokens, mask, v_offset: int, V_total: int, ws: Workspace,
                         out: Optional[dict] = None, stream=None) -> dict:
    """Statistics of one vocabulary shard: dict(stats [S,T,4] f32, zy [S,T] f32)."""
    S, T, d = H.shape
    Vs = W_shard.shape[0]
    _need(H, "H", torch.bfloat16)
    _need(W_shard, "W_shard", torch.bfloat16, (Vs, d))
    _need(tokens, "tokens", torch.int32, (S, T))
    _need(mask, "mask", torch.uint8, (S, T))
    if out is None:
        out = {"stats": torch.empty((S, T, 4), dtype=torch.float32, device=H.device),
               "zy": torch.empty((S, T), dtype=torch.float32, device=H.device)}
    st = _lib().grpo_score_fwd_shard(_ptr(H), _ptr(W_shard), GRPO_BF16, _ptr(tokens), _ptr(mask),
                                     S, T, d, Vs, int(v_offset), int(V_total), _ptr(out["stats"]),
                                     _ptr(out["zy"]), ws.ptr, ws.nbytes, _stream(stream))
    _check(st, "grpo_score_fwd_shard")
    return out


def grpo_merge_shard_stats(stats, zy, tokens, mask, V_total: int, ws: Workspace,
                           out: Optional[dict] = None, stream=None) -> dict:
    """Merge of stacked shard statistics (stats [P,S,T,4], zy [P,S,T]) into the forward outputs."""
    P, S, T = zy.shape
    _need(stats, "stats", torch.float32, (P, S, T, 4))
    _need(zy, "zy", torch.float32, (P, S, T))
    if out is None:
        f = dict(dtype=torch.float32, device=zy.device)
        out = {"logp": torch.empty((S, T), **f), "lse": torch.empty((S, T), **f),
               "entropy": torch.empty((S, T), **f),
               "argmax": torch.empty((S, T), dtype=torch.int32, device=zy.device),
               "valid_count": torch.empty((S,), dtype=torch.int32, device=zy.device)}
    st = _lib().grpo_merge_shard_stats(_ptr(stats), _ptr(zy), P, _ptr(tokens), _ptr(mask), S, T,
                                       int(V_total), _ptr(out["logp"]), _ptr(out["lse"]),
                                       _ptr(out["entropy"]), _ptr(out["argmax"]),
                                       _ptr(out["valid_count"]), ws.ptr, ws.nbytes,
                                       _stream(stream))
    _check(st, "grpo_merge_shard_stats")
    return out


def grpo_loss_bwd_shard(H, W_shard, tokens, mask, v_offset: int, V_total: int, logp, lse,
                        old_logp, ref_logp, adv, valid_count, ws: Workspace, eps_low=0.2,
                        eps_high=0.2, beta=0.04, agg="seq_mean", norm=0.0,
                        out: Optional[dict] = None, stream=None) -> dict:
    """The shard's backward: dict(loss [1], dH_partial [S,T,d] f32, dW_shard [V_shard,d] f32)."""
    S, T, d = H.shape
    Vs = W_shard.shape[0]
    if out is None:
        out = {"loss": torch.empty((1,), dtype=torch.float32, device=H.device),
               "dH_partial": torch.empty((S, T, d), dtype=torch.float32, device=H.device),
               "dW_shard": torch.empty((Vs, d), dtype=torch.float32, device=H.device)}
    st = _lib().grpo_loss_bwd_shard(_ptr(H), _ptr(W_shard), GRPO_BF16, _ptr(tokens), _ptr(mask),
                                    S, T, d, Vs, int(v_offset), int(V_total), _ptr(logp),
                                    _ptr(lse), _ptr(old_logp), _ptr(ref_logp), _ptr(adv),
                                    _ptr(valid_count), float(eps_low), float(eps_high),
                                    float(beta), AGG_MODES[agg], float(norm), _ptr(out["loss"]),
                                    _ptr(out["dH_partial"]), _ptr(out["dW_shard"]), ws.ptr,
                                    ws.nbytes, _stream(stream))
    _check(st, "grpo_loss_bwd_shard")
    return out


def grpo_last_device_error(ws: Workspace, stream=None):
    where = ctypes.c_int32(0)
    st = _lib().grpo_last_device_error(ws.ptr, ctypes.byref(where), _stream(stream))
    return int(st), int(where.value)


def grpo_status_string(status: int) -> str:
    return _lib().grpo_status_string(int(status)).decode()


def grpo_kernel_name(kid: int) -> str:
    return _lib().grpo_kernel_name(int(kid)).decode()


def grpo_timing_enable(on: bool = True):
    _check(_lib().grpo_timing_enable(1 if on else 0), "grpo_timing_enable")


def grpo_timing_reset():
    _check(_lib().grpo_timing_reset(), "grpo_timing_reset")


def grpo_timing_read(kid: int):
    n = ctypes.c_int64(0)
    ms = ctypes.c_double(0.0)
    _check(_lib().grpo_timing_read(int(kid), ctypes.byref(n), ctypes.byref(ms)), "grpo_timing_read")
    return int(n.value), float(ms.value)


def grpo_debug_inject_stall(on: bool):
    _check(_lib().grpo_debug_inject_stall(1 if on else 0), "grpo_debug_inject_stall")


def grpo_set_cta_pair(on: bool):
    _check(_lib().grpo_set_cta_pair(1 if on else 0), "grpo_set_cta_pair")


TILE_DEFAULT = -1
TILE_SINGLE, TILE_CTA_PAIR, TILE_CTA_PAIR_WIDE = 0, 1, 2
ROLE_FWD, ROLE_DZ, ROLE_DH, ROLE_DW = 0, 1, 2, 3


def grpo_set_tile_mode(mode: int):
    """Every GEMM role in one mode: 0 single-CTA 128 x 256 tiles, 1 CTA-pair 256 x 256 tiles
    (cta_group::2), 2 CTA-pair 256 x 512 tiles; -1 (TILE_DEFAULT) restores each role's
    default."""
    _check(_lib().grpo_set_tile_mode(int(mode)), "grpo_set_tile_mode")


def grpo_get_tile_mode() -> int:
    """The mode all four roles share, or -1 when they differ (as by default)."""
    return int(_lib().grpo_get_tile_mode())


def grpo_set_role_tile_mode(role: int, mode: int):
    """Tile mode of one GEMM role (ROLE_FWD, ROLE_DZ, ROLE_DH, ROLE_DW): 0, 1 or 2; -1 restores
    the role's default."""
    _check(_lib().grpo_set_role_tile_mode(int(role), int(mode)), "grpo_set_role_tile_mode")


def grpo_get_role_tile_mode(role: int) -> int:
    m = int(_lib().grpo_get_role_tile_mode(int(role)))
    if m < 0:
        raise ValueError(f"grpo_get_role_tile_mode: bad role {role}")
    return m


def grpo_set_gemm_window(check_kblocks: int, lag: int):
    """Progress window of the dH and dW GEMMs: producers stay within `lag` checkpoints of the
    launch's average, a checkpoint every `check_kblocks` k-blocks (< 0: at the start of every
    (-check_kblocks)-th work unit; 0 turns it off). Default: GEMM_WINDOW_DEFAULT."""
    _check(_lib().grpo_set_gemm_window(int(check_kblocks), int(lag)), "grpo_set_gemm_window")


def timing_table() -> dict:
    """{kernel name: (launches, total ms)} for every kernel the library has launched."""
    out = {}
    for k, name in enumerate(KERNEL_NAMES):
        n, ms = grpo_timing_read(k)
        if n:
            out[name] = (n, ms)
    return out
