"""ctypes binding of libff.so (include/ff.h, include/ff_debug.h).

Argument marshalling only: torch tensors supply device memory and the CUDA
stream; every computation runs in the library's kernels.  The functions keep
the C names.  If the library is not built, or a GPU call is made without a
CUDA device, they raise -- there is no fallback path.
"""
from __future__ import annotations

import ctypes as C
import os

from .build import LIB

FF_OK = 0
FF_SDE_SAMPLE, FF_SDE_EVAL = 0, 1
FF_LP_SUM, FF_LP_MEAN = 0, 1
FF_SCHED_FLOW_SDE, FF_SCHED_DANCE_SDE, FF_SCHED_ODE = 0, 1, 2
FF_ARCH_MMDIT, FF_ARCH_WAN = 0, 1
FF_ACT_NONE, FF_ACT_GELU, FF_ACT_SILU = 0, 1, 2
FF_TSAMPLE_UNIFORM, FF_TSAMPLE_LOGIT_NORMAL, FF_TSAMPLE_DISCRETE = 0, 1, 2
FF_AWM_SUM, FF_AWM_MEAN = 0, 1
FF_AGG_WEIGHTED_SUM, FF_AGG_PER_REWARD = 0, 1
FF_A_MK, FF_A_KM, FF_B_NK, FF_B_KN = 0, 1, 0, 1


class FFError(RuntimeError):
    def __init__(self, func: str, code: int, msg: str):
        super().__init__(f"{func} failed with status {code}: {msg}")
        self.code = code


class DitConfig(C.Structure):
    _fields_ = [("arch", C.c_int), ("hidden", C.c_int), ("heads", C.c_int), ("head_dim", C.c_int),
                ("mlp", C.c_int), ("n_double", C.c_int), ("n_single", C.c_int), ("patch_dim", C.c_int),
                ("txt_dim", C.c_int), ("n_txt", C.c_int), ("grid_f", C.c_int), ("grid_h", C.c_int),
                ("grid_w", C.c_int), ("rope_axes", C.c_int * 3), ("rope_theta", C.c_float),
                ("time_freq_dim", C.c_int)]


class TensorDesc(C.Structure):
    _fields_ = [("name", C.c_char * 64), ("offset", C.c_int64), ("ndim", C.c_int), ("shape", C.c_int64 * 2)]


_P = C.c_void_p
_I = C.c_int
_I64 = C.c_int64
_F = C.c_float
_D = C.c_double
_SZ = C.c_size_t

_SIGS = {
    "ff_last_error": ([], C.c_char_p),
    "ff_version": ([], _I),
    "ff_check_device_status": ([_P, C.POINTER(_I)], _I),
    "ff_prof_enable": ([_I], _I),
    "ff_prof_disable": ([], _I),
    "ff_prof_reset": ([], _I),
    "ff_prof_count": ([C.POINTER(_I)], _I),
    "ff_prof_read": ([_I, C.c_char_p, _I, C.POINTER(_F), C.POINTER(_D), C.POINTER(_D)], _I),
    "ff_sde_schedule": ([_I, _I, _D, _D, _D, C.POINTER(_D), C.POINTER(_D)], _I),
    "ff_sde_workspace_size": ([_I, _I64, C.POINTER(_SZ)], _I),
    "ff_sde_step_logprob": ([_I, _I64, _P, _P, _P, _P, _P, _P, _P, _I, _I, _P, _I, _P, _SZ, _P], _I),
    "ff_philox_normal": ([_I, _I64, C.c_uint64, C.c_uint32, _P, _P], _I),
    "ff_sde_step_logprob_philox": ([_I, _I64, _P, _P, _P, _P, _P, _P, C.c_uint64, C.c_uint32, _I, _P, _I, _P, _SZ,
                                    _P], _I),
    "ff_sde_step_logprob_noalloc": ([_I, _I64, _P, _P, _P, _P, _P, _P, _P, _I, _I, _P, _I, _P], _I),
    "ff_group_advantage": ([_I, _I, _P, _F, _P, _P], _I),
    "ff_grpo_loss_workspace_size": ([_I, _I, C.POINTER(_SZ)], _I),
    "ff_grpo_loss": ([_I, _I, _P, _P, _P, _F, _F, _P, _P, _P, _SZ, _P], _I),
    "ff_grpo_loss_weighted": ([_I, _I, _P, _P, _P, _P, _F, _F, _P, _P, _P, _SZ, _P], _I),
    "ff_group_advantage_multi": ([_I, _I, _I, _P, _P, _I, _F, _P, _P], _I),
    "ff_sde_schedule_window": ([_I, _I, _D, _D, _D, _I, _I, C.POINTER(_D), C.POINTER(_D)], _I),
    "ff_sample_timesteps": ([_I, _I, _P, _F, _F, _P, _I, _P, _P], _I),
    "ff_forward_process": ([_I, _I64, _P, _P, _P, _P, _P], _I),
    "ff_awm_loss_workspace_size": ([_I, _I64, C.POINTER(_SZ)], _I),
    "ff_awm_loss": ([_I, _I64, _P, _P, _P, _P, _I, _P, _P, _P, _P, _SZ, _P], _I),
    "ff_nft_loss_workspace_size": ([_I, _I64, C.POINTER(_SZ)], _I),
    "ff_nft_loss": ([_I, _I64, _P, _P, _P, _P, _P, _F, _I, _P, _P, _P, _P, _SZ, _P], _I),
    "ff_dit_weight_layout": ([C.POINTER(DitConfig), C.POINTER(TensorDesc), _I, C.POINTER(_I), C.POINTER(_I64)], _I),
    "ff_dit_create": ([C.POINTER(DitConfig), _P, C.POINTER(_P)], _I),
    "ff_dit_destroy": ([_P], _I),
    "ff_dit_workspace_size": ([_P, _I, C.POINTER(_SZ)], _I),
    "ff_dit_velocity": ([_P, _I, _P, _P, _P, _P, _P, _SZ, _P], _I),
    "ff_rollout_workspace_size": ([_P, _I, _I, C.POINTER(_SZ)], _I),
    "ff_dit_set_train_recompute": ([_P, _I], _I),
    "ff_dit_set_attention_split": ([_P, _I], _I),
    "ff_dit_train_workspace_size": ([_P, _I, C.POINTER(_SZ)], _I),
    "ff_dit_forward_train": ([_P, _I, _P, _P, _P, _P, _P, _SZ, _P], _I),
    "ff_dit_backward": ([_P, _I, _P, _P, _P, _P, _P, _SZ, _P], _I),
    "ff_sde_logprob_backward": ([_I, _I64, _P, _P, _P, _P, _P, _P, _I, _P, _I, _P, _P], _I),
    "ff_gemm": ([_I, _I, _I, _P, _I64, _I, _P, _I64, _I, _P, _I, _I, _P, _I64, _P], _I),
    "ff_attention_lse_rows": ([_I, _I], _I),
    "ff_attention_forward_workspace_size": ([_I, C.POINTER(_SZ)], _I),
    "ff_attention_forward": ([_I, _I, _I, _I, _P, _I64, _P, _I64, _I, _P, _I64, _P, _I64, _P, _P, _SZ, _P], _I),
    "ff_attention_backward_workspace_size": ([_I, _I, _I, _I, C.POINTER(_SZ)], _I),
    "ff_attention_backward": ([_I, _I, _I, _I, _P, _I64, _P, _P, _I64, _P, _I64, _I, _P, _I64, _P, _P, _I64, _P,
                               _I64, _P, _P, _SZ, _P], _I),
    "ff_cross_attention_forward": ([_I, _I, _I, _I, _P, _I64, _I, _P, _I64, _P, _I64, _P, _P], _I),
    "ff_cross_attention_backward": ([_I, _I, _I, _I, _P, _I64, _P, _P, _I64, _P, _I64, _I, _P, _I64, _P, _I64, _P,
                                     _P, _SZ, _P], _I),
    "ff_rollout": ([_P, _I, _I, _P, _P, _P, _P, _P, _P, _P, _I, _P, _SZ, _P], _I),
    "ff_rollout_philox": ([_P, _I, _I, _P, _P, _P, _P, C.c_uint64, _P, _P, _I, _P, _SZ, _P], _I),
    "ff_debug_gemm": ([_I, _I, _I, _P, _I64, _P, _I64, _P, _I, _I, _P, _I64, _P], _I),
    "ff_debug_gemm_gated": ([_I, _I, _I, _P, _I64, _P, _I64, _P, _P, _I64, _P, _I64, _I, _P], _I),
    "ff_debug_attention": ([_I, _I, _I, _I, _P, _I64, _P, _I64, _I, _P, _I64, _P, _I64, _P], _I),
    "ff_debug_attention_launch": ([_I], _I),
    "ff_debug_attention_plan": ([_I64, _I, _I, _I, _I, C.POINTER(_I), C.POINTER(_I64), C.POINTER(_I64),
                                 C.POINTER(_I64)], _I),
    "ff_debug_ln_modulate": ([_I, _I, _P, _P, _I64, _I, _I, _I, _P, _P], _I),
    "ff_debug_qk_norm_rope": ([_I, _I, _I, _I, _P, _I64, _P, _P, _I, _I, _I, C.POINTER(_I), _F, _P], _I),
    "ff_debug_reduce_chunks": ([_I, _I, _P, _P, C.POINTER(_I64), C.POINTER(_I64), C.POINTER(_I), C.POINTER(_I),
                                C.POINTER(_I), C.POINTER(_I), C.POINTER(_I64), C.POINTER(_I64), _P], _I),
}

_lib = None


def lib() -> C.CDLL:
    """The loaded libff.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"libff.so not found at {LIB}; build it with paper_2602_12529_gb300.build.build()")
        L = C.CDLL(LIB)
        for name, (args, res) in _SIGS.items():
            f = getattr(L, name)
            f.argtypes = args
            f.restype = res
        _lib = L
    return _lib


def _call(name: str, *args) -> None:
    rc = getattr(lib(), name)(*args)
    if rc != FF_OK:
        raise FFError(name, rc, lib().ff_last_error().decode())


# ----------------------------------------------------------------- helpers

def _ptr(t) -> int | None:
    """Device address of a CUDA tensor (None for None)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _stream(stream) -> int:
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return s.cuda_stream


def _ptr_rows(t) -> int | None:
    """Device address of a CUDA matrix whose rows are contiguous (any row
    pitch, passed on as the leading dimension)."""
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if t.dim() != 2 or t.stride(1) != 1:
        raise ValueError("expected a 2-D tensor with contiguous rows")
    return t.data_ptr()


def _check(t, dtype, name):
    if t.dtype != dtype:
        raise TypeError(f"{name}: expected {dtype}, got {t.dtype}")


def _need(t, n: int, name: str):
    """Raise unless tensor t holds at least n elements (the kernels index
    that far; a shorter buffer would be read or written past its end)."""
    if t.numel() < n:
        raise ValueError(f"{name}: {t.numel()} elements, the call touches {n}")


def _rows(t, rows: int, cols: int, name: str):
    """Raise unless t (row pitch t.shape[-1]) holds `rows` rows of at least
    `cols` columns: the attention kernels address row r at r * pitch."""
    if rows <= 0:
        return
    if t is None:
        raise ValueError(f"{name}: missing, {rows} rows needed")
    if t.dim() < 2 or t.shape[-1] < cols or t.numel() // t.shape[-1] < rows:
        raise ValueError(f"{name}: shape {tuple(t.shape)}, the call touches {rows} rows of {cols} columns")


def _sde_args(x_t, v, eps, x_next, t, t_next, sigma, logp, ld, need_eps):
    """dtype and size checks shared by the SDE step wrappers: [B, D] arrays,
    [B] times and sigmas, logp read at b * ld."""
    import torch
    B = x_t.shape[0]
    D = x_t.numel() // B
    arrays = [("x_t", x_t), ("v", v), ("x_next", x_next)] + ([("eps", eps)] if need_eps else [])
    for n_, a in arrays:
        _check(a, torch.float32, n_)
        _need(a, B * D, n_)
    for n_, a in (("t", t), ("t_next", t_next), ("sigma", sigma)):
        _check(a, torch.float32, n_)
        _need(a, B, n_)
    _check(logp, torch.float32, "logp")
    if ld < 1:
        raise ValueError("ld must be >= 1")
    _need(logp, (B - 1) * ld + 1, "logp")
    return B, D


# ------------------------------------------------------------ host queries

def ff_version() -> int:
    return lib().ff_version()


def ff_sde_schedule(kind: int, n_steps: int, shift: float = 1.0, eta: float = 0.7, t_clamp: float = 0.96):
    """Host-only: (t[0..S], sigma[0..S-1]) as Python lists of float."""
    t = (_D * (n_steps + 1))()
    s = (_D * n_steps)()
    _call("ff_sde_schedule", kind, n_steps, shift, eta, t_clamp, t, s)
    return list(t), list(s)


def ff_sde_schedule_window(kind: int, n_steps: int, shift: float, eta: float, t_clamp: float, start: int,
                           length: int):
    """Host-only MixGRPO schedule: sigma zero outside steps [start, start + length)."""
    t = (_D * (n_steps + 1))()
    s = (_D * n_steps)()
    _call("ff_sde_schedule_window", kind, n_steps, shift, eta, t_clamp, start, length, t, s)
    return list(t), list(s)


def ff_sde_workspace_size(B: int, D: int) -> int:
    n = _SZ()
    _call("ff_sde_workspace_size", B, D, C.byref(n))
    return n.value


def ff_grpo_loss_workspace_size(B: int, T: int) -> int:
    n = _SZ()
    _call("ff_grpo_loss_workspace_size", B, T, C.byref(n))
    return n.value


def make_config(cfg: dict) -> DitConfig:
    c = DitConfig()
    c.arch = FF_ARCH_WAN if cfg.get("arch", "mmdit") == "wan" else FF_ARCH_MMDIT
    for k in ("hidden", "heads", "head_dim", "mlp", "n_double", "n_single", "patch_dim", "txt_dim", "n_txt",
              "time_freq_dim"):
        setattr(c, k, int(cfg[k]))
    c.grid_f, c.grid_h, c.grid_w = (int(v) for v in cfg["grid"])
    for i, a in enumerate(cfg["rope_axes"]):
        c.rope_axes[i] = int(a)
    c.rope_theta = float(cfg["rope_theta"])
    return c


def ff_dit_weight_layout(cfg: dict):
    """[(name, offset_elems, shape)], total_elems for a workload dict."""
    c = make_config(cfg)
    n = _I()
    total = _I64()
    _call("ff_dit_weight_layout", C.byref(c), None, 0, C.byref(n), C.byref(total))
    descs = (TensorDesc * n.value)()
    _call("ff_dit_weight_layout", C.byref(c), descs, n.value, C.byref(n), C.byref(total))
    out = []
    for d in descs:
        shape = (d.shape[0], d.shape[1]) if d.ndim == 2 else (d.shape[0],)
        out.append((d.name.decode(), int(d.offset), shape))
    return out, int(total.value)


# --------------------------------------------------------------- GPU calls

def ff_sde_step_logprob(x_t, v, eps, x_next, t, t_next, sigma, logp, mode=FF_SDE_SAMPLE, reduce=FF_LP_SUM,
                        ld=1, ws=None, stream=None):
    import torch
    B, D = _sde_args(x_t, v, eps, x_next, t, t_next, sigma, logp, ld, mode == FF_SDE_SAMPLE)
    if ws is None:
        ws = torch.zeros(ff_sde_workspace_size(B, D), dtype=torch.uint8, device=x_t.device)
    _call("ff_sde_step_logprob", B, D, _ptr(x_t), _ptr(v), _ptr(eps), _ptr(x_next), _ptr(t), _ptr(t_next),
          _ptr(sigma), mode, reduce, _ptr(logp), ld, _ptr(ws), ws.numel(), _stream(stream))


def ff_philox_normal(out, seed: int, rng_stream: int, stream=None):
    """out [B, ...] fp32 (device) = the counter-based standard normals of
    (seed, rng_stream), sample b = row b (include/ff.h)."""
    import torch
    _check(out, torch.float32, "out")
    B = out.shape[0]
    _call("ff_philox_normal", B, out.numel() // B, int(seed), int(rng_stream), _ptr(out), _stream(stream))


def ff_sde_step_logprob_philox(x_t, v, x_next, t, t_next, sigma, logp, seed: int, rng_stream: int,
                               reduce=FF_LP_SUM, ld=1, ws=None, stream=None):
    """The SAMPLE step with eps drawn in the kernel (ff_philox_normal's values)."""
    import torch
    B, D = _sde_args(x_t, v, None, x_next, t, t_next, sigma, logp, ld, False)
    if ws is None:
        ws = torch.zeros(ff_sde_workspace_size(B, D), dtype=torch.uint8, device=x_t.device)
    _call("ff_sde_step_logprob_philox", B, D, _ptr(x_t), _ptr(v), _ptr(x_next), _ptr(t), _ptr(t_next), _ptr(sigma),
          int(seed), int(rng_stream), reduce, _ptr(logp), ld, _ptr(ws), ws.numel(), _stream(stream))


def ff_sde_step_logprob_noalloc(x_t, v, eps, x_next, t, t_next, sigma, logp, mode=FF_SDE_SAMPLE,
                                reduce=FF_LP_SUM, ld=1, stream=None):
    """ff_sde_step_logprob without a workspace: scratch is the library's own
    fixed device array (for callers that cannot allocate device memory)."""
    B, D = _sde_args(x_t, v, eps, x_next, t, t_next, sigma, logp, ld, mode == FF_SDE_SAMPLE)
    _call("ff_sde_step_logprob_noalloc", B, D, _ptr(x_t), _ptr(v), _ptr(eps), _ptr(x_next), _ptr(t), _ptr(t_next),
          _ptr(sigma), mode, reduce, _ptr(logp), ld, _stream(stream))


def ff_sde_logprob_backward(x_t, v, x_next, t, t_next, sigma, grad_logp, grad_v, reduce=FF_LP_SUM, ld: int = 1,
                            stream=None):
    """grad_v = d logp / d v (x_next fixed) times grad_logp[b * ld]."""
    import torch
    B, D = _sde_args(x_t, v, None, x_next, t, t_next, sigma, grad_logp, ld, False)
    _check(grad_v, torch.float32, "grad_v")
    _need(grad_v, B * D, "grad_v")
    _call("ff_sde_logprob_backward", B, D, _ptr(x_t), _ptr(v), _ptr(x_next), _ptr(t), _ptr(t_next), _ptr(sigma),
          reduce, _ptr(grad_logp), ld, _ptr(grad_v), _stream(stream))


def ff_group_advantage(rewards, G: int, eps_A: float, adv, stream=None):
    import torch
    _check(rewards, torch.float32, "rewards")
    _check(adv, torch.float32, "adv")
    n = rewards.numel()
    if n % G:
        raise ValueError("rewards.numel() must be a multiple of G")
    _need(adv, n, "adv")
    _call("ff_group_advantage", n // G, G, _ptr(rewards), eps_A, _ptr(adv), _stream(stream))


def _loss_sizes(B, T, lp_old, adv, loss, grad):
    import torch
    _need(lp_old, B * T, "lp_old")
    _need(adv, B, "adv")
    _need(loss, 1, "loss")
    if grad is not None:
        _check(grad, torch.float32, "grad_lp_new")
        _need(grad, B * T, "grad_lp_new")


def ff_grpo_loss(lp_new, lp_old, adv, clip_lo: float, clip_hi: float, loss, grad_lp_new=None, ws=None,
                 stream=None):
    import torch
    B, T = lp_new.shape
    for n_, a in (("lp_new", lp_new), ("lp_old", lp_old), ("adv", adv), ("loss", loss)):
        _check(a, torch.float32, n_)
    _loss_sizes(B, T, lp_old, adv, loss, grad_lp_new)
    if ws is None:
        ws = torch.zeros(ff_grpo_loss_workspace_size(B, T), dtype=torch.uint8, device=lp_new.device)
    _call("ff_grpo_loss", B, T, _ptr(lp_new), _ptr(lp_old), _ptr(adv), clip_lo, clip_hi, _ptr(loss),
          _ptr(grad_lp_new), _ptr(ws), ws.numel(), _stream(stream))


def ff_grpo_loss_weighted(lp_new, lp_old, adv, step_w, clip_lo: float, clip_hi: float, loss, grad_lp_new=None,
                          ws=None, stream=None):
    import torch
    B, T = lp_new.shape
    for n_, a in (("lp_new", lp_new), ("lp_old", lp_old), ("adv", adv), ("step_w", step_w), ("loss", loss)):
        _check(a, torch.float32, n_)
    _loss_sizes(B, T, lp_old, adv, loss, grad_lp_new)
    _need(step_w, T, "step_w")
    if ws is None:
        ws = torch.zeros(ff_grpo_loss_workspace_size(B, T), dtype=torch.uint8, device=lp_new.device)
    _call("ff_grpo_loss_weighted", B, T, _ptr(lp_new), _ptr(lp_old), _ptr(adv), _ptr(step_w), clip_lo, clip_hi,
          _ptr(loss), _ptr(grad_lp_new), _ptr(ws), ws.numel(), _stream(stream))


def ff_group_advantage_multi(rewards, G: int, weights, mode: int, eps_A: float, adv, stream=None):
    """rewards: [N, K] fp32 (N a multiple of G); weights: [K] fp32; adv: [N] fp32."""
    import torch
    for n_, a in (("rewards", rewards), ("weights", weights), ("adv", adv)):
        _check(a, torch.float32, n_)
    N, K = rewards.shape
    if N % G:
        raise ValueError("rewards.shape[0] must be a multiple of G")
    _call("ff_group_advantage_multi", N // G, G, K, _ptr(rewards), _ptr(weights), mode, eps_A, _ptr(adv),
          _stream(stream))


def ff_sample_timesteps(mode: int, draw, p0: float, p1: float, t_out, grid=None, stream=None):
    import torch
    _check(draw, torch.float32, "draw")
    _check(t_out, torch.float32, "t_out")
    _call("ff_sample_timesteps", mode, draw.numel(), _ptr(draw), p0, p1, _ptr(grid),
          0 if grid is None else grid.numel(), _ptr(t_out), _stream(stream))


def ff_forward_process(x0, eps, t, x_t, stream=None):
    import torch
    for n_, a in (("x0", x0), ("eps", eps), ("t", t), ("x_t", x_t)):
        _check(a, torch.float32, n_)
    B = x0.shape[0]
    for n_, a in (("eps", eps), ("x_t", x_t)):
        _need(a, x0.numel(), n_)
    _need(t, B, "t")
    _call("ff_forward_process", B, x0.numel() // B, _ptr(x0), _ptr(eps), _ptr(t), _ptr(x_t), _stream(stream))


def ff_awm_loss_workspace_size(B: int, D: int) -> int:
    n = _SZ()
    _call("ff_awm_loss_workspace_size", B, D, C.byref(n))
    return n.value


def ff_nft_loss_workspace_size(B: int, D: int) -> int:
    n = _SZ()
    _call("ff_nft_loss_workspace_size", B, D, C.byref(n))
    return n.value


def ff_nft_loss(v, v_old, eps, x0, r, beta: float, reduce: int, loss, grad_v=None, err=None, ws=None, stream=None):
    """DiffusionNFT loss (Eq. 2); err: [B, 2] or None."""
    import torch
    for n_, a in (("v", v), ("v_old", v_old), ("eps", eps), ("x0", x0), ("r", r), ("loss", loss)):
        _check(a, torch.float32, n_)
    B = v.shape[0]
    D = v.numel() // B
    for n_, a in (("v_old", v_old), ("eps", eps), ("x0", x0)) + ((("grad_v", grad_v),) if grad_v is not None else ()):
        _need(a, B * D, n_)
    _need(r, B, "r")
    if err is not None:
        _need(err, 2 * B, "err")
    if ws is None:
        ws = torch.empty(ff_nft_loss_workspace_size(B, D), dtype=torch.uint8, device=v.device)
    _call("ff_nft_loss", B, D, _ptr(v), _ptr(v_old), _ptr(eps), _ptr(x0), _ptr(r), beta, reduce, _ptr(loss),
          _ptr(grad_v), _ptr(err), _ptr(ws), ws.numel(), _stream(stream))


def ff_awm_loss(v, eps, x0, adv, reduce: int, loss, grad_v=None, err=None, ws=None, stream=None):
    import torch
    for n_, a in (("v", v), ("eps", eps), ("x0", x0), ("adv", adv), ("loss", loss)):
        _check(a, torch.float32, n_)
    B = v.shape[0]
    D = v.numel() // B
    for n_, a in (("eps", eps), ("x0", x0)) + ((("grad_v", grad_v),) if grad_v is not None else ()):
        _need(a, B * D, n_)
    _need(adv, B, "adv")
    if err is not None:
        _need(err, B, "err")
    if ws is None:
        ws = torch.empty(ff_awm_loss_workspace_size(B, D), dtype=torch.uint8, device=v.device)
    _call("ff_awm_loss", B, D, _ptr(v), _ptr(eps), _ptr(x0), _ptr(adv), reduce, _ptr(loss), _ptr(grad_v),
          _ptr(err), _ptr(ws), ws.numel(), _stream(stream))


class Dit:
    """Handle of a DiT over a caller-owned bf16 weight blob (torch tensor)."""

    def __init__(self, cfg: dict, blob):
        self.cfg = dict(cfg)
        self._c = make_config(cfg)
        self.blob = blob
        h = _P()
        _call("ff_dit_create", C.byref(self._c), _ptr(blob), C.byref(h))
        self._h = h

    def close(self):
        if self._h is not None and self._h.value:
            lib().ff_dit_destroy(self._h)
        self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def workspace_size(self, B: int) -> int:
        n = _SZ()
        _call("ff_dit_workspace_size", self._h, B, C.byref(n))
        return n.value

    def ff_dit_velocity(self, x_t, txt, t, v_out, ws, stream=None):
        import torch
        _check(x_t, torch.float32, "x_t")
        _check(txt, torch.bfloat16, "txt")
        _check(t, torch.float32, "t")
        _check(v_out, torch.float32, "v_out")
        B = x_t.shape[0]
        _call("ff_dit_velocity", self._h, B, _ptr(x_t), _ptr(txt), _ptr(t), _ptr(v_out), _ptr(ws), ws.numel(),
              _stream(stream))

    def train_workspace_size(self, B: int) -> int:
        n = _SZ()
        _call("ff_dit_train_workspace_size", self._h, B, C.byref(n))
        return n.value

    def ff_dit_forward_train(self, x_t, txt, t, v_out, ws, stream=None):
        import torch
        _check(x_t, torch.float32, "x_t")
        _check(txt, torch.bfloat16, "txt")
        _check(t, torch.float32, "t")
        _check(v_out, torch.float32, "v_out")
        B = x_t.shape[0]
        _call("ff_dit_forward_train", self._h, B, _ptr(x_t), _ptr(txt), _ptr(t), _ptr(v_out), _ptr(ws), ws.numel(),
              _stream(stream))

    def ff_dit_backward(self, txt, dv, grad, ws, dx_t=None, stream=None):
        """grad: fp32 blob of the weight layout's total_elems elements."""
        import torch
        _check(txt, torch.bfloat16, "txt")
        _check(dv, torch.float32, "dv")
        _check(grad, torch.float32, "grad")
        if dx_t is not None:
            _check(dx_t, torch.float32, "dx_t")
        B = dv.shape[0]
        _call("ff_dit_backward", self._h, B, _ptr(txt), _ptr(dv), _ptr(grad), _ptr(dx_t), _ptr(ws), ws.numel(),
              _stream(stream))

    def set_train_recompute(self, on):
        """Training pass keeps the block inputs (and, for True or 1, the attention outputs; 2: the inputs
        only) and re-runs each block in the backward."""
        mode = (1 if on else 0) if isinstance(on, bool) else int(on)
        _call("ff_dit_set_train_recompute", self._h, mode)

    def set_attention_split(self, on: bool):
        """Attention launches may split their last round's query blocks (True, the default); False makes
        every sample's results independent of the rest of the batch, bit for bit."""
        _call("ff_dit_set_attention_split", self._h, 1 if on else 0)

    def rollout_workspace_size(self, B: int, S: int) -> int:
        n = _SZ()
        _call("ff_rollout_workspace_size", self._h, B, S, C.byref(n))
        return n.value

    def ff_rollout(self, x, txt, t, sigma, eps, logp, traj=None, reduce: int = FF_LP_SUM, ws=None, stream=None):
        """x [B, ...] updated in place; t [S+1], sigma [S]; eps [S, B, ...];
        logp [B, S]; traj [S+1, B, ...] or None."""
        import torch
        for n_, a in (("x", x), ("t", t), ("sigma", sigma), ("eps", eps), ("logp", logp)):
            _check(a, torch.float32, n_)
        _check(txt, torch.bfloat16, "txt")
        B, S = x.shape[0], sigma.numel()
        if ws is None:
            ws = torch.empty(self.rollout_workspace_size(B, S), dtype=torch.uint8, device=x.device)
        _call("ff_rollout", self._h, B, S, _ptr(x), _ptr(txt), _ptr(t), _ptr(sigma), _ptr(eps), _ptr(traj),
              _ptr(logp), reduce, _ptr(ws), ws.numel(), _stream(stream))

    def ff_rollout_philox(self, x, txt, t, sigma, seed: int, logp, traj=None, reduce: int = FF_LP_SUM, ws=None,
                          stream=None):
        """ff_rollout with step k's noise drawn on the device from (seed, k)."""
        import torch
        for n_, a in (("x", x), ("t", t), ("sigma", sigma), ("logp", logp)):
            _check(a, torch.float32, n_)
        _check(txt, torch.bfloat16, "txt")
        B, S = x.shape[0], sigma.numel()
        if ws is None:
            ws = torch.empty(self.rollout_workspace_size(B, S), dtype=torch.uint8, device=x.device)
        _call("ff_rollout_philox", self._h, B, S, _ptr(x), _ptr(txt), _ptr(t), _ptr(sigma), int(seed), _ptr(traj),
              _ptr(logp), reduce, _ptr(ws), ws.numel(), _stream(stream))


def ff_check_device_status(stream=None) -> int:
    st = _I()
    rc = lib().ff_check_device_status(_stream(stream), C.byref(st))
    if rc not in (FF_OK, 5):
        raise FFError("ff_check_device_status", rc, lib().ff_last_error().decode())
    return st.value


# ------------------------------------------------------------ launch timing

def ff_prof_enable(max_records: int) -> None:
    _call("ff_prof_enable", max_records)


def ff_prof_disable() -> None:
    _call("ff_prof_disable")


def ff_prof_reset() -> None:
    _call("ff_prof_reset")


def ff_prof_records():
    """[(kernel name, ms, algorithmic flops, algorithmic bytes)] of the timed launches."""
    n = _I()
    _call("ff_prof_count", C.byref(n))
    out = []
    buf = C.create_string_buffer(64)
    for i in range(n.value):
        ms, fl, by = _F(), _D(), _D()
        _call("ff_prof_read", i, buf, 64, C.byref(ms), C.byref(fl), C.byref(by))
        out.append((buf.value.decode(), float(ms.value), float(fl.value), float(by.value)))
    return out


# ------------------------------------------------------------- debug hooks

def ff_debug_gemm(A, B, bias, out, act=FF_ACT_NONE, stream=None):
    M, K = A.shape
    N = B.shape[0]
    import torch
    _call("ff_debug_gemm", M, N, K, _ptr(A), A.stride(0), _ptr(B), B.stride(0), _ptr(bias), act,
          1 if out.dtype == torch.float32 else 0, _ptr(out), out.stride(0), _stream(stream))


def ff_gemm(A, a_layout: int, B, b_layout: int, out, bias=None, act=FF_ACT_NONE, stream=None):
    """out[M, N] = act(op(A) op(B) + bias) with the stored layouts of include/ff.h."""
    import torch
    M = A.shape[0] if a_layout == FF_A_MK else A.shape[1]
    K = A.shape[1] if a_layout == FF_A_MK else A.shape[0]
    N = B.shape[0] if b_layout == FF_B_NK else B.shape[1]
    _call("ff_gemm", M, N, K, _ptr_rows(A), A.stride(0), a_layout, _ptr_rows(B), B.stride(0), b_layout, _ptr(bias),
          act, 1 if out.dtype == torch.float32 else 0, _ptr_rows(out), out.stride(0), _stream(stream))


def ff_attention_forward_workspace_size(head_dim: int) -> int:
    n = _SZ()
    _call("ff_attention_forward_workspace_size", head_dim, C.byref(n))
    return n.value


def ff_attention_forward(B, heads, head_dim, qkv0, out0, n0, qkv1, out1, n1, lse=None, ws=None, stream=None):
    """Joint attention over [segment 0; segment 1]; lse: [B, heads, ff_attention_lse_rows(n0, n1)] fp32 or None.
    ws: the optional scratch that lets the launch split its last round's items (None: a fresh one of
    ff_attention_forward_workspace_size bytes; False: none, the unsplit launch)."""
    import torch
    H = heads * head_dim
    for n_, q_, o_, tag in ((n0, qkv0, out0, "0"), (n1, qkv1, out1, "1")):
        _rows(q_, B * n_, 3 * H, "qkv" + tag)
        _rows(o_, B * n_, H, "out" + tag)
        if n_ > 0:
            _check(q_, torch.bfloat16, "qkv" + tag)
            _check(o_, torch.bfloat16, "out" + tag)
    if lse is not None:
        _check(lse, torch.float32, "lse")
        _need(lse, B * heads * lib().ff_attention_lse_rows(n0, n1), "lse")
    if ws is None:
        dev = (qkv0 if n0 else qkv1).device
        ws = torch.empty(ff_attention_forward_workspace_size(head_dim), dtype=torch.uint8, device=dev)
    elif ws is False:
        ws = None
    _call("ff_attention_forward", B, heads, head_dim, n0, _ptr(qkv0), qkv0.shape[-1], _ptr(out0), out0.shape[-1],
          n1, _ptr(qkv1), qkv1.shape[-1], _ptr(out1), out1.shape[-1], _ptr(lse), _ptr(ws),
          0 if ws is None else ws.numel(), _stream(stream))


def ff_attention_backward(B, heads, head_dim, seg0, seg1, lse, ws=None, stream=None):
    """seg = (n, qkv, out, dout, dqkv) per segment; writes dq, dk, dv into dqkv."""
    import torch
    n0, q0, o0, g0, d0 = seg0
    n1, q1, o1, g1, d1 = seg1
    H = heads * head_dim
    for n_, q_, o_, g_, d_, tag in ((n0, q0, o0, g0, d0, "0"), (n1, q1, o1, g1, d1, "1")):
        _rows(q_, B * n_, 3 * H, "qkv" + tag)
        _rows(o_, B * n_, H, "out" + tag)
        _rows(g_, B * n_, H, "dout" + tag)
        _rows(d_, B * n_, 3 * H, "dqkv" + tag)
        if n_ > 0 and g_ is not None and o_ is not None and g_.shape[-1] != o_.shape[-1]:
            raise ValueError(f"dout{tag} and out{tag} share one row pitch")
    _need(lse, B * heads * lib().ff_attention_lse_rows(n0, n1), "lse")
    if ws is None:
        sz = _SZ()
        _call("ff_attention_backward_workspace_size", B, heads, n0, n1, C.byref(sz))
        ws = torch.empty(sz.value, dtype=torch.uint8, device=lse.device)
    _call("ff_attention_backward", B, heads, head_dim, n0, _ptr(q0), q0.shape[-1], _ptr(o0), _ptr(g0),
          o0.shape[-1], _ptr(d0), d0.shape[-1], n1, _ptr(q1), q1.shape[-1], _ptr(o1), _ptr(g1), o1.shape[-1],
          _ptr(d1), d1.shape[-1], _ptr(lse), _ptr(ws), ws.numel(), _stream(stream))


def ff_cross_attention_forward(B, heads, head_dim, q, nq, kv, nk, out, lse=None, stream=None):
    """Cross-attention: q [B nq, >= H] (q at columns h d), kv [B nk, >= 2H] (k at
    h d, v at H + h d), out [B nq, >= H]; lse [B, heads, ff_attention_lse_rows(nq, 0)] or None."""
    H = heads * head_dim
    _rows(q, B * nq, H, "q")
    _rows(kv, B * nk, 2 * H, "kv")
    _rows(out, B * nq, H, "out")
    if lse is not None:
        _need(lse, B * heads * lib().ff_attention_lse_rows(nq, 0), "lse")
    _call("ff_cross_attention_forward", B, heads, head_dim, nq, _ptr(q), q.shape[-1], nk, _ptr(kv), kv.shape[-1],
          _ptr(out), out.shape[-1], _ptr(lse), _stream(stream))


def ff_cross_attention_backward(B, heads, head_dim, q, nq, out, dout, dq, kv, nk, dkv, lse, ws=None, stream=None):
    """Writes dq (like q) and dk | dv (like kv) from dO (like out) and the forward's lse."""
    import torch
    H = heads * head_dim
    _rows(q, B * nq, H, "q")
    _rows(out, B * nq, H, "out")
    _rows(dout, B * nq, H, "dout")
    _rows(dq, B * nq, H, "dq")
    _rows(kv, B * nk, 2 * H, "kv")
    _rows(dkv, B * nk, 2 * H, "dkv")
    if dout.shape[-1] != out.shape[-1]:
        raise ValueError("dout and out share one row pitch")
    _need(lse, B * heads * lib().ff_attention_lse_rows(nq, 0), "lse")
    if ws is None:
        sz = _SZ()
        _call("ff_attention_backward_workspace_size", B, heads, nq, 0, C.byref(sz))
        ws = torch.empty(sz.value, dtype=torch.uint8, device=lse.device)
    _call("ff_cross_attention_backward", B, heads, head_dim, nq, _ptr(q), q.shape[-1], _ptr(out), _ptr(dout),
          out.shape[-1], _ptr(dq), dq.shape[-1], nk, _ptr(kv), kv.shape[-1], _ptr(dkv), dkv.shape[-1], _ptr(lse),
          _ptr(ws), ws.numel(), _stream(stream))


def ff_debug_gemm_gated(A, B, bias, resid, gate, rows_per_sample, stream=None):
    M, K = A.shape
    N = B.shape[0]
    _call("ff_debug_gemm_gated", M, N, K, _ptr(A), A.stride(0), _ptr(B), B.stride(0), _ptr(bias), _ptr(resid),
          resid.stride(0), _ptr(gate), gate.stride(0), rows_per_sample, _stream(stream))


def ff_debug_attention(B, heads, head_dim, qkv0, out0, n0, qkv1, out1, n1, stream=None):
    H = heads * head_dim
    for n_, q_, o_, tag in ((n0, qkv0, out0, "0"), (n1, qkv1, out1, "1")):
        _rows(q_, B * n_, 3 * H, "qkv" + tag)
        _rows(o_, B * n_, H, "out" + tag)
    _call("ff_debug_attention", B, heads, head_dim, n0, _ptr(qkv0), qkv0.shape[-1], _ptr(out0), out0.shape[-1],
          n1, _ptr(qkv1), qkv1.shape[-1], _ptr(out1), out1.shape[-1], _stream(stream))


def ff_debug_ln_modulate(x, mods, shift_off, scale_off, tokens_per_sample, out, stream=None):
    rows, H = x.shape
    _call("ff_debug_ln_modulate", rows, H, _ptr(x), _ptr(mods), mods.shape[-1], shift_off, scale_off,
          tokens_per_sample, _ptr(out), _stream(stream))


def ff_debug_reduce_chunks(part, out, jobs, B, stream=None):
    """jobs: dicts with part_off, ld_part, ncols, spans [(first, count), ...
    up to 2], per_sample, out_off, ld_out (offsets in floats from part and
    out, both fp32 device tensors)."""
    n = len(jobs)
    arr = lambda t, vals: (t * max(n, 1))(*vals)
    spans = [list(j["spans"]) + [(0, 0)] * (2 - len(j["spans"])) for j in jobs]
    first = (_I * max(2 * n, 2))(*[f for sp in spans for f, _ in sp])
    count = (_I * max(2 * n, 2))(*[c for sp in spans for _, c in sp])
    _call("ff_debug_reduce_chunks", n, B, _ptr(part), _ptr(out), arr(_I64, [j["part_off"] for j in jobs]),
          arr(_I64, [j["ld_part"] for j in jobs]), arr(_I, [j["ncols"] for j in jobs]), first, count,
          arr(_I, [int(bool(j["per_sample"])) for j in jobs]), arr(_I64, [j["out_off"] for j in jobs]),
          arr(_I64, [j["ld_out"] for j in jobs]), _stream(stream))


def ff_debug_qk_norm_rope(qkv, rows_txt, heads, head_dim, q_scale, k_scale, grid, rope_axes, theta, stream=None):
    axes = (_I * 3)(*rope_axes)
    _call("ff_debug_qk_norm_rope", qkv.shape[0], rows_txt, heads, head_dim, _ptr(qkv), qkv.shape[-1],
          _ptr(q_scale), _ptr(k_scale), grid[0], grid[1], grid[2], axes, theta, _stream(stream))

