"""Seeded synthetic inputs shared by the oracle, the tests and the benchmark.

This module holds no arithmetic of the method: it only draws random numbers
(numpy ``default_rng``), rounds them to the storage types the path consumes
(bf16 bit patterns, fp32) and names the workload shapes.  Both sides of every
parity check (the fp64 oracle under ``oracle/`` and the CUDA path) read their
inputs from here, so they see bit-identical data.

Workloads are synthetic stand-ins for the paper's FLUX.1-dev / Qwen-Image / WAN
runs (Sec. 4.1 names FLUX.1-dev with PickScore; Sec. 1 names Flux, Qwen-Image
and WAN).  No weights, prompts or reward models exist here, so weights are
random-init N(0, 0.02), text embeddings and the initial latent are N(0, 1),
rewards are U(0, 1).
"""
from __future__ import annotations

import zlib

import numpy as np

# ---------------------------------------------------------------------------
# Workload shapes.  Keys mirror the C struct ``ff_dit_config`` plus rollout
# parameters.  grid = (frames, rows, cols) of latent patch tokens.
# ---------------------------------------------------------------------------

_MMDIT_TINY = dict(
    name="tiny_mmdit", arch="mmdit", hidden=256, heads=4, head_dim=64, mlp=1024,
    n_double=2, n_single=0, patch_dim=64, txt_dim=256, n_txt=32, grid=(1, 8, 8),
    rope_axes=(8, 28, 28), rope_theta=10000.0, time_freq_dim=256,
    batch=4, group=4, sde_steps=4, steps_run=4, grid_kind="linear", shift=1.0,
    eta=0.7, t_clamp=0.96, clip=0.2, eps_adv=1e-4,
)

_FLUX_BLOCK = dict(
    name="flux_double_block", arch="mmdit", hidden=3072, heads=24, head_dim=128,
    mlp=12288, n_double=1, n_single=0, patch_dim=64, txt_dim=4096, n_txt=512,
    grid=(1, 64, 64), rope_axes=(16, 56, 56), rope_theta=10000.0,
    time_freq_dim=256, batch=4, group=4, sde_steps=10, steps_run=1,
    grid_kind="shifted", shift=3.0, eta=0.7, t_clamp=0.96, clip=0.2, eps_adv=1e-4,
)

_FLUX_REDUCED = dict(
    _FLUX_BLOCK, name="flux_8d16s", n_double=8, n_single=16, grid=(1, 32, 32),
    batch=32, group=16, sde_steps=10, steps_run=10,
)

_QWEN_IMAGE = dict(
    _FLUX_BLOCK, name="qwen_image_60d", n_double=60, n_txt=256, txt_dim=3584,
    grid=(1, 64, 64), batch=4, group=4, steps_run=1,
)

_WAN = dict(
    name="wan_40", arch="wan", hidden=5120, heads=40, head_dim=128, mlp=13824,
    n_double=40, n_single=0, patch_dim=64, txt_dim=4096, n_txt=512,
    grid=(21, 30, 52), rope_axes=(44, 42, 42), rope_theta=10000.0,
    time_freq_dim=256, batch=1, group=8, sde_steps=10, steps_run=2,
    grid_kind="shifted", shift=3.0, eta=0.7, t_clamp=0.96, clip=0.2, eps_adv=1e-4,
)

CONFIGS = {c["name"]: c for c in (_MMDIT_TINY, _FLUX_BLOCK, _FLUX_REDUCED, _QWEN_IMAGE, _WAN)}


def config(name: str, **overrides) -> dict:
    """A copy of a named workload with fields overridden (for small test cases)."""
    c = dict(CONFIGS[name])
    c.update(overrides)
    return c


def n_img(cfg: dict) -> int:
    f, h, w = cfg["grid"]
    return f * h * w


# ---------------------------------------------------------------------------
# Storage-type helpers (rounding only, no method arithmetic).
# ---------------------------------------------------------------------------

def bf16_bits(x) -> np.ndarray:
    """Round float32 values to bf16 (round-to-nearest-even), return uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = ((u >> 16) & 1) + np.uint32(0x7FFF)
    return ((u + rounding) >> 16).astype(np.uint16)


def bf16_value(bits) -> np.ndarray:
    """Exact float32 value of bf16 bit patterns."""
    b = np.ascontiguousarray(bits, dtype=np.uint16)
    return (b.astype(np.uint32) << 16).view(np.float32)


def _rng(seed: int, tag: str) -> np.random.Generator:
    return np.random.default_rng([int(seed), zlib.crc32(tag.encode())])


# ---------------------------------------------------------------------------
# Weights.  Every tensor is drawn from its own stream keyed by (seed, name), so
# any subset of a model can be regenerated on either side without the rest.
# kind: "matrix" -> N(0, std); "bias" -> N(0, bias_std) (0 by default);
#       "scale" -> 1 + N(0, scale_std) (1 by default).
# ---------------------------------------------------------------------------

def weight(name: str, shape, kind: str, seed: int = 0, std: float = 0.02,
           bias_std: float = 0.0, scale_std: float = 0.0) -> np.ndarray:
    """bf16 bit pattern (uint16) of one named parameter tensor."""
    shape = tuple(int(s) for s in shape)
    n = int(np.prod(shape)) if shape else 1
    if kind == "matrix":
        v = _rng(seed, name).standard_normal(n, dtype=np.float32) * np.float32(std)
    elif kind == "bias":
        if bias_std == 0.0:
            v = np.zeros(n, np.float32)
        else:
            v = _rng(seed, name).standard_normal(n, dtype=np.float32) * np.float32(bias_std)
    elif kind == "scale":
        v = np.ones(n, np.float32)
        if scale_std != 0.0:
            v += _rng(seed, name).standard_normal(n, dtype=np.float32) * np.float32(scale_std)
    else:
        raise ValueError(f"unknown weight kind {kind!r}")
    return bf16_bits(v).reshape(shape)


def weight_kind(name: str) -> str:
    """Kind of a parameter from its name: '*.b' bias, '*.scale' norm scale, else matrix."""
    if name.endswith(".b"):
        return "bias"
    if name.endswith(".scale"):
        return "scale"
    return "matrix"


def weights(specs, seed: int = 0, std: float = 0.02, bias_std: float = 0.0,
            scale_std: float = 0.0) -> dict:
    """{name: bf16 bits} for an iterable of (name, shape)."""
    return {n: weight(n, s, weight_kind(n), seed, std, bias_std, scale_std) for n, s in specs}


# ---------------------------------------------------------------------------
# Activations and rollout randomness: text embeddings seed 1, initial latent
# seed 2, step-k noise seed 100 + k, rewards seed 7, old-log-prob jitter seed 9.
# ---------------------------------------------------------------------------

def text_embeds(cfg: dict, seed: int = 1, batch: int | None = None) -> np.ndarray:
    """bf16 bits [B, N_t, D_txt], values N(0, 1) (cached prompt embeddings)."""
    B = cfg["batch"] if batch is None else batch
    shape = (B, cfg["n_txt"], cfg["txt_dim"])
    v = _rng(seed, "txt").standard_normal(int(np.prod(shape)), dtype=np.float32)
    return bf16_bits(v).reshape(shape)


def initial_latent(cfg: dict, seed: int = 2, batch: int | None = None) -> np.ndarray:
    """fp32 [B, N_i, P] initial noise x_T ~ N(0, 1)."""
    B = cfg["batch"] if batch is None else batch
    shape = (B, n_img(cfg), cfg["patch_dim"])
    return _rng(seed, "x_T").standard_normal(int(np.prod(shape)), dtype=np.float32).reshape(shape)


def step_noise(cfg: dict, k: int, seed: int = 100, batch: int | None = None) -> np.ndarray:
    """fp32 [B, N_i, P] Gaussian noise eps of SDE step k (seed 100 + k)."""
    B = cfg["batch"] if batch is None else batch
    shape = (B, n_img(cfg), cfg["patch_dim"])
    return _rng(seed + k, "eps").standard_normal(int(np.prod(shape)), dtype=np.float32).reshape(shape)


def gaussian(shape, seed: int, tag: str = "gauss") -> np.ndarray:
    n = int(np.prod(shape))
    return _rng(seed, tag).standard_normal(n, dtype=np.float32).reshape(shape)


def uniform(shape, seed: int, tag: str = "unif") -> np.ndarray:
    n = int(np.prod(shape))
    return _rng(seed, tag).random(n, dtype=np.float32).reshape(shape)


def rewards(n: int, seed: int = 7) -> np.ndarray:
    """fp32 [n] rewards U(0, 1) (synthetic stand-in for a reward model)."""
    return uniform((n,), seed, "reward")


def logprob_jitter(shape, seed: int = 9, std: float = 0.01) -> np.ndarray:
    """fp32 noise N(0, std^2) added to new log-probs to make synthetic old ones."""
    return gaussian(shape, seed, "lp_jitter") * np.float32(std)
