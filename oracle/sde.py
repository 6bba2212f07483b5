"""Flow-SDE sampler and its transition log-probability (fp64).

Follows Sec. 3.1 of the paper: Eq. 1 (the SDE update that replaces the ODE
step x_{t+dt} = x_t + v dt) and Table 1 (noise schedules sigma_t).

Readings (the paper leaves these open):
  * Time runs from 1 (noise) to 0 (data) with x_t = (1 - t) x_0 + t eps, the
    convention under which the AWM target of Eq. 3 is eps - x_0.  Sampling
    steps therefore have dt = t_next - t < 0, and the noise term sigma sqrt(dt)
    of Eq. 1 is read as sigma sqrt(|dt|).  With Delta = t - t_next > 0:
        mean = x - [v + sigma^2 / (2 t) (x + (1 - t) v)] * Delta
        std  = sigma * sqrt(Delta)
  * sigma_t and the drift's 1/(2t) use the step's starting time t
    (Euler-Maruyama).
  * Flow-SDE sigma_t = eta sqrt(t / (1 - t)) is singular at t = 1; t is
    clamped to t_clamp (0.96) inside the square root.
  * The log-probability is the exact log-density of the Gaussian transition,
    summed over all D elements of a sample ("sum"), or divided by D ("mean").
  * A step with std = 0 (the ODE row of Table 1) has no density; its log-prob
    is reported as 0.
"""
from __future__ import annotations

import math

import numpy as np


def time_grid(n_steps: int, shift: float = 1.0) -> np.ndarray:
    """t_0 = 1 > t_1 > ... > t_S = 0: linear grid, then the time shift
    t' = s t / (1 + (s - 1) t) (shift s = 1 leaves the grid linear)."""
    t = 1.0 - np.arange(n_steps + 1, dtype=np.float64) / n_steps
    if shift != 1.0:
        t = shift * t / (1.0 + (shift - 1.0) * t)
    return t


def sigma_flow_sde(t, eta: float, t_clamp: float = 0.96):
    """Table 1, Flow-SDE row: sigma_t = eta sqrt(t / (1 - t)), t clamped."""
    tc = np.minimum(np.asarray(t, dtype=np.float64), t_clamp)
    return eta * np.sqrt(tc / (1.0 - tc))


def sigma_dance_sde(t, eta: float):
    """Table 1, Dance-SDE row: constant sigma_t = eta."""
    return np.full_like(np.asarray(t, dtype=np.float64), eta)


def sigma_ode(t):
    """Table 1, ODE row: sigma_t = 0 (deterministic)."""
    return np.zeros_like(np.asarray(t, dtype=np.float64))


def window_sigma(sigma, start: int, length: int) -> np.ndarray:
    """MixGRPO (Sec. 3.1): SDE noise on steps start .. start + length - 1 only,
    the deterministic ODE update (sigma = 0) on every other step."""
    s = np.array(sigma, dtype=np.float64)
    k = np.arange(s.size)
    s[(k < start) | (k >= start + length)] = 0.0
    return s


def sde_mean_std(x, v, t: float, t_next: float, sigma: float):
    """Mean and std of the Gaussian transition of Eq. 1 for one sample.

    x, v: arrays of one sample (any shape); t, t_next, sigma: scalars.
    """
    x = np.asarray(x, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    delta = float(t) - float(t_next)
    drift = v + (sigma * sigma) / (2.0 * t) * (x + (1.0 - t) * v)
    mean = x - drift * delta
    std = sigma * math.sqrt(delta)
    return mean, std


def gaussian_logprob(x_next, mean, std: float, reduce: str = "sum") -> float:
    """log N(x_next; mean, std^2 I) summed (or averaged) over all elements."""
    x_next = np.asarray(x_next, dtype=np.float64)
    d = x_next.size
    if std == 0.0:
        return 0.0
    r = (x_next - mean).ravel()
    lp = -0.5 * float(np.dot(r, r)) / (std * std) - d * math.log(std) - 0.5 * d * math.log(2.0 * math.pi)
    return lp / d if reduce == "mean" else lp


def sde_step_logprob(x, v, t, t_next, sigma, eps=None, x_next=None, reduce: str = "sum"):
    """One SDE step for a batch.

    x, v: [B, ...]; t, t_next, sigma: [B].  Sample mode (eps given):
    x_next = mean + std * eps.  Eval mode (x_next given): x_next is taken as is.
    Returns (x_next [B, ...] float64, logp [B] float64).
    """
    x = np.asarray(x, dtype=np.float64)
    B = x.shape[0]
    out = np.empty_like(x)
    lp = np.empty(B, dtype=np.float64)
    for b in range(B):
        mean, std = sde_mean_std(x[b], v[b], float(t[b]), float(t_next[b]), float(sigma[b]))
        if x_next is None:
            out[b] = mean + std * np.asarray(eps[b], dtype=np.float64)
        else:
            out[b] = np.asarray(x_next[b], dtype=np.float64)
        lp[b] = gaussian_logprob(out[b], mean, std, reduce)
    return out, lp


def sde_logprob_grad_v(x, v, x_next, t, t_next, sigma, reduce: str = "sum") -> np.ndarray:
    """d logp_b / d v_b of the Eq. 1 transition with x_next held fixed (the
    training pass re-scores the rollout's x_next under the current v).

    logp = -|x_next - mean|^2 / (2 std^2) + const depends on v only through
    mean, and d mean_j / d v_j = -Delta (1 + sigma^2 (1 - t) / (2 t)), so
        d logp / d v_j = (x_next_j - mean_j) / std^2 * d mean_j / d v_j
    (divided by D for the "mean" reduction).  Zero where std = 0 (no density).
    x, v, x_next: [B, ...]; t, t_next, sigma: [B].
    """
    x = np.asarray(x, dtype=np.float64)
    out = np.zeros_like(x)
    for b in range(x.shape[0]):
        tb, sb = float(t[b]), float(sigma[b])
        mean, std = sde_mean_std(x[b], v[b], tb, float(t_next[b]), sb)
        if std == 0.0:
            continue
        delta = tb - float(t_next[b])
        dmean_dv = -delta * (1.0 + sb * sb * (1.0 - tb) / (2.0 * tb))
        g = (np.asarray(x_next[b], dtype=np.float64) - mean) / (std * std) * dmean_dv
        out[b] = g / x[b].size if reduce == "mean" else g
    return out
