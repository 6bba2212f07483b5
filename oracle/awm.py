"""Advantage Weighted Matching (fp64): the forward process, training-time
sampling and the loss of Eq. 3 (paper Sec. 3.2).

Readings (the paper leaves these open):
  * The forward (noising) process is x_t = (1 - t) x_0 + t eps, the
    convention under which Eq. 3's regression target is eps - x_0 (the same
    convention as the sampler in ``oracle.sde``).
  * Eq. 3's expectation over (t, eps) is estimated by the batch mean over
    samples b, each with its own t_b, eps_b and advantage A_b:
        L = (1 / B) sum_b A_b e_b,  e_b = ||v_b - (eps_b - x0_b)||^2
    with ||.||^2 the sum of squares over the D elements of a sample as
    printed ("sum"); "mean" divides e_b by D (the per-element MSE
    normalisation of flow-matching pre-training).
  * dL/dv_b = (2 / B) A_b (v_b - (eps_b - x0_b)), divided by D for "mean".
  * Training times (Sec. 3.2, "uniform, logit-normal, or discrete"):
      uniform       t = t_min + (t_max - t_min) u,  u ~ U[0, 1)
      logit-normal  t = 1 / (1 + exp(-(m + s z))),  z ~ N(0, 1)
      discrete      t = grid[min(floor(u n), n - 1)] over a grid of n times
    The random draws u or z are inputs, not drawn here.  The discrete index
    is a floating-point decision that picks an integer, so it is taken in
    float32 (u and n rounded to float32, their product rounded once), the
    precision the kernel uses; everything else is float64.
"""
from __future__ import annotations

import math

import numpy as np


def sample_timesteps(mode: str, draw, p0: float = 0.0, p1: float = 1.0, grid=None) -> np.ndarray:
    """mode "uniform" (p0, p1 = t_min, t_max), "logit_normal" (p0, p1 = m, s)
    or "discrete" (grid of times); draw: the u or z of each sample."""
    d = np.asarray(draw, dtype=np.float64)
    if mode == "uniform":
        return p0 + (p1 - p0) * d
    if mode == "logit_normal":
        return np.array([1.0 / (1.0 + math.exp(-(p0 + p1 * z))) for z in d.ravel()]).reshape(d.shape)
    if mode == "discrete":
        g = np.asarray(grid, dtype=np.float64)
        n = g.size
        prod = np.float32(d.ravel()).astype(np.float32) * np.float32(n)   # one float32 rounding
        idx = np.array([max(0, min(int(math.floor(float(x))), n - 1)) for x in prod]).reshape(d.shape)
        return g[idx]
    raise ValueError(mode)


def forward_process(x0, eps, t) -> np.ndarray:
    """x_t = (1 - t_b) x0_b + t_b eps_b per sample; x0, eps: [B, ...], t: [B]."""
    x0 = np.asarray(x0, dtype=np.float64)
    eps = np.asarray(eps, dtype=np.float64)
    t = np.asarray(t, dtype=np.float64).reshape((-1,) + (1,) * (x0.ndim - 1))
    return (1.0 - t) * x0 + t * eps


def awm_loss(v, eps, x0, adv, reduce: str = "sum"):
    """Eq. 3 over a batch.  Returns (loss, dloss/dv [B, ...], e [B])."""
    v = np.asarray(v, dtype=np.float64)
    eps = np.asarray(eps, dtype=np.float64)
    x0 = np.asarray(x0, dtype=np.float64)
    B = v.shape[0]
    D = v[0].size
    a = np.asarray(adv, dtype=np.float64).reshape(B)
    r = v - (eps - x0)
    e = np.array([float(np.dot(r[b].ravel(), r[b].ravel())) for b in range(B)])
    scale = 1.0 / D if reduce == "mean" else 1.0
    e = e * scale
    loss = float(np.sum(a * e) / B)
    grad = (2.0 * scale / B) * a.reshape((-1,) + (1,) * (v.ndim - 1)) * r
    return loss, grad, e
