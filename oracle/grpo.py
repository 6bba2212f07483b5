"""Group-relative advantage and clipped-ratio policy loss (fp64).

The paper names these steps (Sec. 2.3: advantage computation in the trainer,
``compute_advantages``; Sec. 3.1: Flow-GRPO policy-gradient training) without
printing formulas.  Readings used here:
  * Samples are grouped in contiguous blocks of G (one prompt per group).
    A = (r - mean_g) / (std_g + eps_A) with the population std (ddof = 0).
  * Loss: the PPO-style clipped surrogate with ratio rho = exp(lp_new - lp_old)
    per (sample, step), advantages broadcast over steps, no KL term, averaged
    over all B * T pairs and negated so that it is minimised:
        L = -(1 / (B T)) sum_{b,k} min(rho A_b, clip(rho, 1 - e_lo, 1 + e_hi) A_b)
  * Gradient w.r.t. lp_new: -A rho / (B T) where the unclipped term is the
    minimum (ties count as unclipped), else 0.
"""
from __future__ import annotations

import numpy as np


def group_advantage(rewards, group: int, eps: float = 1e-4) -> np.ndarray:
    r = np.asarray(rewards, dtype=np.float64).reshape(-1, group)
    mean = r.mean(axis=1, keepdims=True)
    std = np.sqrt(((r - mean) ** 2).mean(axis=1, keepdims=True))
    return ((r - mean) / (std + eps)).ravel()


def grpo_loss(lp_new, lp_old, adv, clip_lo: float = 0.2, clip_hi: float = 0.2):
    """Returns (loss, dloss/dlp_new [B, T])."""
    lp_new = np.asarray(lp_new, dtype=np.float64)
    lp_old = np.asarray(lp_old, dtype=np.float64)
    B, T = lp_new.shape
    a = np.asarray(adv, dtype=np.float64).reshape(B, 1)
    rho = np.exp(lp_new - lp_old)
    unclipped = rho * a
    clipped = np.clip(rho, 1.0 - clip_lo, 1.0 + clip_hi) * a
    take_unclipped = unclipped <= clipped
    obj = np.where(take_unclipped, unclipped, clipped)
    loss = -obj.sum() / (B * T)
    grad = np.where(take_unclipped, -a * rho / (B * T), 0.0)
    return float(loss), grad
