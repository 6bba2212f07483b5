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
  * GRPO-Guard's timestep-dependent reweighting (Sec. 3.1) multiplies the
    term of step k by a weight w_k (loss and gradient); the weights are not
    given in the paper and are an input (all ones = plain GRPO).
  * Multi-reward aggregation (Sec. 2.3, "weighted-sum and GDPO-style
    per-reward normalization") over K rewards R[b, k] with weights w_k:
      weighted sum: r_b = sum_k w_k R[b, k], then the group normalisation
      above;
      per reward:   each reward column is group-normalised on its own,
                    A_b = sum_k w_k A[b, k] (no further normalisation).
"""
from __future__ import annotations

import numpy as np


def group_advantage(rewards, group: int, eps: float = 1e-4) -> np.ndarray:
    r = np.asarray(rewards, dtype=np.float64).reshape(-1, group)
    mean = r.mean(axis=1, keepdims=True)
    std = np.sqrt(((r - mean) ** 2).mean(axis=1, keepdims=True))
    return ((r - mean) / (std + eps)).ravel()


def group_advantage_multi(rewards, group: int, weights, mode: str = "weighted_sum", eps: float = 1e-4) -> np.ndarray:
    """rewards: [N, K] (N = groups * G); weights: [K]; mode "weighted_sum" or
    "per_reward".  Returns the [N] advantages."""
    R = np.asarray(rewards, dtype=np.float64)
    w = np.asarray(weights, dtype=np.float64)
    N, K = R.shape
    if mode == "weighted_sum":
        return group_advantage(R @ w, group, eps)
    if mode == "per_reward":
        out = np.zeros(N)
        for k in range(K):
            out += w[k] * group_advantage(R[:, k], group, eps)
        return out
    raise ValueError(mode)


def grpo_loss(lp_new, lp_old, adv, clip_lo: float = 0.2, clip_hi: float = 0.2, step_w=None):
    """Returns (loss, dloss/dlp_new [B, T]); step_w: [T] weights or None."""
    lp_new = np.asarray(lp_new, dtype=np.float64)
    lp_old = np.asarray(lp_old, dtype=np.float64)
    B, T = lp_new.shape
    a = np.asarray(adv, dtype=np.float64).reshape(B, 1)
    w = np.ones((1, T)) if step_w is None else np.asarray(step_w, dtype=np.float64).reshape(1, T)
    rho = np.exp(lp_new - lp_old)
    unclipped = rho * a
    clipped = np.clip(rho, 1.0 - clip_lo, 1.0 + clip_hi) * a
    take_unclipped = unclipped <= clipped
    obj = np.where(take_unclipped, unclipped, clipped)
    loss = -(w * obj).sum() / (B * T)
    grad = np.where(take_unclipped, -w * a * rho / (B * T), 0.0)
    return float(loss), grad
