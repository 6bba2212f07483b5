"""Trajectory sampling (fp64): S denoise steps of Eq. 1 with the DiT
velocity, per-step transition log-probs kept (paper Sec. 3.1).

A plain composition of ``oracle.dit`` (the velocity) and ``oracle.sde`` (the
step and its log-prob): at step k every sample moves from t_k to t_{k+1}
with sigma_k and noise eps[k].  Its pins are those of the two modules plus
the composition checks in tests/test_oracle_rollout.py.
"""
from __future__ import annotations

import numpy as np

from . import dit, sde


def rollout(P, cfg, x0, txt, t_grid, sigma, eps, reduce: str = "sum", velocity=None):
    """x0: [B, ...]; t_grid: [S + 1]; sigma: [S]; eps: [S, B, ...].
    Returns (trajectory [S + 1, B, ...], logp [B, S])."""
    vel = velocity or (dit.wan_velocity if cfg.get("arch") == "wan" else dit.velocity)
    x = np.asarray(x0, dtype=np.float64)
    S = len(sigma)
    B = x.shape[0]
    traj = [x]
    lp = np.zeros((B, S))
    for k in range(S):
        t = np.full(B, float(t_grid[k]))
        tn = np.full(B, float(t_grid[k + 1]))
        sg = np.full(B, float(sigma[k]))
        v = vel(P, cfg, x, txt, t)
        x, lp[:, k] = sde.sde_step_logprob(x, v, t, tn, sg, eps=eps[k], reduce=reduce)
        traj.append(x)
    return np.stack(traj), lp
