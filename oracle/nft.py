"""DiffusionNFT loss of Eq. 2 (fp64).  Test infrastructure only (see
oracle/__init__.py).

Eq. 2:  L = E_{c,t} [ r ||v+ - v||^2 + (1 - r) ||v- - v||^2 ],  r in [0, 1],
with v+ / v- the implicit positive / negative policies and v the
flow-matching target.  The paper names v+ and v- without defining them.
Reading (the definitions of the cited DiffusionNFT method): with v_old the
frozen velocity of the sampling policy, v_theta the trained one and a
strength beta > 0,
    v+ = (1 - beta) v_old + beta v_theta,   v- = (1 + beta) v_old - beta v_theta,
and the target v = eps - x0 of the interpolation x_t = (1 - t) x0 + t eps (the
convention under which Eq. 3's target is eps - x0).  The expectation is the
batch mean; "sum" keeps the squared norms, "mean" divides them by D.
"""
from __future__ import annotations

import numpy as np


def implicit_policies(v, v_old, beta: float):
    """(v+, v-) of the reading above."""
    v = np.asarray(v, dtype=np.float64)
    v_old = np.asarray(v_old, dtype=np.float64)
    return (1.0 - beta) * v_old + beta * v, (1.0 + beta) * v_old - beta * v


def nft_loss(v, v_old, eps, x0, r, beta: float, reduce: str = "sum"):
    """Returns (loss, dL/dv [B, ...], per-sample errors [B, 2] = (e+, e-)),
    e+- = ||v+- - (eps - x0)||^2 per sample (divided by D for "mean").
    v, v_old, eps, x0: [B, ...]; r: [B]."""
    v = np.asarray(v, dtype=np.float64)
    B = v.shape[0]
    target = np.asarray(eps, dtype=np.float64) - np.asarray(x0, dtype=np.float64)
    vp, vn = implicit_policies(v, v_old, beta)
    rp, rn = vp - target, vn - target
    D = v[0].size
    scale = 1.0 / D if reduce == "mean" else 1.0
    ax = tuple(range(1, v.ndim))
    err = np.stack([(rp * rp).sum(axis=ax), (rn * rn).sum(axis=ax)], axis=1) * scale
    rr = np.asarray(r, dtype=np.float64).reshape((B,) + (1,) * (v.ndim - 1))
    loss = float((rr.reshape(B) * err[:, 0] + (1.0 - rr.reshape(B)) * err[:, 1]).mean())
    # d/dv of r ||v+ - v||^2 is 2 r beta (v+ - v); of (1 - r) ||v- - v||^2, -2 (1 - r) beta (v- - v)
    grad = 2.0 * beta * (rr * rp - (1.0 - rr) * rn) * scale / B
    return loss, grad, err
