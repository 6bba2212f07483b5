"""Dense products of the training backward (fp64).

The Flow-GRPO update (Sec. 3.1) differentiates the policy loss through the
velocity network; for each Linear y = x W^T + b on T tokens that needs
  dx = dy W,   dW = dy^T x,   db = sum over tokens of dy.
``gemm`` is the plain statement of the three products with explicit operand
storage (a library matmul is the step), ``linear_backward`` their
composition.  Pinned by brute force and by central differences of a scalar
loss (tests/test_oracle_linalg.py).
"""
from __future__ import annotations

import numpy as np

from . import dit


def gemm(A, B, a_layout: str = "MK", b_layout: str = "NK", bias=None, act: str = "none") -> np.ndarray:
    """out = act(op(A) op(B) + bias); A stored [M, K] ("MK") or [K, M]
    ("KM"), B stored [N, K] ("NK", out = A B^T) or [K, N] ("KN")."""
    a = np.asarray(A, dtype=np.float64)
    b = np.asarray(B, dtype=np.float64)
    a = a if a_layout == "MK" else a.T
    b = b.T if b_layout == "NK" else b
    out = a @ b
    if bias is not None:
        out = out + np.asarray(bias, dtype=np.float64)
    if act == "gelu":
        out = dit.gelu_tanh(out)
    elif act == "silu":
        out = out / (1.0 + np.exp(-out))
    return out


def linear_backward(x, W, dy):
    """Gradients of sum(dy * (x W^T + b)) w.r.t. x, W and b."""
    x = np.asarray(x, dtype=np.float64)
    W = np.asarray(W, dtype=np.float64)
    dy = np.asarray(dy, dtype=np.float64)
    return gemm(dy, W, "MK", "KN"), gemm(dy, x, "KM", "KN"), dy.sum(axis=0)
