"""Pins of the dense-product oracle: brute force for every operand layout,
and the Linear backward against central differences of a scalar loss."""
import numpy as np
import pytest

from oracle import linalg


@pytest.mark.parametrize("al,bl", [("MK", "NK"), ("MK", "KN"), ("KM", "NK"), ("KM", "KN")])
def test_gemm_layouts_brute_force(al, bl):
    rng = np.random.default_rng(0)
    M, N, K = 3, 4, 5
    A = rng.standard_normal((M, K) if al == "MK" else (K, M))
    B = rng.standard_normal((N, K) if bl == "NK" else (K, N))
    bias = rng.standard_normal(N)
    got = linalg.gemm(A, B, al, bl, bias)
    a = lambda m, k: A[m, k] if al == "MK" else A[k, m]
    b = lambda k, n: B[n, k] if bl == "NK" else B[k, n]
    for m in range(M):
        for n in range(N):
            want = sum(a(m, k) * b(k, n) for k in range(K)) + bias[n]
            assert got[m, n] == pytest.approx(want, rel=1e-13, abs=1e-13)


def test_linear_backward_central_differences():
    rng = np.random.default_rng(1)
    T, Nin, Nout = 4, 3, 5
    x, W, b, g = (rng.standard_normal((T, Nin)), rng.standard_normal((Nout, Nin)), rng.standard_normal(Nout),
                  rng.standard_normal((T, Nout)))
    loss = lambda x_, W_, b_: float(np.sum(g * (x_ @ W_.T + b_)))
    dx, dW, db = linalg.linear_backward(x, W, g)
    h = 1e-6
    for arr, grad in ((x, dx), (W, dW), (b, db)):
        it = np.nditer(arr, flags=["multi_index"])
        for _ in it:
            i = it.multi_index
            p_, m_ = arr.copy(), arr.copy()
            p_[i] += h
            m_[i] -= h
            args_p = [p_ if arr is v else v for v in (x, W, b)]
            args_m = [m_ if arr is v else v for v in (x, W, b)]
            fd = (loss(*args_p) - loss(*args_m)) / (2 * h)
            assert grad[i] == pytest.approx(fd, rel=1e-7, abs=1e-9)
