"""Pins of the fp64 oracle for AWM (Eq. 3): the forward process, the
training-time samplers and the advantage-weighted matching loss."""
import math

import numpy as np
import pytest
from scipy.special import expit

from oracle import awm, sde


def test_forward_process_endpoints_and_linearity():
    rng = np.random.default_rng(0)
    x0, eps = rng.standard_normal((3, 5, 4)), rng.standard_normal((3, 5, 4))
    np.testing.assert_array_equal(awm.forward_process(x0, eps, np.zeros(3)), x0)
    np.testing.assert_array_equal(awm.forward_process(x0, eps, np.ones(3)), eps)
    t = np.array([0.25, 0.5, 0.9])
    xt = awm.forward_process(x0, eps, t)
    for b in range(3):   # per-sample time, hand formula
        np.testing.assert_allclose(xt[b], (1 - t[b]) * x0[b] + t[b] * eps[b], rtol=0, atol=1e-15)
    # d x_t / d t = eps - x0: the regression target of Eq. 3
    h = 1e-6
    d = (awm.forward_process(x0, eps, t + h) - awm.forward_process(x0, eps, t - h)) / (2 * h)
    np.testing.assert_allclose(d, eps - x0, atol=1e-8)


def test_exact_velocity_makes_the_ode_step_follow_the_forward_process():
    """With v = eps - x0 (zero AWM loss) the deterministic sampler step of
    Eq. 1 (sigma = 0) lands exactly on the forward process at t_next: this
    ties the sign conventions of the sampler and of Eq. 3 together."""
    rng = np.random.default_rng(1)
    x0, eps = rng.standard_normal(16), rng.standard_normal(16)
    t, tn = 0.8, 0.55
    xt = awm.forward_process(x0[None], eps[None], [t])[0]
    mean, std = sde.sde_mean_std(xt, eps - x0, t, tn, 0.0)
    assert std == 0.0
    np.testing.assert_allclose(mean, awm.forward_process(x0[None], eps[None], [tn])[0], atol=1e-14)


def test_awm_loss_brute_force_and_zero_at_the_target():
    rng = np.random.default_rng(2)
    B, D = 3, 7
    v, eps, x0 = rng.standard_normal((B, D)), rng.standard_normal((B, D)), rng.standard_normal((B, D))
    a = np.array([0.5, -1.25, 2.0])
    loss, grad, e = awm.awm_loss(v, eps, x0, a, "sum")
    want_e = [sum((v[b, j] - (eps[b, j] - x0[b, j])) ** 2 for j in range(D)) for b in range(B)]
    np.testing.assert_allclose(e, want_e, rtol=1e-14)
    assert loss == pytest.approx(sum(a[b] * want_e[b] for b in range(B)) / B, rel=1e-14)
    l0, g0, e0 = awm.awm_loss(eps - x0, eps, x0, a)
    assert l0 == 0.0 and np.all(g0 == 0.0) and np.all(e0 == 0.0)
    # "mean" is "sum" over D
    lm, gm, em = awm.awm_loss(v, eps, x0, a, "mean")
    assert lm == pytest.approx(loss / D, rel=1e-14)
    np.testing.assert_allclose(gm, grad / D, rtol=1e-14)


def test_awm_loss_gradient_by_central_differences():
    rng = np.random.default_rng(3)
    B, D = 2, 5
    v, eps, x0 = rng.standard_normal((B, D)), rng.standard_normal((B, D)), rng.standard_normal((B, D))
    a = np.array([1.5, -0.7])
    for reduce in ("sum", "mean"):
        _, grad, _ = awm.awm_loss(v, eps, x0, a, reduce)
        h = 1e-6
        for b in range(B):
            for j in range(D):
                vp, vm = v.copy(), v.copy()
                vp[b, j] += h
                vm[b, j] -= h
                fd = (awm.awm_loss(vp, eps, x0, a, reduce)[0] - awm.awm_loss(vm, eps, x0, a, reduce)[0]) / (2 * h)
                assert grad[b, j] == pytest.approx(fd, rel=1e-6, abs=1e-9)


def test_awm_loss_is_linear_in_the_advantage():
    rng = np.random.default_rng(4)
    v, eps, x0 = rng.standard_normal((4, 3)), rng.standard_normal((4, 3)), rng.standard_normal((4, 3))
    a1, a2 = rng.standard_normal(4), rng.standard_normal(4)
    l1, l2, l12 = (awm.awm_loss(v, eps, x0, a)[0] for a in (a1, a2, 2 * a1 - 3 * a2))
    assert l12 == pytest.approx(2 * l1 - 3 * l2, rel=1e-12)


def test_timestep_samplers():
    u = np.array([0.0, 0.25, 0.5, 0.999999])
    np.testing.assert_allclose(awm.sample_timesteps("uniform", u, 0.1, 0.9), 0.1 + 0.8 * u)
    # logit-normal: t = sigmoid(m + s z); z = 0 gives sigmoid(m); z -> -z with m = 0 gives 1 - t
    z = np.array([-2.0, -0.3, 0.0, 0.7, 3.0])
    np.testing.assert_allclose(awm.sample_timesteps("logit_normal", z, 0.4, 1.3), expit(0.4 + 1.3 * z), rtol=1e-15)
    t0 = awm.sample_timesteps("logit_normal", z, 0.0, 1.0)
    np.testing.assert_allclose(t0 + awm.sample_timesteps("logit_normal", -z, 0.0, 1.0), 1.0, atol=1e-15)
    assert np.all(np.diff(t0) > 0)
    # discrete: u in [k/n, (k+1)/n) picks grid[k]
    grid = sde.time_grid(4, 3.0)[:4]
    uu = np.array([0.0, 0.2499, 0.25, 0.74, 0.75, 0.9999999])
    np.testing.assert_array_equal(awm.sample_timesteps("discrete", uu, grid=grid), grid[[0, 0, 1, 2, 3, 3]])
