"""Pins of the fp64 oracle for the Flow-SDE step (Eq. 1, Table 1) and its
Gaussian transition log-probability.  CPU only."""
import math
import os

import numpy as np
import pytest
import scipy.stats

from oracle import sde

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _load(name):
    rows = []
    with open(os.path.join(GOLDEN, name)) as f:
        for line in f:
            line = line.strip()
            if line and not line.startswith("#"):
                rows.append([float(v) for v in line.split()])
    return np.array(rows)


def test_sigma_table_values():
    # Table 1 Flow-SDE row at hand-worked points (tests/golden/flow_sde_sigma.txt)
    for t, eta, tc, want in _load("flow_sde_sigma.txt"):
        got = sde.sigma_flow_sde(t, eta, tc)
        assert abs(got - want) <= 1e-15 * max(1.0, want), (t, got, want)


def test_sigma_other_rows():
    t = np.linspace(0.1, 1.0, 7)
    assert np.all(sde.sigma_dance_sde(t, 0.3) == 0.3)   # Dance-SDE: constant
    assert np.all(sde.sigma_ode(t) == 0.0)              # ODE: zero


def test_shifted_grid_values():
    g = sde.time_grid(10, 3.0)
    for k, want in _load("shifted_time_grid.txt"):
        assert abs(g[int(k)] - want) <= 1e-15, (k, g[int(k)], want)
    lin = sde.time_grid(4)
    assert np.array_equal(lin, [1.0, 0.75, 0.5, 0.25, 0.0])
    assert np.all(np.diff(g) < 0)


def test_sigma_zero_is_euler_ode_step():
    # Table 1 ODE row / Sec. 3.1: with sigma = 0, Eq. 1 is x_{t+dt} = x_t + v dt
    rng = np.random.default_rng(0)
    x, v = rng.standard_normal(50), rng.standard_normal(50)
    t, tn = 0.75, 0.5
    mean, std = sde.sde_mean_std(x, v, t, tn, 0.0)
    assert std == 0.0
    np.testing.assert_array_equal(mean, x + v * (tn - t))


def _analytic_velocity(x, t, s0):
    # x_0 ~ N(0, s0^2), eps ~ N(0, 1), x_t = (1-t) x_0 + t eps:
    # v(x, t) = E[eps - x_0 | x_t = x] = (t - (1-t) s0^2) / ((1-t)^2 s0^2 + t^2) * x
    return (t - (1 - t) * s0 ** 2) / ((1 - t) ** 2 * s0 ** 2 + t ** 2) * x


@pytest.mark.parametrize("eta,steps,tol", [(0.0, 200, 0.01), (0.7, 200, 0.01), (0.7, 50, 0.015)])
def test_sde_rollout_recovers_gaussian_data(eta, steps, tol):
    # The reverse SDE of Eq. 1 driven by the exact velocity of Gaussian data must
    # carry N(0,1) noise at t=1 to data variance s0^2 at t=0.  A flipped drift
    # sign or a wrong score term makes the variance drift away.
    s0 = 0.5
    n = 200_000
    rng = np.random.default_rng(1)
    x = rng.standard_normal(n)
    grid = sde.time_grid(steps)
    for k in range(steps):
        t, tn = grid[k], grid[k + 1]
        sig = float(sde.sigma_flow_sde(t, eta, 0.96))
        mean, std = sde.sde_mean_std(x, _analytic_velocity(x, t, s0), t, tn, sig)
        x = mean + std * rng.standard_normal(n)
    assert abs(x.var() - s0 ** 2) < tol, x.var()
    assert abs(x.mean()) < 0.01


def test_sde_rollout_wrong_sign_diverges():
    # Guard that the variance test above is sensitive: flipping the score term's
    # sign (a plausible mistake) must fail it.
    s0, n, steps = 0.5, 100_000, 100
    rng = np.random.default_rng(2)
    x = rng.standard_normal(n)
    grid = sde.time_grid(steps)
    for k in range(steps):
        t, tn = grid[k], grid[k + 1]
        sig = float(sde.sigma_flow_sde(t, 0.7, 0.96))
        v = _analytic_velocity(x, t, s0)
        delta = t - tn
        mean = x - (v - sig ** 2 / (2 * t) * (x + (1 - t) * v)) * delta
        x = mean + sig * math.sqrt(delta) * rng.standard_normal(n)
    assert abs(x.var() - s0 ** 2) > 0.05


def test_transition_std_monte_carlo():
    rng = np.random.default_rng(3)
    n = 1_000_000
    x, v = np.zeros(n), np.zeros(n)
    t, tn, sig = 0.8, 0.6, 1.3
    mean, std = sde.sde_mean_std(x, v, t, tn, sig)
    xn = mean + std * rng.standard_normal(n)
    assert abs(np.var(xn - mean) / (sig ** 2 * (t - tn)) - 1.0) < 5e-3


def test_logprob_at_mean_is_normaliser():
    rng = np.random.default_rng(4)
    D = 1000
    mean = rng.standard_normal(D)
    s = 0.37
    lp = sde.gaussian_logprob(mean, mean, s)
    assert lp == pytest.approx(-D * (math.log(s) + 0.5 * math.log(2 * math.pi)), rel=1e-14)


def test_logprob_sample_mode_closed_form():
    rng = np.random.default_rng(5)
    B, D = 3, 512
    x, v, eps = rng.standard_normal((3, B, D))
    t = np.full(B, 0.75)
    tn = np.full(B, 0.5)
    sig = sde.sigma_flow_sde(t, 0.7)
    xn, lp = sde.sde_step_logprob(x, v, t, tn, sig, eps=eps)
    s = sig * np.sqrt(t - tn)
    want = -0.5 * (eps ** 2).sum(1) - D * np.log(s) - 0.5 * D * math.log(2 * math.pi)
    np.testing.assert_allclose(lp, want, rtol=1e-12)
    # eval mode on the sampled x_next gives the same log-prob
    _, lp2 = sde.sde_step_logprob(x, v, t, tn, sig, x_next=xn)
    np.testing.assert_allclose(lp2, lp, rtol=1e-12)
    _, lpm = sde.sde_step_logprob(x, v, t, tn, sig, x_next=xn, reduce="mean")
    np.testing.assert_allclose(lpm, lp / D, rtol=1e-14)


def test_logprob_one_element_matches_scipy():
    rng = np.random.default_rng(6)
    for _ in range(20):
        x, v, e = rng.standard_normal(3)
        t, tn = sorted(rng.uniform(0.05, 0.95, 2))[::-1]
        sig = rng.uniform(0.1, 2.0)
        mean, std = sde.sde_mean_std(np.array([x]), np.array([v]), t, tn, sig)
        xn = mean + std * e
        lp = sde.gaussian_logprob(xn, mean, std)
        assert lp == pytest.approx(scipy.stats.norm.logpdf(xn[0], loc=mean[0], scale=std), rel=1e-12)


def test_ode_step_logprob_is_zero():
    x = np.ones((1, 8))
    xn, lp = sde.sde_step_logprob(x, x, [0.5], [0.25], [0.0], eps=np.ones((1, 8)))
    assert lp[0] == 0.0
    np.testing.assert_array_equal(xn, x - x * 0.25)


def test_mixgrpo_window_keeps_sigma_inside_and_zeroes_outside():
    t = sde.time_grid(10, 3.0)
    s = sde.sigma_flow_sde(t[:-1], 0.7)
    w = sde.window_sigma(s, 3, 2)
    np.testing.assert_array_equal(w[3:5], s[3:5])
    assert np.all(w[:3] == 0.0) and np.all(w[5:] == 0.0)
    assert np.array_equal(sde.window_sigma(s, 0, 10), s)
    # an ODE step scores log-prob 0 and moves x by the drift only
    x, v = np.ones(4), np.full(4, 0.5)
    mean, std = sde.sde_mean_std(x, v, t[0], t[1], w[0])
    assert std == 0.0 and sde.gaussian_logprob(mean, mean, std) == 0.0
    np.testing.assert_allclose(mean, x - v * (t[0] - t[1]))
