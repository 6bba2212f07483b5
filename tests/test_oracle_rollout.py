"""Pins of the fp64 rollout oracle: it is the step-by-step composition of the
pinned velocity and SDE step, an ODE rollout scores log-prob 0 everywhere,
and a rollout driven by the exact flow velocity of a point mass lands on it."""
import numpy as np

from oracle import rollout as orollout
from oracle import sde as osde


def _field(P, cfg, x, txt, t):
    # exact velocity field of a flow whose data is the point x0 = c:
    # x_t = (1 - t) c + t eps  =>  v = (x_t - c) / t
    return (x - P) / t.reshape((-1,) + (1,) * (x.ndim - 1))


def test_single_step_is_one_velocity_and_one_sde_step():
    rng = np.random.default_rng(0)
    c = rng.standard_normal((2, 8))
    x0 = rng.standard_normal((2, 8))
    eps = rng.standard_normal((1, 2, 8))
    tr, lp = orollout.rollout(c, {}, x0, None, [0.9, 0.6], [0.4], eps, velocity=_field)
    v = _field(c, {}, x0, None, np.full(2, 0.9))
    want_x, want_lp = osde.sde_step_logprob(x0, v, np.full(2, 0.9), np.full(2, 0.6), np.full(2, 0.4), eps=eps[0])
    np.testing.assert_array_equal(tr[1], want_x)
    np.testing.assert_array_equal(lp[:, 0], want_lp)


def test_ode_rollout_of_a_point_mass_reaches_the_point():
    """sigma = 0 everywhere: every log-prob is 0, and with the exact velocity
    field of a point mass c the Euler steps stay on the straight path to c,
    reaching it at t = 0 (each step is exact for a straight path)."""
    rng = np.random.default_rng(1)
    c = rng.standard_normal((3, 5))
    e = rng.standard_normal((3, 5))
    grid = osde.time_grid(6, 3.0)
    x0 = (1 - grid[0]) * c + grid[0] * e
    S = len(grid) - 1
    tr, lp = orollout.rollout(c, {}, x0, None, grid[:-1].tolist() + [1e-12], np.zeros(S), np.zeros((S, 3, 5)),
                              velocity=_field)
    assert np.all(lp == 0.0)
    for k in range(S):
        np.testing.assert_allclose(tr[k], (1 - grid[k]) * c + grid[k] * e, atol=1e-12)
    np.testing.assert_allclose(tr[S], c, atol=1e-9)
