"""Pins of the DiffusionNFT loss (Eq. 2, oracle/nft.py): closed forms of the
special cases, the quadratic's minimiser, and central differences."""
import numpy as np
import pytest

from oracle import awm, nft


def _batch(seed=0, B=3, D=24):
    rng = np.random.default_rng(seed)
    return (rng.standard_normal((B, D)), rng.standard_normal((B, D)), rng.standard_normal((B, D)),
            rng.standard_normal((B, D)), rng.uniform(0, 1, B))


def test_beta_one_reward_one_is_flow_matching():
    # beta = 1 makes v+ = v_theta; r = 1 keeps only that term: the plain
    # flow-matching loss, i.e. AWM (Eq. 3) with every advantage 1
    v, vo, e, x0, _ = _batch()
    for reduce in ("sum", "mean"):
        L, g, _ = nft.nft_loss(v, vo, e, x0, np.ones(3), 1.0, reduce)
        La, ga, _ = awm.awm_loss(v, e, x0, np.ones(3), reduce)
        assert L == pytest.approx(La, rel=1e-13)
        np.testing.assert_allclose(g, ga, rtol=1e-13)


def test_reward_zero_keeps_the_negative_term():
    v, vo, e, x0, _ = _batch(1)
    beta = 0.3
    L, _, err = nft.nft_loss(v, vo, e, x0, np.zeros(3), beta)
    vn = (1 + beta) * vo - beta * v
    assert L == pytest.approx(float(((vn - (e - x0)) ** 2).sum(axis=1).mean()), rel=1e-13)
    np.testing.assert_allclose(err[:, 1], ((vn - (e - x0)) ** 2).sum(axis=1), rtol=1e-13)


def test_equal_policies():
    # v_theta = v_old gives v+ = v- = v_old: the loss is ||v_old - target||^2 for any r, and the
    # gradient is 2 beta (2 r - 1) (v_old - target) / B
    v, vo, e, x0, r = _batch(2)
    beta = 0.7
    L, g, err = nft.nft_loss(vo, vo, e, x0, r, beta)
    res = vo - (e - x0)
    assert L == pytest.approx(float((res ** 2).sum(axis=1).mean()), rel=1e-13)
    np.testing.assert_allclose(err[:, 0], err[:, 1], rtol=1e-13)
    np.testing.assert_allclose(g, 2 * beta * (2 * r[:, None] - 1) * res / 3, rtol=1e-12, atol=1e-15)


def test_gradient_vanishes_at_the_minimiser():
    # the loss is a convex quadratic in v_theta with minimiser
    # v* = v_old + (2 r - 1) (target - v_old) / beta
    v, vo, e, x0, r = _batch(3)
    beta = 0.4
    tgt = e - x0
    vstar = vo + (2 * r[:, None] - 1) * (tgt - vo) / beta
    _, g, _ = nft.nft_loss(vstar, vo, e, x0, r, beta)
    np.testing.assert_allclose(g, 0, atol=1e-12)
    L0, _, _ = nft.nft_loss(vstar, vo, e, x0, r, beta)
    L1, _, _ = nft.nft_loss(vstar + 1e-3 * np.random.default_rng(9).standard_normal(v.shape), vo, e, x0, r, beta)
    assert L1 > L0


@pytest.mark.parametrize("reduce", ["sum", "mean"])
def test_gradient_by_central_differences(reduce):
    v, vo, e, x0, r = _batch(4, B=4, D=10)
    beta = 0.25
    _, g, _ = nft.nft_loss(v, vo, e, x0, r, beta, reduce)
    d = np.random.default_rng(5).standard_normal(v.shape)
    h = 1e-6
    num = (nft.nft_loss(v + h * d, vo, e, x0, r, beta, reduce)[0] -
           nft.nft_loss(v - h * d, vo, e, x0, r, beta, reduce)[0]) / (2 * h)
    assert num == pytest.approx(float((g * d).sum()), rel=1e-7)
