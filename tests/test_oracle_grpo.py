"""Pins of the fp64 oracle for the group advantage and the clipped GRPO loss."""
import itertools

import numpy as np
import pytest

from oracle import grpo


def test_advantage_zero_mean_and_scaled_std():
    rng = np.random.default_rng(0)
    G, ng, eps = 16, 5, 1e-4
    r = rng.random(G * ng)
    a = grpo.group_advantage(r, G, eps).reshape(ng, G)
    rg = r.reshape(ng, G)
    s = rg.std(axis=1)
    np.testing.assert_allclose(a.mean(axis=1), 0.0, atol=1e-14)
    np.testing.assert_allclose(a.std(axis=1), s / (s + eps), rtol=1e-12)


def test_advantage_constant_group_and_singleton():
    assert np.all(grpo.group_advantage(np.full(8, 0.3), 4) == 0.0)
    assert np.all(grpo.group_advantage(np.arange(5.0), 1) == 0.0)


def test_advantage_permutation_equivariant_and_group_local():
    rng = np.random.default_rng(1)
    r = rng.random(12)
    a = grpo.group_advantage(r, 4)
    perm = np.concatenate([rng.permutation(4) + 4 * g for g in range(3)])
    np.testing.assert_allclose(grpo.group_advantage(r[perm], 4), a[perm], rtol=0, atol=1e-15)
    r2 = r.copy()
    r2[4:8] += 10.0          # shifting one group leaves every advantage unchanged
    np.testing.assert_allclose(grpo.group_advantage(r2, 4), a, atol=1e-9)


def test_advantage_hand_values():
    # rewards (0, 1) in one group: mean 0.5, std 0.5 -> A = +-0.5 / (0.5 + eps)
    a = grpo.group_advantage([0.0, 1.0], 2, eps=0.0)
    np.testing.assert_array_equal(a, [-1.0, 1.0])


def test_loss_ratio_one_is_minus_mean_advantage():
    rng = np.random.default_rng(2)
    B, T = 6, 3
    lp = rng.standard_normal((B, T))
    adv = rng.standard_normal(B)
    loss, grad = grpo.grpo_loss(lp, lp, adv)
    assert loss == pytest.approx(-adv.mean(), rel=1e-14)
    np.testing.assert_allclose(grad, -np.repeat(adv[:, None], T, 1) / (B * T), rtol=1e-14)


def _case_analysis(rho, a, e):
    # PPO clipping written as its four cases instead of min(): a positive
    # advantage is capped above at 1 + e, a negative one below at 1 - e.
    if a >= 0:
        return -(1 + e) * a if rho > 1 + e else -rho * a
    return -(1 - e) * a if rho < 1 - e else -rho * a


def test_loss_all_branches_brute_force():
    e = 0.2
    rhos = [0.5, 0.79, 0.9, 1.0, 1.1, 1.21, 2.0]
    advs = [-1.5, -0.2, 0.3, 2.0]
    pairs = list(itertools.product(rhos, advs))
    B = len(pairs)
    lp_old = np.zeros((B, 1))
    lp_new = np.log([[p[0]] for p in pairs])
    adv = np.array([p[1] for p in pairs])
    loss, _ = grpo.grpo_loss(lp_new, lp_old, adv, e, e)
    want = np.mean([_case_analysis(r, a, e) for r, a in pairs])
    assert loss == pytest.approx(want, rel=1e-13)


def test_loss_gradient_finite_differences():
    rng = np.random.default_rng(3)
    B, T = 5, 4
    lp_old = rng.standard_normal((B, T))
    lp_new = lp_old + rng.normal(0, 0.3, (B, T))
    adv = rng.standard_normal(B)
    _, g = grpo.grpo_loss(lp_new, lp_old, adv)
    h = 1e-6
    for b, k in itertools.product(range(B), range(T)):
        rho = np.exp(lp_new[b, k] - lp_old[b, k])
        if min(abs(rho - 0.8), abs(rho - 1.2)) < 1e-3:
            continue   # too close to a kink
        p, m = lp_new.copy(), lp_new.copy()
        p[b, k] += h
        m[b, k] -= h
        fd = (grpo.grpo_loss(p, lp_old, adv)[0] - grpo.grpo_loss(m, lp_old, adv)[0]) / (2 * h)
        assert g[b, k] == pytest.approx(fd, abs=1e-8)


def test_multi_reward_single_reward_and_one_hot_weights():
    rng = np.random.default_rng(7)
    G, ng, K = 4, 3, 3
    R = rng.random((G * ng, K))
    for mode in ("weighted_sum", "per_reward"):
        # K = 1 with weight 1 is the single-reward advantage
        np.testing.assert_allclose(grpo.group_advantage_multi(R[:, :1], G, [1.0], mode),
                                   grpo.group_advantage(R[:, 0], G), rtol=1e-14)
        # a one-hot weight picks that reward
        np.testing.assert_allclose(grpo.group_advantage_multi(R, G, [0.0, 1.0, 0.0], mode),
                                   grpo.group_advantage(R[:, 1], G), rtol=1e-14, atol=1e-15)


def test_multi_reward_modes_differ_and_follow_their_definitions():
    rng = np.random.default_rng(8)
    G, ng, K = 5, 2, 2
    R = rng.random((G * ng, K)) * np.array([1.0, 100.0])   # rewards on very different scales
    w = np.array([0.7, 0.3])
    ws = grpo.group_advantage_multi(R, G, w, "weighted_sum")
    pr = grpo.group_advantage_multi(R, G, w, "per_reward")
    # brute force, one group at a time
    for g in range(ng):
        rows = slice(g * G, (g + 1) * G)
        r = R[rows] @ w
        np.testing.assert_allclose(ws[rows], (r - r.mean()) / (r.std() + 1e-4), rtol=1e-13)
        want = sum(w[k] * (R[rows, k] - R[rows, k].mean()) / (R[rows, k].std() + 1e-4) for k in range(K))
        np.testing.assert_allclose(pr[rows], want, rtol=1e-13)
    # the weighted sum is dominated by the large-scale reward, per-reward normalisation is not
    assert np.max(np.abs(ws - pr)) > 0.1
    np.testing.assert_allclose(pr.reshape(ng, G).mean(axis=1), 0.0, atol=1e-13)


def test_step_weights_reduce_to_plain_grpo_and_drop_steps():
    rng = np.random.default_rng(9)
    B, T = 3, 4
    lp_new, lp_old = rng.standard_normal((B, T)) * 0.1, rng.standard_normal((B, T)) * 0.1
    adv = rng.standard_normal(B)
    l1, g1 = grpo.grpo_loss(lp_new, lp_old, adv)
    lw, gw = grpo.grpo_loss(lp_new, lp_old, adv, step_w=np.ones(T))
    assert lw == l1 and np.array_equal(gw, g1)
    # weight 0 on steps 1..3 leaves step 0 only, still averaged over B * T
    w = np.array([1.0, 0.0, 0.0, 0.0])
    l0, g0 = grpo.grpo_loss(lp_new, lp_old, adv, step_w=w)
    ls, _ = grpo.grpo_loss(lp_new[:, :1], lp_old[:, :1], adv)
    assert l0 == pytest.approx(ls / T, rel=1e-14)
    assert np.all(g0[:, 1:] == 0.0)
    # linear in the weights, gradient by central differences
    w2 = rng.random(T)
    lw2, gw2 = grpo.grpo_loss(lp_new, lp_old, adv, step_w=w2)
    h = 1e-7
    for b in range(B):
        for k in range(T):
            p, m = lp_new.copy(), lp_new.copy()
            p[b, k] += h
            m[b, k] -= h
            fd = (grpo.grpo_loss(p, lp_old, adv, step_w=w2)[0] - grpo.grpo_loss(m, lp_old, adv, step_w=w2)[0]) / (2 * h)
            assert gw2[b, k] == pytest.approx(fd, rel=1e-5, abs=1e-10)
