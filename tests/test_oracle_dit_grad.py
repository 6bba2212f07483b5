"""Pins of the fp64 MMDiT gradient (oracle/dit_grad.py) and of the log-prob
gradient (oracle/sde.py): every elementary backward and the whole
vector-Jacobian product against central differences of the forward."""
import numpy as np
import pytest

import synth
from oracle import dit, dit_grad, sde

TINY = dict(name="grad", arch="mmdit", hidden=32, heads=2, head_dim=16, mlp=64,
            n_double=1, n_single=1, patch_dim=8, txt_dim=24, n_txt=3, grid=(1, 2, 3),
            rope_axes=(4, 6, 6), rope_theta=100.0, time_freq_dim=16, batch=2)


def _params(cfg, seed=0):
    return dit.widen_params(synth.weights(dit.param_specs(cfg), seed=seed, std=0.2,
                                          bias_std=0.1, scale_std=0.2))


def _inputs(cfg, seed=3):
    rng = np.random.default_rng(seed)
    B = cfg["batch"]
    return (rng.standard_normal((B, synth.n_img(cfg), cfg["patch_dim"])),
            rng.standard_normal((B, cfg["n_txt"], cfg["txt_dim"])),
            rng.uniform(0.1, 0.9, B))


def _central(f, x, dx, h=1e-5):
    return (f(x + h * dx) - f(x - h * dx)) / (2 * h)


def _check_vjp(f, x, dy, grad, rng, trials=3, rtol=1e-6):
    """<grad, dx> against the directional derivative of <dy, f> along dx."""
    for _ in range(trials):
        dx = rng.standard_normal(np.shape(x))
        num = _central(lambda z: float(np.sum(dy * f(z))), x, dx)
        ana = float(np.sum(grad * dx))
        assert abs(num - ana) <= rtol * max(1.0, abs(num)), (num, ana)


# ---------------------------------------------------------------- elementary backwards

def test_linear_bwd():
    rng = np.random.default_rng(0)
    x, w, b = rng.standard_normal((5, 7)), rng.standard_normal((4, 7)), rng.standard_normal(4)
    dy = rng.standard_normal((5, 4))
    dx, dw, db = dit_grad.linear_bwd(x, w, dy)
    _check_vjp(lambda z: dit.linear(z, w, b), x, dy, dx, rng)
    _check_vjp(lambda z: dit.linear(x, z, b), w, dy, dw, rng)
    _check_vjp(lambda z: dit.linear(x, w, z), b, dy, db, rng)


def test_layer_norm_bwd():
    rng = np.random.default_rng(1)
    x = rng.standard_normal((6, 12)) * 2 + 0.5
    dy = rng.standard_normal((6, 12))
    _check_vjp(dit.layer_norm, x, dy, dit_grad.layer_norm_bwd(x, dy), rng)


def test_layer_norm_bwd_is_orthogonal_to_shift_and_scale():
    # LN is invariant to x -> a x + c per row, so the gradient has zero row
    # sum and is orthogonal to x - mean
    rng = np.random.default_rng(2)
    x = rng.standard_normal((4, 16))
    g = dit_grad.layer_norm_bwd(x, rng.standard_normal((4, 16)))
    np.testing.assert_allclose(g.sum(axis=1), 0, atol=1e-10)
    np.testing.assert_allclose((g * (x - x.mean(axis=1, keepdims=True))).sum(axis=1), 0, atol=1e-5)


def test_modulate_bwd():
    rng = np.random.default_rng(3)
    n, sh, sc = rng.standard_normal((5, 8)), rng.standard_normal(8), rng.standard_normal(8)
    dy = rng.standard_normal((5, 8))
    dn, dsh, dsc = dit_grad.modulate_bwd(n, sc, dy)
    _check_vjp(lambda z: dit.modulate(z, sh, sc), n, dy, dn, rng)
    _check_vjp(lambda z: dit.modulate(n, z, sc), sh, dy, dsh, rng)
    _check_vjp(lambda z: dit.modulate(n, sh, z), sc, dy, dsc, rng)


def test_rms_norm_bwd():
    rng = np.random.default_rng(4)
    x, w = rng.standard_normal((5, 3, 16)), rng.standard_normal(16)
    dy = rng.standard_normal((5, 3, 16))
    dx, dw = dit_grad.rms_norm_bwd(x, w, dy)
    _check_vjp(lambda z: dit.rms_norm(z, w), x, dy, dx, rng)
    _check_vjp(lambda z: dit.rms_norm(x, z), w, dy, dw, rng)


def test_rope_bwd_is_the_inverse_rotation():
    rng = np.random.default_rng(5)
    x, ang = rng.standard_normal((6, 2, 8)), rng.uniform(-3, 3, (6, 4))
    dy = rng.standard_normal((6, 2, 8))
    _check_vjp(lambda z: dit.apply_rope(z, ang), x, dy, dit_grad.rope_bwd(dy, ang), rng)
    # a rotation: the backward undoes the forward
    np.testing.assert_allclose(dit_grad.rope_bwd(dit.apply_rope(x, ang), ang), x, atol=1e-12)


@pytest.mark.parametrize("fn,grad", [(dit.gelu_tanh, dit_grad.gelu_tanh_grad), (dit.silu, dit_grad.silu_grad)])
def test_activation_grads(fn, grad):
    x = np.linspace(-6, 6, 97)
    h = 1e-6
    np.testing.assert_allclose(grad(x), (fn(x + h) - fn(x - h)) / (2 * h), atol=1e-8)


def test_activation_grad_special_values():
    # GELU'(0) = 1/2, SiLU'(0) = 1/2; both tend to 1 for large x and 0 for very negative x
    assert dit_grad.gelu_tanh_grad(np.array([0.0]))[0] == pytest.approx(0.5)
    assert dit_grad.silu_grad(np.array([0.0]))[0] == pytest.approx(0.5)
    np.testing.assert_allclose(dit_grad.gelu_tanh_grad(np.array([30.0, -30.0])), [1.0, 0.0], atol=1e-12)
    np.testing.assert_allclose(dit_grad.silu_grad(np.array([60.0, -60.0])), [1.0, 0.0], atol=1e-12)


# ---------------------------------------------------------------- the whole network

def _cfg(**kw):
    c = dict(TINY)
    c.update(kw)
    return c


@pytest.mark.parametrize("nd,ns", [(1, 1), (2, 0), (0, 2)])
def test_velocity_vjp_matches_central_differences(nd, ns):
    cfg = _cfg(n_double=nd, n_single=ns)
    P = _params(cfg)
    x, txt, t = _inputs(cfg)
    rng = np.random.default_rng(11)
    dv = rng.standard_normal((cfg["batch"], synth.n_img(cfg), cfg["patch_dim"]))
    v, G, dx = dit_grad.velocity_vjp(P, cfg, x, txt, t, dv)
    # the forward it reverses is the oracle's velocity
    np.testing.assert_allclose(v, dit.velocity(P, cfg, x, txt, t), rtol=1e-12, atol=1e-12)

    def loss(Pm, xm=x):
        return float(np.sum(dv * dit.velocity(Pm, cfg, xm, txt, t)))

    h = 1e-5
    # one direction per tensor: a dropped or mis-signed term in any tensor's
    # gradient shows up in its own check
    for name in P:
        d = rng.standard_normal(P[name].shape)
        Pp, Pm = dict(P), dict(P)
        Pp[name] = P[name] + h * d
        Pm[name] = P[name] - h * d
        num = (loss(Pp) - loss(Pm)) / (2 * h)
        ana = float(np.sum(G[name] * d))
        assert abs(num - ana) <= 1e-6 * max(1.0, abs(num)), (name, num, ana)
    d = rng.standard_normal(x.shape)
    num = (loss(P, x + h * d) - loss(P, x - h * d)) / (2 * h)
    assert abs(num - float(np.sum(dx * d))) <= 1e-6 * max(1.0, abs(num))


def test_velocity_vjp_is_linear_in_dv():
    cfg = _cfg()
    P = _params(cfg, seed=1)
    x, txt, t = _inputs(cfg, seed=4)
    rng = np.random.default_rng(12)
    shape = (cfg["batch"], synth.n_img(cfg), cfg["patch_dim"])
    d1, d2 = rng.standard_normal(shape), rng.standard_normal(shape)
    _, G1, _ = dit_grad.velocity_vjp(P, cfg, x, txt, t, d1)
    _, G2, _ = dit_grad.velocity_vjp(P, cfg, x, txt, t, d2)
    _, G3, _ = dit_grad.velocity_vjp(P, cfg, x, txt, t, 2 * d1 - d2)
    for k in P:
        np.testing.assert_allclose(G3[k], 2 * G1[k] - G2[k], atol=1e-10)
    _, G0, dx0 = dit_grad.velocity_vjp(P, cfg, x, txt, t, np.zeros(shape))
    assert all(not np.any(g) for g in G0.values()) and not np.any(dx0)


def test_final_bias_gradient_is_the_token_sum_of_dv():
    cfg = _cfg()
    P = _params(cfg, seed=2)
    x, txt, t = _inputs(cfg, seed=5)
    dv = np.random.default_rng(13).standard_normal((cfg["batch"], synth.n_img(cfg), cfg["patch_dim"]))
    _, G, _ = dit_grad.velocity_vjp(P, cfg, x, txt, t, dv)
    np.testing.assert_allclose(G["final.b"], dv.sum(axis=(0, 1)), rtol=1e-13)


# ---------------------------------------------------------------- the log-prob gradient

@pytest.mark.parametrize("reduce", ["sum", "mean"])
def test_sde_logprob_grad_v(reduce):
    rng = np.random.default_rng(20)
    B, D = 3, 40
    x, v = rng.standard_normal((B, D)), rng.standard_normal((B, D))
    t = np.array([0.9, 0.5, 0.3])
    tn = t - np.array([0.1, 0.2, 0.3])
    sig = np.array([0.7, 0.4, 0.0])          # the last step is deterministic: zero gradient
    x_next = x + rng.standard_normal((B, D)) * 0.3
    g = sde.sde_logprob_grad_v(x, v, x_next, t, tn, sig, reduce)
    for b in range(B):
        def lp(vb):
            vv = v.copy()
            vv[b] = vb
            return sde.sde_step_logprob(x, vv, t, tn, sig, x_next=x_next, reduce=reduce)[1][b]
        d = rng.standard_normal(D)
        num = (lp(v[b] + 1e-6 * d) - lp(v[b] - 1e-6 * d)) / 2e-6
        assert num == pytest.approx(float(g[b] @ d), rel=1e-6, abs=1e-9)
    assert not np.any(g[2])


def test_sde_logprob_grad_zero_at_the_mean():
    # a sample drawn at the mean is the density's maximum: zero gradient in v
    rng = np.random.default_rng(21)
    x, v = rng.standard_normal((2, 16)), rng.standard_normal((2, 16))
    t, tn, sig = np.array([0.8, 0.6]), np.array([0.6, 0.3]), np.array([0.5, 0.9])
    x_mean, _ = sde.sde_step_logprob(x, v, t, tn, sig, eps=np.zeros((2, 16)))
    np.testing.assert_allclose(sde.sde_logprob_grad_v(x, v, x_mean, t, tn, sig), 0, atol=1e-12)


# ---------------------------------------------------------------- the WAN-style network

WAN_TINY = dict(name="wan_grad", arch="wan", hidden=32, heads=2, head_dim=16, mlp=64,
                n_double=2, n_single=0, patch_dim=8, txt_dim=24, n_txt=3, grid=(2, 2, 3),
                rope_axes=(4, 6, 6), rope_theta=100.0, time_freq_dim=16, batch=2)


def _wan_params(cfg, seed=0):
    return dit.widen_params(synth.weights(dit.wan_param_specs(cfg), seed=seed, std=0.2,
                                          bias_std=0.1, scale_std=0.2))


@pytest.mark.parametrize("L", [1, 2])
def test_wan_velocity_vjp_matches_central_differences(L):
    cfg = dict(WAN_TINY, n_double=L)
    P = _wan_params(cfg)
    x, txt, t = _inputs(cfg)
    rng = np.random.default_rng(21)
    dv = rng.standard_normal((cfg["batch"], synth.n_img(cfg), cfg["patch_dim"]))
    v, G, dx = dit_grad.wan_velocity_vjp(P, cfg, x, txt, t, dv)
    np.testing.assert_allclose(v, dit.wan_velocity(P, cfg, x, txt, t), rtol=1e-12, atol=1e-12)

    def loss(Pm, xm=x):
        return float(np.sum(dv * dit.wan_velocity(Pm, cfg, xm, txt, t)))

    h = 1e-5
    for name in P:
        d = rng.standard_normal(P[name].shape)
        Pp, Pm = dict(P), dict(P)
        Pp[name] = P[name] + h * d
        Pm[name] = P[name] - h * d
        num = (loss(Pp) - loss(Pm)) / (2 * h)
        ana = float(np.sum(G[name] * d))
        assert abs(num - ana) <= 1e-6 * max(1.0, abs(num)), (name, num, ana)
    d = rng.standard_normal(x.shape)
    num = (loss(P, x + h * d) - loss(P, x - h * d)) / (2 * h)
    assert abs(num - float(np.sum(dx * d))) <= 1e-6 * max(1.0, abs(num))


def test_wan_velocity_vjp_is_linear_in_dv():
    cfg = WAN_TINY
    P = _wan_params(cfg, seed=1)
    x, txt, t = _inputs(cfg, seed=4)
    rng = np.random.default_rng(22)
    shape = (cfg["batch"], synth.n_img(cfg), cfg["patch_dim"])
    d1, d2 = rng.standard_normal(shape), rng.standard_normal(shape)
    _, G1, x1 = dit_grad.wan_velocity_vjp(P, cfg, x, txt, t, d1)
    _, G2, x2 = dit_grad.wan_velocity_vjp(P, cfg, x, txt, t, d2)
    _, G3, x3 = dit_grad.wan_velocity_vjp(P, cfg, x, txt, t, 2 * d1 - d2)
    for k in P:
        np.testing.assert_allclose(G3[k], 2 * G1[k] - G2[k], atol=1e-10)
    np.testing.assert_allclose(x3, 2 * x1 - x2, atol=1e-10)


def test_wan_bias_gradients_are_token_sums():
    """final.b sums dv over every token; the final layer's shift bias
    (final.mod.b[:H]) sums the final LN-modulate input gradient, which is
    dv W_final; and a block's modulation bias gradient equals the
    shared-modulation gradient summed over the blocks' own contributions."""
    cfg = WAN_TINY
    P = _wan_params(cfg, seed=2)
    x, txt, t = _inputs(cfg, seed=5)
    dv = np.random.default_rng(23).standard_normal((cfg["batch"], synth.n_img(cfg), cfg["patch_dim"]))
    _, G, _ = dit_grad.wan_velocity_vjp(P, cfg, x, txt, t, dv)
    H = cfg["hidden"]
    np.testing.assert_allclose(G["final.b"], dv.sum(axis=(0, 1)), rtol=1e-13)
    np.testing.assert_allclose(G["final.mod.b"][:H], (dv @ P["final.w"]).sum(axis=(0, 1)), rtol=1e-12)
    # mod.b receives what every block's bias receives (e0 + b_l: same partials)
    np.testing.assert_allclose(G["mod.b"], sum(G[f"blocks.{l}.mod.b"] for l in range(cfg["n_double"])),
                               rtol=1e-12, atol=1e-14)


# ---------------------------------------------------------------- the pins catch planted mistakes

def _worst_mismatch(vjp, vel, cfg, P):
    """Largest |numeric - analytic| / max(1, |numeric|) over one random
    direction per parameter tensor and one for x_t."""
    x, txt, t = _inputs(cfg)
    rng = np.random.default_rng(31)
    dv = rng.standard_normal((cfg["batch"], synth.n_img(cfg), cfg["patch_dim"]))
    _, G, dx = vjp(P, cfg, x, txt, t, dv)

    def loss(Pm, xm=x):
        return float(np.sum(dv * vel(Pm, cfg, xm, txt, t)))

    h, worst = 1e-5, 0.0
    for name in P:
        d = rng.standard_normal(P[name].shape)
        Pp, Pm = dict(P), dict(P)
        Pp[name] = P[name] + h * d
        Pm[name] = P[name] - h * d
        num = (loss(Pp) - loss(Pm)) / (2 * h)
        worst = max(worst, abs(num - float(np.sum(G[name] * d))) / max(1.0, abs(num)))
    d = rng.standard_normal(x.shape)
    num = (loss(P, x + h * d) - loss(P, x - h * d)) / (2 * h)
    return max(worst, abs(num - float(np.sum(dx * d))) / max(1.0, abs(num)))


def _ln_no_projection(x, dn, eps=dit.LN_EPS):
    mu = x.mean(axis=-1, keepdims=True)
    s = np.sqrt(((x - mu) ** 2).mean(axis=-1, keepdims=True) + eps)
    return (dn - dn.mean(axis=-1, keepdims=True)) / s          # drops - n mean(dn n)


_RMS_BWD = dit_grad.rms_norm_bwd


def _rms_sign(x, w, dy, eps=dit.RMS_EPS):
    dx, dw = _RMS_BWD(x, w, dy, eps)
    return dx, -dw                                              # wrong sign of the scale gradient


def _rope_untransposed(dy, angles):
    return dit.apply_rope(dy, angles)                          # rotation not transposed


def _silu_half(x):
    return 1.0 / (1.0 + np.exp(-x))                            # drops the x sigma (1 - sigma) term


def _gelu_no_cubic(x):
    th = np.tanh(np.sqrt(2.0 / np.pi) * (x + 0.044715 * x ** 3))
    return 0.5 * (1.0 + th) + 0.5 * x * (1.0 - th * th) * np.sqrt(2.0 / np.pi)   # drops 3 c x^2


def _modulate_no_scale(n, scale, dy):
    return dy, dy.sum(axis=0), (dy * n).sum(axis=0)             # drops the (1 + scale) factor


@pytest.mark.parametrize("arch", ["mmdit", "wan"])
@pytest.mark.parametrize("target,wrong", [("layer_norm_bwd", _ln_no_projection), ("rms_norm_bwd", _rms_sign),
                                          ("rope_bwd", _rope_untransposed), ("silu_grad", _silu_half),
                                          ("gelu_tanh_grad", _gelu_no_cubic), ("modulate_bwd", _modulate_no_scale)])
def test_planted_mistakes_fail_the_central_difference_pin(monkeypatch, arch, target, wrong):
    if arch == "wan":
        cfg, P = dict(WAN_TINY, n_double=1), _wan_params(dict(WAN_TINY, n_double=1))
        vjp, vel = dit_grad.wan_velocity_vjp, dit.wan_velocity
    else:
        cfg = _cfg()
        P, vjp, vel = _params(cfg), dit_grad.velocity_vjp, dit.velocity
    assert _worst_mismatch(vjp, vel, cfg, P) <= 1e-6
    monkeypatch.setattr(dit_grad, target, wrong)
    assert _worst_mismatch(vjp, vel, cfg, P) > 1e-4
