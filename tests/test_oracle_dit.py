"""Pins of the fp64 oracle for the MMDiT velocity pieces: attention, RoPE,
norms, activations, timestep embedding, modulation, and whole-model invariants."""
import math

import numpy as np
import pytest
import scipy.special

import synth
from oracle import dit

TINY = dict(name="pin", arch="mmdit", hidden=64, heads=2, head_dim=32, mlp=128,
            n_double=1, n_single=1, patch_dim=16, txt_dim=48, n_txt=5, grid=(1, 3, 4),
            rope_axes=(4, 14, 14), rope_theta=10000.0, time_freq_dim=32, batch=2)


def _params(cfg, seed=0, **kw):
    kw.setdefault("bias_std", 0.05)
    kw.setdefault("scale_std", 0.1)
    return dit.widen_params(synth.weights(dit.param_specs(cfg), seed=seed, std=0.1, **kw))


def _inputs(cfg, seed=3):
    rng = np.random.default_rng(seed)
    B = cfg["batch"]
    x = rng.standard_normal((B, synth.n_img(cfg), cfg["patch_dim"]))
    txt = rng.standard_normal((B, cfg["n_txt"], cfg["txt_dim"]))
    t = rng.uniform(0.1, 1.0, B)
    return x, txt, t


# ---------------------------------------------------------------- attention

def _attention_loop(q, k, v):
    nq, nh, d = q.shape
    out = np.zeros((nq, nh, v.shape[-1]))
    for h in range(nh):
        for i in range(nq):
            scores = [sum(q[i, h, c] * k[j, h, c] for c in range(d)) / math.sqrt(d)
                      for j in range(k.shape[0])]
            m = max(scores)
            w = [math.exp(s - m) for s in scores]
            z = sum(w)
            for j in range(k.shape[0]):
                out[i, h] += w[j] / z * v[j, h]
    return out


def test_attention_matches_explicit_loops():
    rng = np.random.default_rng(0)
    q, k, v = rng.standard_normal((3, 7, 2, 8))
    np.testing.assert_allclose(dit.attention(q, k, v, q_chunk=3), _attention_loop(q, k, v), rtol=1e-12)


def test_attention_special_cases():
    rng = np.random.default_rng(1)
    nk, d = 9, 16
    v = rng.standard_normal((nk, 1, d))
    q = rng.standard_normal((4, 1, d))
    k_same = np.repeat(rng.standard_normal((1, 1, d)), nk, axis=0)
    np.testing.assert_allclose(dit.attention(q, k_same, v), np.repeat(v.mean(0, keepdims=True), 4, 0), rtol=1e-12)
    k = rng.standard_normal((nk, 1, d))
    np.testing.assert_allclose(dit.attention(np.zeros((2, 1, d)), k, v), np.repeat(v.mean(0, keepdims=True), 2, 0), rtol=1e-12)
    # a key aligned with a huge query wins: output is that key's value
    k = np.zeros((nk, 1, d))
    k[5, 0, 0] = 1.0
    qp = np.zeros((1, 1, d))
    qp[0, 0, 0] = 1e4
    np.testing.assert_allclose(dit.attention(qp, k, v)[0, 0], v[5, 0], rtol=1e-12)


# --------------------------------------------------------------------- RoPE

def test_rope_properties():
    rng = np.random.default_rng(2)
    axes = (4, 14, 14)
    x = rng.standard_normal((6, 2, 32))
    pos = rng.integers(0, 50, (6, 3)).astype(float)
    y = dit.apply_rope(x, dit.rope_angles(pos, axes))
    np.testing.assert_allclose(np.linalg.norm(y, axis=-1), np.linalg.norm(x, axis=-1), rtol=1e-13)
    z = dit.apply_rope(x, dit.rope_angles(np.zeros((6, 3)), axes))
    np.testing.assert_array_equal(z, x)
    # <R_m q, R_n k> depends only on m - n (per axis)
    q, k = rng.standard_normal((2, 1, 1, 32))
    def dot(m, n):
        a = dit.apply_rope(q, dit.rope_angles(np.array([m], float), axes))
        b = dit.apply_rope(k, dit.rope_angles(np.array([n], float), axes))
        return float((a * b).sum())
    assert dot([1, 5, 9], [0, 2, 4]) == pytest.approx(dot([11, 13, 20], [10, 10, 15]), rel=1e-10)


def test_rope_single_pair_rotation():
    # axis of width 2 at theta^0 = 1: a plain 2-D rotation by the position
    x = np.array([[[1.0, 0.0]]])
    y = dit.apply_rope(x, dit.rope_angles(np.array([[math.pi / 2]]), (2,)))
    np.testing.assert_allclose(y[0, 0], [0.0, 1.0], atol=1e-15)


def test_image_positions():
    p = dit.image_positions((2, 3, 4))
    assert p.shape == (24, 3)
    np.testing.assert_array_equal(p[0], [0, 0, 0])
    np.testing.assert_array_equal(p[5], [0, 1, 1])
    np.testing.assert_array_equal(p[23], [1, 2, 3])


# ------------------------------------------------------ norms / activations

def test_layer_norm_and_rms_norm():
    rng = np.random.default_rng(3)
    x = rng.standard_normal((5, 64)) * 3 + 1
    y = dit.layer_norm(x)
    np.testing.assert_allclose(y.mean(-1), 0, atol=1e-14)
    var = x.var(-1)
    np.testing.assert_allclose(y.var(-1), var / (var + dit.LN_EPS), rtol=1e-12)
    r = dit.rms_norm(x, np.full(64, 2.5))
    ms = (x ** 2).mean(-1)
    np.testing.assert_allclose(np.sqrt((r ** 2).mean(-1)), 2.5 * np.sqrt(ms / (ms + dit.RMS_EPS)), rtol=1e-12)


def test_gelu_tanh_within_known_bound_of_exact_gelu():
    x = np.linspace(-8, 8, 4001)
    exact = 0.5 * x * (1 + scipy.special.erf(x / math.sqrt(2)))
    assert np.max(np.abs(dit.gelu_tanh(x) - exact)) < 1e-3
    assert dit.gelu_tanh(np.array([0.0]))[0] == 0.0


def test_silu():
    x = np.linspace(-20, 20, 101)
    np.testing.assert_allclose(dit.silu(x), x * scipy.special.expit(x), rtol=1e-13, atol=1e-300)


def test_timestep_embedding():
    e = dit.timestep_embedding(np.array([0.0, 1.0]), 8)
    np.testing.assert_array_equal(e[0], [1, 1, 1, 1, 0, 0, 0, 0])
    # frequency 0 is 1: the first cos/sin pair sees 1000 t radians
    assert e[1, 0] == pytest.approx(math.cos(1000.0))
    assert e[1, 4] == pytest.approx(math.sin(1000.0))
    # last frequency of 4 is 1e4^(-3/4)
    assert e[1, 3] == pytest.approx(math.cos(1000.0 * 1e4 ** -0.75))


# ------------------------------------------------------------- whole model

def test_param_count_of_qwen_shaped_model():
    c = synth.config("qwen_image_60d")
    n = sum(int(np.prod(s)) for _, s in dit.param_specs(c))
    H, F = 3072, 12288
    per_block = 2 * (4 * H * H + 2 * H * F + 3 * H + H + F + H + 2 * 128) + 12 * H * H + 12 * H
    assert n > 60 * per_block
    assert 20.0e9 < n < 20.8e9


def test_zero_modulation_makes_blocks_identity():
    cfg = dict(TINY)
    P = _params(cfg)
    P["mod.w"][:] = 0.0
    P["mod.b"][:] = 0.0
    x, txt, t = _inputs(cfg)
    v = dit.velocity(P, cfg, x, txt, t)
    want = dit.linear(dit.layer_norm(dit.linear(x, P["img_in.w"], P["img_in.b"])), P["final.w"], P["final.b"])
    np.testing.assert_allclose(v, want, rtol=1e-12, atol=1e-14)


def test_velocity_invariants():
    cfg = dict(TINY)
    P = _params(cfg)
    x, txt, t = _inputs(cfg)
    v = dit.velocity(P, cfg, x, txt, t)
    assert v.shape == x.shape
    # text tokens all sit at RoPE position 0: permuting them leaves v unchanged
    perm = np.random.default_rng(9).permutation(cfg["n_txt"])
    np.testing.assert_allclose(dit.velocity(P, cfg, x, txt[:, perm], t), v, rtol=1e-11, atol=1e-13)
    # samples are independent
    v1 = dit.velocity(P, cfg, x[1:], txt[1:], t[1:])
    np.testing.assert_allclose(v1[0], v[1], rtol=1e-12, atol=1e-14)
    # restricting the output rows changes nothing in them
    rows = np.array([0, 7, 11])
    np.testing.assert_allclose(dit.velocity(P, cfg, x, txt, t, img_rows=rows), v[:, rows], rtol=1e-12, atol=1e-14)
    cfg_d = dict(cfg, n_single=0)
    Pd = _params(cfg_d)
    vd = dit.velocity(Pd, cfg_d, x, txt, t)
    np.testing.assert_allclose(dit.velocity(Pd, cfg_d, x, txt, t, img_rows=rows), vd[:, rows], rtol=1e-12, atol=1e-14)
    # moving image tokens changes v (RoPE is live)
    x2 = x.copy()
    x2[:, [0, 5]] = x2[:, [5, 0]]
    v2 = dit.velocity(P, cfg, x2, txt, t)
    assert np.abs(v2[:, 0] - v[:, 5]).max() > 1e-6


# ------------------------------------------------------------------ WAN

WAN_TINY = dict(name="wan_pin", arch="wan", hidden=64, heads=2, head_dim=32, mlp=96, n_double=2, n_single=0,
                patch_dim=16, txt_dim=40, n_txt=6, grid=(2, 3, 4), rope_axes=(12, 10, 10), rope_theta=10000.0,
                time_freq_dim=32, batch=2)


def _wan_params(cfg, seed=0):
    return dit.widen_params(synth.weights(dit.wan_param_specs(cfg), seed=seed, std=0.1, bias_std=0.05,
                                          scale_std=0.1))


def test_wan_zero_modulation_and_cross_weights_give_closed_form():
    # gates 0 and a zero cross-attention output projection make every block
    # the identity, so v = final(LN-modulated embedding) with (shift, scale) = e + b_final
    cfg = dict(WAN_TINY)
    P = _wan_params(cfg)
    P["mod.w"][:] = 0.0
    P["mod.b"][:] = 0.0
    for l in range(cfg["n_double"]):
        P[f"blocks.{l}.mod.b"][:] = 0.0
        P[f"blocks.{l}.cross_proj.w"][:] = 0.0
        P[f"blocks.{l}.cross_proj.b"][:] = 0.0
    x, txt, t = _inputs(cfg)
    v = dit.wan_velocity(P, cfg, x, txt, t)
    emb = dit.timestep_embedding(t, cfg["time_freq_dim"])
    e = dit.linear(dit.silu(dit.linear(emb, P["t_embed.fc1.w"], P["t_embed.fc1.b"])), P["t_embed.fc2.w"],
                   P["t_embed.fc2.b"])
    H = cfg["hidden"]
    for b in range(x.shape[0]):
        xe = dit.linear(x[b], P["img_in.w"], P["img_in.b"])
        h = dit.modulate(dit.layer_norm(xe), e[b] + P["final.mod.b"][:H], e[b] + P["final.mod.b"][H:])
        np.testing.assert_allclose(v[b], dit.linear(h, P["final.w"], P["final.b"]), rtol=1e-12, atol=1e-14)


def test_wan_invariants():
    cfg = dict(WAN_TINY)
    P = _wan_params(cfg)
    x, txt, t = _inputs(cfg)
    v = dit.wan_velocity(P, cfg, x, txt, t)
    assert v.shape == x.shape
    # text tokens enter only through (unrotated) cross-attention keys/values:
    # their order does not matter
    perm = np.random.default_rng(3).permutation(cfg["n_txt"])
    np.testing.assert_allclose(dit.wan_velocity(P, cfg, x, txt[:, perm], t), v, rtol=1e-11, atol=1e-13)
    v1 = dit.wan_velocity(P, cfg, x[1:], txt[1:], t[1:])
    np.testing.assert_allclose(v1[0], v[1], rtol=1e-12, atol=1e-14)
    rows = np.array([1, 13, 23])
    np.testing.assert_allclose(dit.wan_velocity(P, cfg, x, txt, t, img_rows=rows), v[:, rows], rtol=1e-12,
                               atol=1e-14)
    # the frame axis is live: swapping two frames' tokens changes v
    x2 = x.copy()
    x2[:, [0, 12]] = x2[:, [12, 0]]
    assert np.abs(dit.wan_velocity(P, cfg, x2, txt, t)[:, 0] - v[:, 12]).max() > 1e-6


def test_wan_param_count():
    c = synth.config("wan_40")
    n = sum(int(np.prod(s)) for _, s in dit.wan_param_specs(c))
    H, F = 5120, 13824
    per_block = 8 * H * H + 2 * H * F
    assert 40 * per_block < n < 40 * per_block * 1.02


def test_attention_backward_central_differences():
    """The attention backward against central differences of the scalar
    sum(dO * attention(q, k, v)); rowsum(dP P) = rowsum(dO O) is the D of
    the backward."""
    rng = np.random.default_rng(21)
    nq, nk, nh, d = 3, 4, 2, 4
    q, k, v, g = (rng.standard_normal((nq, nh, d)), rng.standard_normal((nk, nh, d)),
                  rng.standard_normal((nk, nh, d)), rng.standard_normal((nq, nh, d)))
    dq, dk, dv = dit.attention_backward(q, k, v, g)
    loss = lambda q_, k_, v_: float(np.sum(g * dit.attention(q_, k_, v_)))
    h = 1e-6
    for arr, grad in ((q, dq), (k, dk), (v, dv)):
        it = np.nditer(arr, flags=["multi_index"])
        for _ in it:
            i = it.multi_index
            p_, m_ = arr.copy(), arr.copy()
            p_[i] += h
            m_[i] -= h
            pick = lambda a_: [a_ if arr is x else x for x in (q, k, v)]
            fd = (loss(*pick(p_)) - loss(*pick(m_))) / (2 * h)
            assert grad[i] == pytest.approx(fd, rel=1e-6, abs=1e-8)


def test_attention_lse_matches_logsumexp():
    from scipy.special import logsumexp
    rng = np.random.default_rng(22)
    q, k = rng.standard_normal((5, 2, 8)) * 3, rng.standard_normal((7, 2, 8)) * 3
    got = dit.attention_lse(q, k)
    for hh in range(2):
        want = logsumexp(q[:, hh, :] @ k[:, hh, :].T / math.sqrt(8), axis=1)
        np.testing.assert_allclose(got[:, hh], want, rtol=1e-13)
