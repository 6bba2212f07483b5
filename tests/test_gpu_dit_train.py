"""GPU parity of the training pass (ff_dit_forward_train, ff_dit_backward,
ff_sde_logprob_backward) against the fp64 oracle's vector-Jacobian product
(oracle/dit_grad.py), tensor by tensor, on small MMDiTs and WAN-style models;
properties of the Flux-shaped block at full size."""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import dit as odit
from oracle import dit_grad, sde
from oracle import grpo as ogrpo

pytestmark = pytest.mark.gpu

# Per-tensor RMS-relative bound for the gradients: every product runs on
# bf16 operands (unit roundoff 2^-8) with fp32 accumulation, and a gradient
# passes through about ten such roundings between dv and a weight, so the
# relative error grows to about sqrt(10) 2^-8 ~ 1.2e-2; 3e-2 leaves a margin.
G_TOL = 3e-2
V_TOL = 2e-2

SMALL = dict(name="train_small", arch="mmdit", hidden=256, heads=2, head_dim=128, mlp=512,
             n_double=1, n_single=1, patch_dim=64, txt_dim=128, n_txt=16, grid=(1, 4, 8),
             rope_axes=(16, 56, 56), rope_theta=10000.0, time_freq_dim=256, batch=2)


def _cfg(**kw):
    c = dict(SMALL)
    c.update(kw)
    return c


class Run:
    """Model, inputs and one training pass on the GPU."""

    def __init__(self, cfg, dev, seed=0, std=0.05):
        import torch
        from paper_2602_12529_gb300 import ffi, weights
        self.cfg = cfg
        self.W = {}

        def get(name, shape):
            a = synth.weight(name, shape, synth.weight_kind(name), seed, std, 0.05, 0.2)
            self.W[name] = a
            return a

        self.blob = weights.pack(cfg, get, dev)
        self.specs, self.total = weights.layout(cfg)
        self.model = ffi.Dit(cfg, self.blob)
        B = cfg["batch"]
        self.B = B
        self.x = synth.initial_latent(cfg, batch=B)
        self.txt = synth.text_embeds(cfg, batch=B)
        self.t = np.linspace(0.9, 0.35, B).astype(np.float32)
        self.dev = dev
        self.xg = torch.from_numpy(self.x).to(dev)
        self.tg = torch.from_numpy(self.txt.view(np.int16)).to(dev).view(torch.bfloat16)
        self.tt = torch.from_numpy(self.t).to(dev)
        self.ws = torch.empty(self.model.train_workspace_size(B), dtype=torch.uint8, device=dev)
        self.v = torch.empty_like(self.xg)
        self.model.ff_dit_forward_train(self.xg, self.tg, self.tt, self.v, self.ws)

    def backward(self, dv):
        import torch
        from paper_2602_12529_gb300 import ffi
        grad = torch.zeros(self.total, dtype=torch.float32, device=self.dev)
        dx = torch.empty_like(self.xg)
        dvg = dv if isinstance(dv, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(dv, np.float32)).to(self.dev)
        self.model.ff_dit_backward(self.tg, dvg, grad, self.ws, dx_t=dx)
        torch.cuda.synchronize()
        assert ffi.ff_check_device_status() == 0
        return grad.cpu().numpy(), dx.cpu().numpy()

    def tensors(self, grad):
        return {name: grad[off:off + int(np.prod(shape))].reshape(shape) for name, off, shape in self.specs}

    def oracle(self, dv):
        P = odit.widen_params(self.W)
        vjp = dit_grad.wan_velocity_vjp if self.cfg["arch"] == "wan" else dit_grad.velocity_vjp
        return vjp(P, self.cfg, self.x, odit.widen(self.txt), self.t.astype(np.float64), dv)


def _compare(run, grad, dx, want_G, want_dx):
    got = run.tensors(grad)
    errs = {k: rms_rel(got[k], want_G[k]) for k in want_G}
    bad = {k: e for k, e in errs.items() if not e <= G_TOL}
    assert not bad, sorted(bad.items(), key=lambda kv: -kv[1])[:8]
    assert rms_rel(dx, want_dx) <= G_TOL


TINY64 = {k: v for k, v in synth.config("tiny_mmdit").items() if k in SMALL}


@pytest.mark.parametrize("over", [{}, {"n_double": 2, "n_single": 0}, {"n_double": 0, "n_single": 2},
                                  {"grid": (1, 3, 5), "n_txt": 5, "batch": 8},
                                  {"batch": 3, "n_txt": 8, "grid": (1, 4, 6)},
                                  dict(TINY64),
                                  dict(TINY64, n_double=1, n_single=1, grid=(1, 3, 5), n_txt=5, batch=8),
                                  # more than 16 samples: the B-row products (modulation, time MLP) on the
                                  # tensor-core GEMM instead of the row kernels
                                  {"batch": 20, "n_txt": 8, "grid": (1, 2, 4)}])
def test_backward_matches_oracle(cuda, over):
    cfg = _cfg(**over)
    run = Run(cfg, cuda)
    dv = np.random.default_rng(5).standard_normal((cfg["batch"], synth.n_img(cfg), cfg["patch_dim"])).astype(np.float32)
    grad, dx = run.backward(dv)
    v_ref, G, dx_ref = run.oracle(dv.astype(np.float64))
    assert rms_rel(run.v.cpu().numpy(), v_ref) <= V_TOL
    _compare(run, grad, dx, G, dx_ref)


def test_forward_train_equals_velocity_and_backward_is_deterministic(cuda):
    import torch
    cfg = _cfg()
    run = Run(cfg, cuda, seed=1)
    ws = torch.empty(run.model.workspace_size(run.B), dtype=torch.uint8, device=cuda)
    v = torch.empty_like(run.xg)
    run.model.ff_dit_velocity(run.xg, run.tg, run.tt, v, ws)
    torch.cuda.synchronize()
    assert torch.equal(v, run.v)
    dv = np.random.default_rng(6).standard_normal(tuple(v.shape)).astype(np.float32)
    g1, d1 = run.backward(dv)
    g2, d2 = run.backward(dv)
    assert np.array_equal(g1, g2) and np.array_equal(d1, d2)


WAN_TRAIN = dict(name="wan_train", arch="wan", hidden=256, heads=2, head_dim=128, mlp=512, n_double=1,
                 n_single=0, patch_dim=64, txt_dim=128, n_txt=16, grid=(2, 4, 4), rope_axes=(44, 42, 42),
                 rope_theta=10000.0, time_freq_dim=256, batch=2)


@pytest.mark.parametrize("over", [{}, {"n_double": 2},
                                  {"heads": 4, "head_dim": 64, "rope_axes": (20, 22, 22)},
                                  {"grid": (1, 3, 5), "n_txt": 5, "batch": 8},
                                  {"batch": 3, "n_txt": 8, "grid": (2, 2, 6), "n_double": 2},
                                  {"batch": 20, "n_txt": 8, "grid": (1, 2, 4)}])
def test_wan_backward_matches_oracle(cuda, over):
    """The WAN-style block's backward (affine LN, ungated cross-attention with
    text keys / values, shared modulation) against wan_velocity_vjp."""
    cfg = dict(WAN_TRAIN, **over)
    run = Run(cfg, cuda)
    dv = np.random.default_rng(7).standard_normal((cfg["batch"], synth.n_img(cfg), cfg["patch_dim"])).astype(np.float32)
    grad, dx = run.backward(dv)
    v_ref, G, dx_ref = run.oracle(dv.astype(np.float64))
    assert rms_rel(run.v.cpu().numpy(), v_ref) <= V_TOL
    _compare(run, grad, dx, G, dx_ref)


@pytest.mark.parametrize("hidden,over", [
    (4096, {}),
    (5120, {}),
    # latent queries and text keys both past one 128-token tile: 256 latent
    # tokens (two K/V tiles of the self-attention), 160 text tokens (two key
    # tiles of the cross-attention, the second ragged)
    (5120, {"grid": (2, 8, 16), "n_txt": 160, "batch": 1}),
])
def test_wan_backward_matches_oracle_wide_rows(cuda, hidden, over):
    """Rows of 4096 and 5120 columns (the WAN model's width): the LN backward
    runs 512-thread CTAs there.  Few tokens keep the fp64 oracle quick; the
    weight scale shrinks with the width so activations stay O(1).  With
    weights of std 0.01 and biases of std 0.05 the text keys and values are
    nearly parallel, so D = rowsum(dO O) of the cross-attention backward
    subtracts nearly equal terms; D is formed from O to about 16 bits (the
    forward keeps O's bf16 rounding residual), without which the
    cross-attention branch's gradients miss the bound at width 4096."""
    cfg = dict(WAN_TRAIN, hidden=hidden, heads=hidden // 128, grid=(1, 2, 4), n_txt=8, batch=2)
    cfg.update(over)
    run = Run(cfg, cuda, std=0.01)
    dv = np.random.default_rng(7).standard_normal((cfg["batch"], synth.n_img(cfg), cfg["patch_dim"])).astype(np.float32)
    grad, dx = run.backward(dv)
    v_ref, G, dx_ref = run.oracle(dv.astype(np.float64))
    assert rms_rel(run.v.cpu().numpy(), v_ref) <= V_TOL
    _compare(run, grad, dx, G, dx_ref)


def test_wan_forward_train_equals_velocity_and_backward_is_deterministic(cuda):
    import torch
    cfg = dict(WAN_TRAIN, n_double=2)
    run = Run(cfg, cuda, seed=2)
    ws = torch.empty(run.model.workspace_size(run.B), dtype=torch.uint8, device=cuda)
    v = torch.empty_like(run.xg)
    run.model.ff_dit_velocity(run.xg, run.tg, run.tt, v, ws)
    torch.cuda.synchronize()
    assert torch.equal(v, run.v)
    dv = np.random.default_rng(9).standard_normal(tuple(v.shape)).astype(np.float32)
    g1, d1 = run.backward(dv)
    g2, d2 = run.backward(dv)
    assert np.array_equal(g1, g2) and np.array_equal(d1, d2)


@pytest.mark.parametrize("cfg", [dict(WAN_TRAIN, n_double=1), dict(WAN_TRAIN, n_double=3),
                                 _cfg(n_double=2, n_single=0), _cfg(n_double=0, n_single=3),
                                 _cfg(n_double=2, n_single=2, grid=(1, 3, 5), n_txt=5, batch=8)])
@pytest.mark.parametrize("mode", [1, 2])
def test_recompute_gives_the_same_gradient(cuda, cfg, mode):
    """Recompute mode (block inputs kept, each block re-run before its
    backward; mode 1 also keeps the self / joint attention outputs and the
    re-run skips that attention) gives bit for bit the stored-activation
    pass's v and gradients, for WAN-style and MMDiT models."""
    import torch
    from paper_2602_12529_gb300 import ffi
    L = cfg["n_double"] + cfg["n_single"]
    run = Run(cfg, cuda, seed=3)
    dv = np.random.default_rng(10).standard_normal(tuple(run.v.shape)).astype(np.float32)
    g1, d1 = run.backward(dv)
    run.model.set_train_recompute(mode)
    ws = torch.empty(run.model.train_workspace_size(run.B), dtype=torch.uint8, device=cuda)
    assert ws.numel() < run.ws.numel() or L == 1
    v2 = torch.empty_like(run.v)
    run.model.ff_dit_forward_train(run.xg, run.tg, run.tt, v2, ws)
    grad = torch.zeros(run.total, dtype=torch.float32, device=cuda)
    dx = torch.empty_like(run.xg)
    run.model.ff_dit_backward(run.tg, torch.from_numpy(dv).to(cuda), grad, ws, dx_t=dx)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    assert torch.equal(v2, run.v)
    assert np.array_equal(grad.cpu().numpy(), g1) and np.array_equal(dx.cpu().numpy(), d1)
    run.model.set_train_recompute(False)


def test_sde_logprob_backward_parity(cuda):
    import torch
    from paper_2602_12529_gb300 import ffi
    rng = np.random.default_rng(8)
    B, D = 5, 4096 * 3 + 64
    x, v = rng.standard_normal((B, D)).astype(np.float32), rng.standard_normal((B, D)).astype(np.float32)
    t = np.array([0.95, 0.8, 0.5, 0.3, 0.2], np.float32)
    tn = (t - np.array([0.1, 0.2, 0.1, 0.05, 0.2], np.float32)).astype(np.float32)
    sig = np.array([0.7, 0.5, 0.0, 0.9, 0.3], np.float32)
    xn = (x + 0.3 * rng.standard_normal((B, D))).astype(np.float32)
    g = rng.standard_normal((B, 3)).astype(np.float32)      # read with ld = 3 (column 1)
    dev = cuda
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    for reduce, name in ((ffi.FF_LP_SUM, "sum"), (ffi.FF_LP_MEAN, "mean")):
        out = torch.empty(B, D, dtype=torch.float32, device=dev)
        gcol = T(g.ravel()[1:])           # element b * 3 is g[b, 1]
        ffi.ff_sde_logprob_backward(T(x), T(v), T(xn), T(t), T(tn), T(sig), gcol, out, reduce=reduce, ld=3)
        torch.cuda.synchronize()
        want = sde.sde_logprob_grad_v(x, v, xn, t.astype(np.float64), tn.astype(np.float64),
                                      sig.astype(np.float64), name) * g[:, 1:2]
        got = out.cpu().numpy()
        assert not np.any(got[2])
        for b in range(B):
            if sig[b] > 0:
                assert rms_rel(got[b], want[b]) <= 1e-5, (name, b)


def test_grpo_training_step_chain(cuda):
    """One Flow-GRPO training step for a batch: re-score the rollout's
    x_next under the current velocity (forward_train, SDE EVAL log-prob),
    clipped loss and its gradient, then d loss / d theta through
    ff_sde_logprob_backward and ff_dit_backward.  The oracle takes the same
    loss gradient and goes through its own log-prob and network backward."""
    import torch
    from paper_2602_12529_gb300 import ffi
    cfg = _cfg(batch=4, n_txt=8)
    run = Run(cfg, cuda, seed=2)
    B, Ni, Pd = run.B, synth.n_img(cfg), cfg["patch_dim"]
    P = odit.widen_params(run.W)
    t = run.t.astype(np.float64)
    tn = t - 0.1
    sig = sde.sigma_flow_sde(t, 0.7)
    v_o = odit.velocity(P, cfg, run.x, odit.widen(run.txt), t)
    eps = synth.gaussian((B, Ni, Pd), seed=31)
    x_next, _ = sde.sde_step_logprob(run.x, v_o, t, tn, sig, eps=eps)
    x_next = x_next.astype(np.float32)
    dev = cuda
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)
    tg, tng, sg = T(t), T(tn), T(sig)
    lp = torch.empty(B, 1, dtype=torch.float32, device=dev)
    ws = torch.zeros(ffi.ff_sde_workspace_size(B, Ni * Pd), dtype=torch.uint8, device=dev)
    xn_g = T(x_next)
    ffi.ff_sde_step_logprob(run.xg, run.v, None, xn_g, tg, tng, sg, lp, mode=ffi.FF_SDE_EVAL, ws=ws)
    lp_old = lp + T(synth.logprob_jitter((B, 1), seed=9))
    adv = T(synth.gaussian((B,), seed=32))
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    glp = torch.empty(B, 1, dtype=torch.float32, device=dev)
    ffi.ff_grpo_loss(lp, lp_old, adv, 0.2, 0.2, loss, grad_lp_new=glp)
    dv = torch.empty_like(run.xg)
    ffi.ff_sde_logprob_backward(run.xg, run.v, xn_g, tg, tng, sg, glp, dv, ld=1)
    grad, dx = run.backward(dv)
    g = glp.cpu().numpy()[:, 0].astype(np.float64)
    _, g_want = ogrpo.grpo_loss(lp.cpu().numpy().astype(np.float64), lp_old.cpu().numpy().astype(np.float64),
                                adv.cpu().numpy())
    np.testing.assert_allclose(g, g_want[:, 0], rtol=1e-5)
    dv_o = sde.sde_logprob_grad_v(run.x, v_o, x_next, t, tn, sig) * g[:, None, None]
    assert rms_rel(dv.cpu().numpy(), dv_o) <= V_TOL
    _, G, dx_ref = run.oracle(dv_o)
    _compare(run, grad, dx, G, dx_ref)


def test_flux_block_training_pass_properties(cuda):
    """Flux-shaped double-stream block (H 3072, 24 x 128 heads, MLP 12288,
    512 text + 4096 image tokens, batch 4) at full size: the training
    forward equals the velocity call bit for bit; the backward is
    deterministic, finite, linear in dv, and its final-bias gradient is the
    token sum of dv."""
    import torch
    cfg = synth.config("flux_double_block")
    run = Run(cfg, cuda, std=0.02)
    ws = torch.empty(run.model.workspace_size(run.B), dtype=torch.uint8, device=cuda)
    v = torch.empty_like(run.xg)
    run.model.ff_dit_velocity(run.xg, run.tg, run.tt, v, ws)
    torch.cuda.synchronize()
    assert torch.equal(v, run.v)
    del ws
    rng = np.random.default_rng(7)
    d1 = torch.from_numpy(rng.standard_normal(tuple(v.shape)).astype(np.float32)).to(cuda)
    d2 = torch.from_numpy(rng.standard_normal(tuple(v.shape)).astype(np.float32)).to(cuda)
    g1, x1 = run.backward(d1)
    g1b, _ = run.backward(d1)
    assert np.array_equal(g1, g1b)
    assert np.all(np.isfinite(g1)) and np.all(np.isfinite(x1))
    g2, x2 = run.backward(d2)
    g12, x12 = run.backward(d1 + d2)
    got = run.tensors(g12)
    s1, s2 = run.tensors(g1), run.tensors(g2)
    for name in got:
        assert rms_rel(got[name], s1[name] + s2[name]) <= G_TOL, name
    fb = run.tensors(g1)["final.b"]
    np.testing.assert_allclose(fb, d1.double().sum(dim=(0, 1)).cpu().numpy(), rtol=1e-4, atol=1e-3)


def test_wan_full_width_training_pass_properties(cuda):
    """Two WAN-style blocks at full width (H 5120, 40 x 128 heads, MLP 13824,
    32760 latent + 512 text tokens, batch 1): the training forward equals the
    velocity call bit for bit; the backward is deterministic and finite, its
    final-bias gradient is the token sum of dv, and recompute mode gives the
    same gradient bit for bit."""
    import torch
    cfg = synth.config("wan_40", n_double=2, batch=1)
    run = Run(cfg, cuda, std=0.02)
    ws = torch.empty(run.model.workspace_size(run.B), dtype=torch.uint8, device=cuda)
    v = torch.empty_like(run.xg)
    run.model.ff_dit_velocity(run.xg, run.tg, run.tt, v, ws)
    torch.cuda.synchronize()
    assert torch.equal(v, run.v)
    del ws
    d1 = torch.from_numpy(np.random.default_rng(8).standard_normal(tuple(v.shape)).astype(np.float32)).to(cuda)
    g1, x1 = run.backward(d1)
    g1b, x1b = run.backward(d1)
    assert np.array_equal(g1, g1b) and np.array_equal(x1, x1b)
    assert np.all(np.isfinite(g1)) and np.all(np.isfinite(x1))
    fb = run.tensors(g1)["final.b"]
    np.testing.assert_allclose(fb, d1.double().sum(dim=(0, 1)).cpu().numpy(), rtol=1e-4, atol=1e-3)
    # every tensor receives a gradient
    assert all(float(np.abs(a).max()) > 0 for a in run.tensors(g1).values())
    del run.ws
    torch.cuda.empty_cache()
    run.model.set_train_recompute(True)
    ws = torch.empty(run.model.train_workspace_size(run.B), dtype=torch.uint8, device=cuda)
    v2 = torch.empty_like(run.xg)
    run.model.ff_dit_forward_train(run.xg, run.tg, run.tt, v2, ws)
    grad = torch.zeros(run.total, dtype=torch.float32, device=cuda)
    dx = torch.empty_like(run.xg)
    run.model.ff_dit_backward(run.tg, d1, grad, ws, dx_t=dx)
    torch.cuda.synchronize()
    assert torch.equal(v2, run.v)
    assert np.array_equal(grad.cpu().numpy(), g1) and np.array_equal(dx.cpu().numpy(), x1)
    run.model.set_train_recompute(False)


def test_nft_training_step_chain(cuda):
    """A DiffusionNFT step (Eq. 2): the trained velocity from the training
    forward, the frozen old policy's velocity from a second model, the loss
    with dL/dv, then the DiT backward; against the oracle chain."""
    import torch
    from oracle import awm as oawm
    from oracle import nft as onft
    from paper_2602_12529_gb300 import ffi
    cfg = _cfg(batch=4, n_txt=8)
    run = Run(cfg, cuda, seed=3)
    old = Run(cfg, cuda, seed=4)
    B, Ni, Pd = run.B, synth.n_img(cfg), cfg["patch_dim"]
    eps, x0 = synth.gaussian((B, Ni, Pd), 60, "eps"), synth.gaussian((B, Ni, Pd), 61, "x0")
    r = synth.uniform((B,), 62, "r")
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(cuda)
    loss = torch.empty(1, dtype=torch.float32, device=cuda)
    dv = torch.empty_like(run.xg)
    beta = 0.5
    ffi.ff_nft_loss(run.v, old.v, T(eps), T(x0), T(r), beta, ffi.FF_AWM_MEAN, loss, dv)
    grad, dx = run.backward(dv)
    P = odit.widen_params(run.W)
    t = run.t.astype(np.float64)
    v_o = odit.velocity(P, cfg, run.x, odit.widen(run.txt), t)
    vold_o = odit.velocity(odit.widen_params(old.W), cfg, old.x, odit.widen(old.txt), t)
    L_o, dv_o, _ = onft.nft_loss(v_o, vold_o, eps, x0, r, beta, "mean")
    assert abs(float(loss.item()) - L_o) <= V_TOL * abs(L_o)
    assert rms_rel(dv.cpu().numpy(), dv_o) <= V_TOL
    _, G, dx_ref = run.oracle(dv_o)
    _compare(run, grad, dx, G, dx_ref)
