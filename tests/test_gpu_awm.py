"""GPU parity of the widened rows through the C ABI: AWM (training-time
samplers, forward process, Eq. 3 loss and gradient, and a whole AWM step
with the velocity), multi-reward advantage aggregation, GRPO-Guard step
weights and the MixGRPO SDE window."""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import awm as oawm
from oracle import dit as odit
from oracle import grpo as ogrpo
from oracle import sde as osde

pytestmark = pytest.mark.gpu


def _t(a, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def test_timestep_samplers_parity(cuda):
    import torch
    from paper_2602_12529_gb300 import ffi
    B = 1000
    u = synth.uniform((B,), 21, "t_u")
    u[:4] = [0.0, 0.25, 0.5, 0.9999999]
    z = synth.gaussian((B,), 22, "t_z")
    out = torch.empty(B, dtype=torch.float32, device=cuda)
    ffi.ff_sample_timesteps(ffi.FF_TSAMPLE_UNIFORM, _t(u, cuda), 0.05, 0.95, out)
    torch.cuda.synchronize()
    np.testing.assert_allclose(out.cpu().numpy(), oawm.sample_timesteps("uniform", u, 0.05, 0.95), rtol=2e-7, atol=1e-7)
    ffi.ff_sample_timesteps(ffi.FF_TSAMPLE_LOGIT_NORMAL, _t(z, cuda), 0.3, 1.1, out)
    torch.cuda.synchronize()
    np.testing.assert_allclose(out.cpu().numpy(), oawm.sample_timesteps("logit_normal", z, 0.3, 1.1), rtol=2e-6, atol=1e-7)
    t_grid, _ = ffi.ff_sde_schedule(ffi.FF_SCHED_FLOW_SDE, 10, 3.0, 0.7, 0.96)
    grid = np.asarray(t_grid[:10], np.float32)
    ffi.ff_sample_timesteps(ffi.FF_TSAMPLE_DISCRETE, _t(u, cuda), 0.0, 0.0, out, grid=_t(grid, cuda))
    torch.cuda.synchronize()
    # the index is an integer decision: bit-exact against the oracle's fp32 index
    np.testing.assert_array_equal(out.cpu().numpy(), oawm.sample_timesteps("discrete", u, grid=grid).astype(np.float32))


@pytest.mark.parametrize("B,D", [(4, 262144), (3, 12340), (1, 4)])
def test_forward_process_parity(cuda, B, D):
    import torch
    from paper_2602_12529_gb300 import ffi
    x0, eps = synth.gaussian((B, D), 30, "x0"), synth.gaussian((B, D), 31, "eps")
    t = np.linspace(0.0, 1.0, B).astype(np.float32)
    xt = torch.empty((B, D), dtype=torch.float32, device=cuda)
    ffi.ff_forward_process(_t(x0, cuda), _t(eps, cuda), _t(t, cuda), xt)
    torch.cuda.synchronize()
    want = oawm.forward_process(x0, eps, t)
    got = xt.cpu().numpy()
    assert np.max(np.abs(got - want)) <= 2e-7 * max(1.0, np.max(np.abs(want)))
    # t = 0 and t = 1 reproduce x0 and eps exactly
    np.testing.assert_array_equal(got[0], x0[0])
    if B > 1:
        np.testing.assert_array_equal(got[-1], eps[-1])
    # in place over x0
    x0g = _t(x0, cuda)
    ffi.ff_forward_process(x0g, _t(eps, cuda), _t(t, cuda), x0g)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(x0g.cpu().numpy(), got)


@pytest.mark.parametrize("B,D,reduce", [(4, 262144, 0), (4, 262144, 1), (5, 12340, 0), (2, 4, 1), (64, 4096, 0)])
def test_awm_loss_parity(cuda, B, D, reduce):
    import torch
    from paper_2602_12529_gb300 import ffi
    v = synth.gaussian((B, D), 40, "v")
    eps, x0 = synth.gaussian((B, D), 41, "eps"), synth.gaussian((B, D), 42, "x0")
    adv = synth.gaussian((B,), 43, "adv")
    loss = torch.zeros(1, dtype=torch.float32, device=cuda)
    grad = torch.empty((B, D), dtype=torch.float32, device=cuda)
    err = torch.empty(B, dtype=torch.float32, device=cuda)
    ffi.ff_awm_loss(_t(v, cuda), _t(eps, cuda), _t(x0, cuda), _t(adv, cuda), reduce, loss, grad, err)
    torch.cuda.synchronize()
    want, want_g, want_e = oawm.awm_loss(v, eps, x0, adv, "mean" if reduce else "sum")
    np.testing.assert_allclose(err.cpu().numpy(), want_e, rtol=2e-5)
    assert abs(float(loss.item()) - want) <= 2e-5 * float(np.mean(np.abs(adv) * want_e))
    g = grad.cpu().numpy()
    assert np.max(np.abs(g - want_g)) <= 1e-6 * np.max(np.abs(want_g))
    # the gradient output is optional and leaves the loss unchanged
    first = float(loss.item())
    ffi.ff_awm_loss(_t(v, cuda), _t(eps, cuda), _t(x0, cuda), _t(adv, cuda), reduce, loss)
    torch.cuda.synchronize()
    assert float(loss.item()) == first


def test_awm_loss_is_zero_at_the_flow_target(cuda):
    import torch
    from paper_2602_12529_gb300 import ffi
    B, D = 3, 8192
    eps, x0 = synth.gaussian((B, D), 44, "eps"), synth.gaussian((B, D), 45, "x0")
    v = (eps - x0).astype(np.float32)
    loss = torch.full((1,), 7.0, dtype=torch.float32, device=cuda)
    err = torch.full((B,), 7.0, dtype=torch.float32, device=cuda)
    ffi.ff_awm_loss(_t(v, cuda), _t(eps, cuda), _t(x0, cuda), _t(np.ones(B, np.float32), cuda), 0, loss, None, err)
    torch.cuda.synchronize()
    # fp32 eps - x0 computed the same way on both sides: exactly zero
    assert float(loss.item()) == 0.0 and np.all(err.cpu().numpy() == 0.0)


def test_awm_step_end_to_end_small_model(cuda):
    """One AWM training step on a small MMDiT: t from the logit-normal
    sampler, x_t by the forward process, v = v_theta(x_t, t), Eq. 3 loss;
    every stage against the oracle's composition on the same inputs."""
    import torch
    from paper_2602_12529_gb300 import ffi, weights
    cfg = synth.config("tiny_mmdit")
    B = cfg["batch"]
    W = {}

    def get(name, shape):
        a = synth.weight(name, shape, synth.weight_kind(name), 0, 0.02, 0.02, 0.1)
        W[name] = a
        return a

    model = ffi.Dit(cfg, weights.pack(cfg, get, cuda))
    x0 = synth.initial_latent(cfg, seed=50)
    eps = synth.initial_latent(cfg, seed=51)
    z = synth.gaussian((B,), 52, "awm_z")
    txt = synth.text_embeds(cfg, seed=53)
    adv = ogrpo.group_advantage(synth.rewards(B, seed=54), B).astype(np.float32)
    tg = torch.empty(B, dtype=torch.float32, device=cuda)
    ffi.ff_sample_timesteps(ffi.FF_TSAMPLE_LOGIT_NORMAL, _t(z, cuda), 0.0, 1.0, tg)
    xt = torch.empty_like(_t(x0, cuda))
    ffi.ff_forward_process(_t(x0, cuda), _t(eps, cuda), tg, xt)
    v = torch.empty_like(xt)
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=cuda)
    model.ff_dit_velocity(xt, _t(txt.view(np.int16), cuda).view(torch.bfloat16), tg, v, ws)
    loss = torch.zeros(1, dtype=torch.float32, device=cuda)
    ffi.ff_awm_loss(v, _t(eps, cuda), _t(x0, cuda), _t(adv, cuda), ffi.FF_AWM_MEAN, loss)
    torch.cuda.synchronize()
    t_want = oawm.sample_timesteps("logit_normal", z, 0.0, 1.0)
    np.testing.assert_allclose(tg.cpu().numpy(), t_want, rtol=2e-6)
    xt_want = oawm.forward_process(x0, eps, tg.cpu().numpy())
    assert np.max(np.abs(xt.cpu().numpy() - xt_want)) <= 1e-6 * np.max(np.abs(xt_want))
    v_want = odit.velocity(odit.widen_params(W), cfg, xt.cpu().numpy().astype(np.float64), odit.widen(txt),
                           tg.cpu().numpy().astype(np.float64))
    assert rms_rel(v.cpu().numpy(), v_want) <= 2e-2
    # the loss from the GPU's own velocity matches the oracle's loss formula on it
    want, _, _ = oawm.awm_loss(v.cpu().numpy(), eps, x0, adv, "mean")
    assert abs(float(loss.item()) - want) <= 1e-5 * abs(want) + 1e-7


@pytest.mark.parametrize("ng,G,K", [(3, 16, 3), (2, 5, 2), (4, 100, 1), (1, 4096, 4)])
@pytest.mark.parametrize("mode", [0, 1])
def test_group_advantage_multi_parity(cuda, ng, G, K, mode):
    import torch
    from paper_2602_12529_gb300 import ffi
    R = synth.uniform((ng * G, K), 60 + G, "rk") * np.float32(1.0) + np.arange(K, dtype=np.float32) * np.float32(10.0)
    if ng > 1:
        R[:G] = R[0]   # a constant group
    w = (synth.uniform((K,), 61, "wk") + np.float32(0.1)).astype(np.float32)
    adv = torch.empty(ng * G, dtype=torch.float32, device=cuda)
    ffi.ff_group_advantage_multi(_t(R, cuda), G, _t(w, cuda), mode, 1e-4, adv)
    torch.cuda.synchronize()
    want = ogrpo.group_advantage_multi(R, G, w, "per_reward" if mode else "weighted_sum", 1e-4)
    got = adv.cpu().numpy()
    np.testing.assert_allclose(got, want, rtol=2e-4, atol=2e-5)
    if ng > 1:
        assert np.all(got[:G] == 0.0)


@pytest.mark.parametrize("B,T", [(32, 10), (4096, 16)])
def test_grpo_loss_step_weights_parity(cuda, B, T):
    import torch
    from paper_2602_12529_gb300 import ffi
    lp_new = synth.gaussian((B, T), 70, "lpn") * np.float32(50.0) - np.float32(1e3)
    lp_old = lp_new + synth.gaussian((B, T), 71, "lp_jitter") * np.float32(0.3)
    adv = synth.gaussian((B,), 72, "adv")
    w = synth.uniform((T,), 73, "step_w") * np.float32(2.0)
    loss = torch.zeros(1, dtype=torch.float32, device=cuda)
    grad = torch.zeros((B, T), dtype=torch.float32, device=cuda)
    ffi.ff_grpo_loss_weighted(_t(lp_new, cuda), _t(lp_old, cuda), _t(adv, cuda), _t(w, cuda), 0.2, 0.2, loss, grad)
    torch.cuda.synchronize()
    want, want_g = ogrpo.grpo_loss(lp_new, lp_old, adv, 0.2, 0.2, step_w=w)
    assert abs(float(loss.item()) - want) <= 1e-3 * max(abs(want), np.abs(adv).mean())
    rho = np.exp(lp_new.astype(np.float64) - lp_old.astype(np.float64))
    away = np.minimum(np.abs(rho - 0.8), np.abs(rho - 1.2)) > 1e-4
    np.testing.assert_allclose(grad.cpu().numpy()[away], want_g[away], rtol=1e-4, atol=1e-12)
    # all-ones weights reproduce the unweighted loss exactly
    l1 = torch.zeros(1, dtype=torch.float32, device=cuda)
    ffi.ff_grpo_loss_weighted(_t(lp_new, cuda), _t(lp_old, cuda), _t(adv, cuda), _t(np.ones(T, np.float32), cuda),
                              0.2, 0.2, l1)
    l0 = torch.zeros(1, dtype=torch.float32, device=cuda)
    ffi.ff_grpo_loss(_t(lp_new, cuda), _t(lp_old, cuda), _t(adv, cuda), 0.2, 0.2, l0)
    torch.cuda.synchronize()
    assert float(l1.item()) == float(l0.item())


def test_mixgrpo_window_steps(cuda):
    """Steps outside the SDE window are ODE steps: x_next is the drift update
    and the log-prob is 0; steps inside match the stochastic oracle."""
    import torch
    from paper_2602_12529_gb300 import ffi
    S, B, D = 6, 2, 4096
    t_grid, sig = ffi.ff_sde_schedule_window(ffi.FF_SCHED_FLOW_SDE, S, 3.0, 0.7, 0.96, 2, 2)
    x = synth.gaussian((B, D), 80, "x")
    for k in range(S):
        v = synth.gaussian((B, D), 81 + k, "v")
        e = synth.gaussian((B, D), 90 + k, "e")
        t = np.full(B, t_grid[k], np.float32)
        tn = np.full(B, t_grid[k + 1], np.float32)
        sg = np.full(B, sig[k], np.float32)
        out = torch.empty((B, D), dtype=torch.float32, device=cuda)
        lp = torch.zeros(B, dtype=torch.float32, device=cuda)
        ffi.ff_sde_step_logprob(_t(x, cuda), _t(v, cuda), _t(e, cuda), out, _t(t, cuda), _t(tn, cuda), _t(sg, cuda),
                                lp, mode=ffi.FF_SDE_SAMPLE)
        torch.cuda.synchronize()
        want_x, want_lp = osde.sde_step_logprob(x, v, t, tn, sg, eps=e)
        got_lp = lp.cpu().numpy()
        if 2 <= k < 4:
            assert sig[k] > 0 and np.all(got_lp != 0.0)
            np.testing.assert_allclose(got_lp, want_lp, rtol=1e-3)
        else:
            assert sig[k] == 0.0 and np.all(got_lp == 0.0)
        assert np.max(np.abs(out.cpu().numpy() - want_x)) <= 1e-5 * np.max(np.abs(want_x))
        x = out.cpu().numpy()
