"""GPU parity of the SDE step + log-prob, the group advantage and the GRPO
loss against the fp64 oracle, through the C ABI."""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import grpo as ogrpo
from oracle import sde as osde

pytestmark = pytest.mark.gpu


def _t(a, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def _sde_case(B, D, seed, t, tn, sigma):
    x = synth.gaussian((B, D), seed, "x")
    v = synth.gaussian((B, D), seed + 1, "v")
    e = synth.gaussian((B, D), seed + 2, "e")
    f32 = lambda a: np.asarray(a, np.float32)
    return x, v, e, f32(t), f32(tn), f32(sigma)


def _check_sample(ffi, dev, x, v, e, t, tn, sg, reduce=0, inplace=False, ld=1):
    import torch
    B, D = x.shape
    xg, vg, eg = _t(x, dev), _t(v, dev), _t(e, dev)
    out = xg if inplace else torch.empty_like(xg)
    lp = torch.zeros(B * ld, dtype=torch.float32, device=dev)
    ffi.ff_sde_step_logprob(xg, vg, eg, out, _t(t, dev), _t(tn, dev), _t(sg, dev), lp,
                            mode=ffi.FF_SDE_SAMPLE, reduce=reduce, ld=ld)
    torch.cuda.synchronize()
    want_x, want_lp = osde.sde_step_logprob(x, v, t, tn, sg, eps=e, reduce="mean" if reduce else "sum")
    got_x = out.cpu().numpy()
    got_lp = lp.cpu().numpy()[::ld]
    assert rms_rel(got_x, want_x) <= 1e-5
    assert np.max(np.abs(got_x - want_x)) <= 1e-5 * np.max(np.abs(want_x))
    for b in range(B):
        if want_lp[b] == 0.0:
            assert got_lp[b] == 0.0
        else:
            assert abs(got_lp[b] - want_lp[b]) <= 1e-3 * abs(want_lp[b]), (b, got_lp[b], want_lp[b])
    return got_x, got_lp


@pytest.mark.parametrize("B,D", [(4, 4096), (3, 12340), (1, 4), (4, 262144), (32, 65536), (1, 2096640)])
def test_sde_sample_parity(cuda, B, D):
    from paper_2602_12529_gb300 import ffi
    grid = osde.time_grid(10, 3.0)
    t = np.array([grid[k % 10] for k in range(B)])
    tn = np.array([grid[k % 10 + 1] for k in range(B)])
    sg = osde.sigma_flow_sde(t, 0.7, 0.96)
    x, v, e, t, tn, sg = _sde_case(B, D, 11, t, tn, sg)
    _, lp = _check_sample(ffi, cuda, x, v, e, t, tn, sg)
    # quadratic part alone, the sampled residual is std * eps
    sd = sg.astype(np.float64) * np.sqrt(t.astype(np.float64) - tn.astype(np.float64))
    quad = lp + D * np.log(sd) + 0.5 * D * np.log(2 * np.pi)
    np.testing.assert_allclose(quad, -0.5 * (e.astype(np.float64) ** 2).sum(1), rtol=1e-3)


def test_sde_mean_reduce_strided_inplace_and_ode(cuda):
    from paper_2602_12529_gb300 import ffi
    B, D = 4, 8192
    t = np.array([0.75, 0.5, 0.9, 0.3])
    tn = np.array([0.5, 0.25, 0.8, 0.1])
    sg = np.array([0.7, 0.0, 1.1, 0.4])   # sample 1 is an ODE step
    x, v, e, t, tn, sg = _sde_case(B, D, 21, t, tn, sg)
    _check_sample(ffi, cuda, x, v, e, t, tn, sg, reduce=ffi.FF_LP_MEAN, inplace=True, ld=3)


def test_sde_eval_mode(cuda):
    import torch
    from paper_2602_12529_gb300 import ffi
    B, D = 2, 65536
    t, tn = np.array([0.9643, 0.5]), np.array([0.9, 0.4])
    sg = osde.sigma_flow_sde(t, 0.7, 0.96)
    x, v, e, t, tn, sg = _sde_case(B, D, 31, t, tn, sg)
    # score a given x_next (here: another draw, so the quadratic term is large)
    xn = synth.gaussian((B, D), 99, "xn")
    lp = torch.zeros(B, dtype=torch.float32, device=cuda)
    xng = _t(xn, cuda)
    ffi.ff_sde_step_logprob(_t(x, cuda), _t(v, cuda), None, xng, _t(t, cuda), _t(tn, cuda), _t(sg, cuda), lp,
                            mode=ffi.FF_SDE_EVAL)
    torch.cuda.synchronize()
    _, want = osde.sde_step_logprob(x, v, t, tn, sg, x_next=xn)
    np.testing.assert_allclose(lp.cpu().numpy(), want, rtol=1e-3)
    assert np.array_equal(xng.cpu().numpy(), xn)   # eval mode does not write x_next


@pytest.mark.parametrize("ng,G", [(2, 16), (1, 4), (5, 1), (3, 4096), (10000, 8), (7, 33)])
def test_group_advantage_parity(cuda, ng, G):
    import torch
    from paper_2602_12529_gb300 import ffi
    r = synth.rewards(ng * G, seed=7 + G)
    if ng > 1:
        r[:G] = 0.25   # a constant group
    if ng > 2:
        r[G:2 * G] = 0.3   # one whose fp32 sum is inexact
    rg = _t(r, cuda)
    adv = torch.empty_like(rg)
    ffi.ff_group_advantage(rg, G, 1e-4, adv)
    ffi.ff_group_advantage(rg, G, 1e-4, rg)   # in place
    torch.cuda.synchronize()
    want = ogrpo.group_advantage(r, G, 1e-4)
    np.testing.assert_allclose(adv.cpu().numpy(), want, rtol=1e-5, atol=1e-6)
    np.testing.assert_array_equal(rg.cpu().numpy(), adv.cpu().numpy())
    if ng > 1:
        assert np.all(adv.cpu().numpy()[:G] == 0.0)
    if ng > 2:
        assert np.all(adv.cpu().numpy()[G:2 * G] == 0.0)


@pytest.mark.parametrize("B,T,noise,adv_mean", [(32, 10, 0.01, 0.0), (8, 3, 0.5, 0.0), (4, 1, 0.3, 0.0),
                                                  (4096, 256, 0.4, 0.0), (1000, 10, 0.3, 0.7),
                                                  (333, 7, 0.05, -1.5)])
def test_grpo_loss_parity(cuda, B, T, noise, adv_mean):
    import torch
    from paper_2602_12529_gb300 import ffi
    lp_new = synth.gaussian((B, T), 5, "lpn") * np.float32(50.0) - np.float32(1e3)
    lp_old = lp_new + synth.gaussian((B, T), 9, "lp_jitter") * np.float32(noise)
    adv = synth.gaussian((B,), 6, "adv") + np.float32(adv_mean)
    loss = torch.zeros(1, dtype=torch.float32, device=cuda)
    grad = torch.zeros((B, T), dtype=torch.float32, device=cuda)
    ws = torch.zeros(ffi.ff_grpo_loss_workspace_size(B, T), dtype=torch.uint8, device=cuda)
    ffi.ff_grpo_loss(_t(lp_new, cuda), _t(lp_old, cuda), _t(adv, cuda), 0.2, 0.2, loss, grad, ws=ws)
    torch.cuda.synchronize()
    want, want_g = ogrpo.grpo_loss(lp_new, lp_old, adv, 0.2, 0.2)
    got = float(loss.item())
    # relative bound on the loss itself (every case here has |loss| >= 0.05)
    assert abs(want) >= 0.05
    assert abs(got - want) <= 1e-3 * abs(want), (got, want)
    # the single launch leaves its ticket at zero: a second call on the same
    # workspace gives the identical loss
    ffi.ff_grpo_loss(_t(lp_new, cuda), _t(lp_old, cuda), _t(adv, cuda), 0.2, 0.2, loss, grad, ws=ws)
    torch.cuda.synchronize()
    assert float(loss.item()) == got
    assert int(ws[:4].view(torch.int32).item()) == 0
    # gradients: identical branch decisions away from the clip kinks
    rho = np.exp(lp_new.astype(np.float64) - lp_old.astype(np.float64))
    away = np.minimum(np.abs(rho - 0.8), np.abs(rho - 1.2)) > 1e-4
    np.testing.assert_allclose(grad.cpu().numpy()[away], want_g[away], rtol=1e-4, atol=1e-12)
    # without the optional gradient output
    ffi.ff_grpo_loss(_t(lp_new, cuda), _t(lp_old, cuda), _t(adv, cuda), 0.2, 0.2, loss, None)
    torch.cuda.synchronize()
    assert float(loss.item()) == got


def test_loss_ratio_one_is_minus_mean_advantage(cuda):
    import torch
    from paper_2602_12529_gb300 import ffi
    B, T = 16, 10
    lp = synth.gaussian((B, T), 3, "lp")
    adv = synth.gaussian((B,), 4, "a")
    loss = torch.zeros(1, dtype=torch.float32, device=cuda)
    ffi.ff_grpo_loss(_t(lp, cuda), _t(lp, cuda), _t(adv, cuda), 0.2, 0.2, loss)
    torch.cuda.synchronize()
    assert abs(loss.item() + adv.astype(np.float64).mean()) <= 1e-6


@pytest.mark.parametrize("shapes", [[(4, 262144), (1, 2096640), (32, 4096), (4, 262144)]])
def test_sde_single_launch_reuses_its_workspace(cuda, shapes):
    """One workspace, zeroed once, serves calls of different shapes in
    stream order: the last block of each sample hands its ticket back, so
    the ticket words are zero after every call and repeated calls give
    bit-identical log-probs."""
    import torch
    from paper_2602_12529_gb300 import ffi
    size = max(ffi.ff_sde_workspace_size(B, D) for B, D in shapes)
    ws = torch.zeros(size, dtype=torch.uint8, device=cuda)
    grid = osde.time_grid(10, 3.0)
    for i, (B, D) in enumerate(shapes):
        t = np.array([grid[(i + b) % 10] for b in range(B)])
        tn = np.array([grid[(i + b) % 10 + 1] for b in range(B)])
        x, v, e, t, tn, sg = _sde_case(B, D, 40 + i, t, tn, osde.sigma_flow_sde(t, 0.7, 0.96))
        xg, vg, eg, tg, tng, sgg = (_t(a, cuda) for a in (x, v, e, t, tn, sg))
        out = torch.empty_like(xg)
        lps = []
        for _ in range(2):
            lp = torch.full((B,), 7.0, dtype=torch.float32, device=cuda)
            ffi.ff_sde_step_logprob(xg, vg, eg, out, tg, tng, sgg, lp, ws=ws)
            torch.cuda.synchronize()
            lps.append(lp.cpu().numpy())
            assert int(ws[:256 * 1024].view(torch.int32).abs().sum().item()) == 0
        np.testing.assert_array_equal(lps[0], lps[1])
        _, want_lp = osde.sde_step_logprob(x, v, t, tn, sg, eps=e)
        np.testing.assert_allclose(lps[0], want_lp, rtol=1e-3)
