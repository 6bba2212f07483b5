"""GPU checks of ff_rollout (trajectory sampling) on the tiny MMDiT with 4
SDE steps: identical to the same steps issued one call at a time, and
stage-wise parity with the fp64 oracle along the GPU's own trajectory."""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import dit as odit
from oracle import sde as osde

pytestmark = pytest.mark.gpu


def _t(a, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a)).to(dev)


def _setup(cuda, window=None):
    import torch
    from paper_2602_12529_gb300 import ffi, weights
    cfg = synth.config("tiny_mmdit")
    W = {}

    def get(name, shape):
        a = synth.weight(name, shape, synth.weight_kind(name), 0, 0.02, 0.02, 0.1)
        W[name] = a
        return a

    model = ffi.Dit(cfg, weights.pack(cfg, get, cuda))
    S, B = cfg["sde_steps"], cfg["batch"]
    if window is None:
        tg, sg = ffi.ff_sde_schedule(ffi.FF_SCHED_FLOW_SDE, S, cfg["shift"], cfg["eta"], cfg["t_clamp"])
    else:
        tg, sg = ffi.ff_sde_schedule_window(ffi.FF_SCHED_FLOW_SDE, S, cfg["shift"], cfg["eta"], cfg["t_clamp"], *window)
    tg[-1] = 1e-3   # the last step stops just short of t = 0 (the drift's 1/t)
    x0 = synth.initial_latent(cfg)
    eps = np.stack([synth.step_noise(cfg, k) for k in range(S)])
    txt = synth.text_embeds(cfg)
    return ffi, model, W, cfg, S, B, np.float32(tg), np.float32(sg), x0, eps, txt


@pytest.mark.parametrize("window", [None, (1, 2)])
def test_rollout_equals_stepwise_calls(cuda, window):
    import torch
    ffi, model, W, cfg, S, B, tg, sg, x0, eps, txt = _setup(cuda, window)
    txtg = _t(txt.view(np.int16), cuda).view(torch.bfloat16)
    x = _t(x0, cuda)
    traj = torch.empty((S + 1,) + x.shape, dtype=torch.float32, device=cuda)
    lp = torch.empty((B, S), dtype=torch.float32, device=cuda)
    model.ff_rollout(x, txtg, _t(tg, cuda), _t(sg, cuda), _t(eps, cuda), lp, traj=traj)
    # the same steps, one call at a time
    xs = _t(x0, cuda)
    v = torch.empty_like(xs)
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=cuda)
    lps = torch.empty((B, S), dtype=torch.float32, device=cuda)
    for k in range(S):
        tk = torch.full((B,), float(tg[k]), device=cuda)
        tn = torch.full((B,), float(tg[k + 1]), device=cuda)
        sk = torch.full((B,), float(sg[k]), device=cuda)
        model.ff_dit_velocity(xs, txtg, tk, v, ws)
        out = torch.empty_like(xs)
        lk = torch.empty(B, dtype=torch.float32, device=cuda)
        ffi.ff_sde_step_logprob(xs, v, _t(eps[k], cuda), out, tk, tn, sk, lk)
        lps[:, k] = lk
        assert torch.equal(traj[k + 1], out), k
        xs = out
    torch.cuda.synchronize()
    assert torch.equal(x, xs) and torch.equal(traj[0], _t(x0, cuda))
    assert torch.equal(lp, lps)
    if window is not None:
        lpc = lp.cpu().numpy()
        assert np.all(lpc[:, 0] == 0.0) and np.all(lpc[:, 3] == 0.0) and np.all(lpc[:, 1:3] != 0.0)
    # without a trajectory buffer, in place on x
    x2 = _t(x0, cuda)
    lp2 = torch.empty_like(lp)
    model.ff_rollout(x2, txtg, _t(tg, cuda), _t(sg, cuda), _t(eps, cuda), lp2)
    torch.cuda.synchronize()
    assert torch.equal(x2, x) and torch.equal(lp2, lp)
    assert ffi.ff_check_device_status() == 0


def test_rollout_stagewise_oracle_parity(cuda):
    import torch
    ffi, model, W, cfg, S, B, tg, sg, x0, eps, txt = _setup(cuda)
    txtg = _t(txt.view(np.int16), cuda).view(torch.bfloat16)
    x = _t(x0, cuda)
    traj = torch.empty((S + 1,) + x.shape, dtype=torch.float32, device=cuda)
    lp = torch.empty((B, S), dtype=torch.float32, device=cuda)
    model.ff_rollout(x, txtg, _t(tg, cuda), _t(sg, cuda), _t(eps, cuda), lp, traj=traj)
    torch.cuda.synchronize()
    P = odit.widen_params(W)
    trc, lpc = traj.cpu().numpy(), lp.cpu().numpy()
    v = torch.empty_like(x)
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=cuda)
    for k in range(S):
        tk = np.full(B, tg[k])
        # the velocity the rollout used at its own state x_k, against the oracle's
        model.ff_dit_velocity(traj[k], txtg, _t(np.float32(tk), cuda), v, ws)
        torch.cuda.synchronize()
        vk = v.cpu().numpy()
        want_v = odit.velocity(P, cfg, trc[k].astype(np.float64), odit.widen(txt), tk.astype(np.float64))
        assert rms_rel(vk, want_v) <= 2e-2, k
        # the SDE step from (x_k, v_k, eps_k), against the oracle's
        want_x, want_lp = osde.sde_step_logprob(trc[k], vk, tk, np.full(B, tg[k + 1]), np.full(B, sg[k]), eps=eps[k])
        assert np.max(np.abs(trc[k + 1] - want_x)) <= 1e-5 * np.max(np.abs(want_x)), k
        np.testing.assert_allclose(lpc[:, k], want_lp, rtol=1e-3)
