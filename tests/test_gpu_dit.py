"""GPU parity of the whole velocity call v_theta(x_t, t) (ff_dit_velocity)
against the fp64 oracle: full output on small MMDiTs, sampled rows on the
Flux-shaped double-stream block."""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import dit as odit

pytestmark = pytest.mark.gpu

V_TOL = 2e-2   # RMS-relative error bound for the bf16 velocity


def _setup(cfg, dev, seed=0, bias_std=0.02, scale_std=0.1, batch=None):
    import torch
    from paper_2602_12529_gb300 import ffi, weights
    cache = {}

    def get(name, shape):
        a = synth.weight(name, shape, synth.weight_kind(name), seed, 0.02, bias_std, scale_std)
        cache[name] = a
        return a

    blob = weights.pack(cfg, get, dev)
    model = ffi.Dit(cfg, blob)
    B = cfg["batch"] if batch is None else batch
    x = synth.initial_latent(cfg, batch=B)
    txt = synth.text_embeds(cfg, batch=B)
    t = np.linspace(1.0, 0.3, B).astype(np.float32)
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=dev)
    xg = torch.from_numpy(x).to(dev)
    tg = torch.from_numpy(txt.view(np.int16)).to(dev).view(torch.bfloat16)
    tt = torch.from_numpy(t).to(dev)
    v = torch.empty_like(xg)
    model.ff_dit_velocity(xg, tg, tt, v, ws)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    return model, cache, x, txt, t, v.cpu().numpy()


@pytest.mark.parametrize("over", [{}, {"n_double": 1, "n_single": 1}, {"n_double": 0, "n_single": 2, "n_txt": 20}])
def test_velocity_small_mmdit_full_parity(cuda, over):
    cfg = synth.config("tiny_mmdit", **over)
    model, W, x, txt, t, v = _setup(cfg, cuda)
    P = odit.widen_params(W)
    want = odit.velocity(P, cfg, x, odit.widen(txt), t.astype(np.float64))
    err = rms_rel(v, want)
    assert err <= V_TOL, err
    for b in range(x.shape[0]):
        assert rms_rel(v[b], want[b]) <= V_TOL


def test_velocity_ragged_grid(cuda):
    # token counts that are not multiples of any tile size
    cfg = synth.config("tiny_mmdit", grid=(1, 7, 9), n_txt=13, batch=3, n_double=1, n_single=1)
    model, W, x, txt, t, v = _setup(cfg, cuda)
    want = odit.velocity(odit.widen_params(W), cfg, x, odit.widen(txt), t.astype(np.float64))
    assert rms_rel(v, want) <= V_TOL


def test_velocity_is_deterministic(cuda):
    import torch
    cfg = synth.config("tiny_mmdit")
    model, W, x, txt, t, v = _setup(cfg, cuda)
    dev = cuda
    ws = torch.empty(model.workspace_size(4), dtype=torch.uint8, device=dev)
    xg = torch.from_numpy(x).to(dev)
    tg = torch.from_numpy(txt.view(np.int16)).to(dev).view(torch.bfloat16)
    v2 = torch.empty_like(xg)
    model.ff_dit_velocity(xg, tg, torch.from_numpy(t).to(dev), v2, ws)
    torch.cuda.synchronize()
    assert np.array_equal(v2.cpu().numpy(), v)


def test_velocity_flux_block_sampled_rows(cuda):
    """Flux-shaped double-stream block (H 3072, 24 x 128 heads, MLP 12288,
    512 text + 4096 image tokens, batch 4): every sample, 48 sampled rows."""
    cfg = synth.config("flux_double_block")
    model, W, x, txt, t, v = _setup(cfg, cuda)
    P = odit.widen_params(W)
    rng = np.random.default_rng(0)
    rows = np.sort(rng.choice(synth.n_img(cfg), 48, replace=False))
    rows[0], rows[-1] = 0, synth.n_img(cfg) - 1
    for b in range(cfg["batch"]):
        want = odit.velocity(P, cfg, x[b:b + 1], odit.widen(txt[b:b + 1]), t[b:b + 1].astype(np.float64),
                             img_rows=rows)[0]
        err = rms_rel(v[b, rows], want)
        assert err <= V_TOL, (b, err)


WAN_SMALL = dict(name="wan_small", arch="wan", hidden=256, heads=4, head_dim=64, mlp=512, n_double=2, n_single=0,
                 patch_dim=64, txt_dim=256, n_txt=20, grid=(3, 4, 6), rope_axes=(24, 20, 20), rope_theta=10000.0,
                 time_freq_dim=256, batch=2)


@pytest.mark.parametrize("over", [{}, {"grid": (2, 5, 7), "n_txt": 13, "batch": 3, "n_double": 1}])
def test_wan_velocity_small_full_parity(cuda, over):
    cfg = dict(WAN_SMALL, **over)
    model, W, x, txt, t, v = _setup(cfg, cuda)
    want = odit.wan_velocity(odit.widen_params(W), cfg, x, odit.widen(txt), t.astype(np.float64))
    err = rms_rel(v, want)
    assert err <= V_TOL, err


def test_wan_block_full_width_sampled_rows(cuda):
    """One WAN block at full width (H 5120, 40 x 128 heads, MLP 13824) over
    the full 21 x 30 x 52 = 32760-token video latent plus 512 text tokens."""
    cfg = synth.config("wan_40", n_double=1)
    model, W, x, txt, t, v = _setup(cfg, cuda)
    P = odit.widen_params(W)
    rng = np.random.default_rng(5)
    rows = np.sort(rng.choice(synth.n_img(cfg), 24, replace=False))
    rows[-1] = synth.n_img(cfg) - 1
    want = odit.wan_velocity(P, cfg, x[:1], odit.widen(txt[:1]), t[:1].astype(np.float64), img_rows=rows)[0]
    err = rms_rel(v[0, rows], want)
    assert err <= V_TOL, err
