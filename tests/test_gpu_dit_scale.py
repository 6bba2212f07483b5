"""GPU checks of ff_dit_velocity at the larger workload shapes.

* Reduced depth, full width and sequence length: the Flux-shaped rollout
  (8 double + 16 single blocks, batch 32, 512 + 1024 tokens) cut to one block
  of each kind, and the Qwen-Image shape (256 + 4096 tokens, D_txt 3584) cut to
  one double block, compared with the fp64 oracle on sampled rows of sampled
  samples.
* Full depth (24 and 60 MMDiT blocks; 40 WAN blocks over 32760 video tokens
  at batch 2), weights drawn on the device: properties that hold at any size
  -- finite output, identical results on a second call, and every sample's
  velocity bit-identical to the one computed in a smaller batch (samples
  never interact).
"""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import dit as odit

pytestmark = pytest.mark.gpu

V_TOL = 2e-2


def _blob_from_synth(cfg, dev, W):
    from paper_2602_12529_gb300 import weights

    def get(name, shape):
        a = synth.weight(name, shape, synth.weight_kind(name), 0, 0.02, 0.02, 0.1)
        W[name] = a
        return a
    return weights.pack(cfg, get, dev)


def _blob_on_device(cfg, dev, seed=0):
    """N(0, 0.02) matrices, zero biases, unit norm scales, drawn on the GPU."""
    import torch
    from paper_2602_12529_gb300 import ffi
    specs, total = ffi.ff_dit_weight_layout(cfg)
    blob = torch.zeros(total, dtype=torch.bfloat16, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    for name, off, shape in specs:
        n = int(np.prod(shape))
        kind = synth.weight_kind(name)
        if kind == "matrix":
            blob[off:off + n] = (torch.randn(n, generator=g, device=dev) * 0.02).to(torch.bfloat16)
        elif kind == "scale":
            blob[off:off + n] = 1.0
    return blob


def _run(cfg, model, x, txt, t, dev):
    import torch
    B = x.shape[0]
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=dev)
    v = torch.empty_like(x)
    model.ff_dit_velocity(x, txt, t, v, ws)
    torch.cuda.synchronize()
    return v


def _inputs(cfg, dev, B):
    import torch
    x = torch.from_numpy(synth.initial_latent(cfg, batch=B)).to(dev)
    txt = torch.from_numpy(synth.text_embeds(cfg, batch=B).view(np.int16)).to(dev).view(torch.bfloat16)
    t = torch.from_numpy(np.linspace(1.0, 0.1, B).astype(np.float32)).to(dev)
    return x, txt, t


@pytest.mark.parametrize("name,over,samples", [
    ("flux_8d16s", {"n_double": 1, "n_single": 1}, (0, 31)),
    ("qwen_image_60d", {"n_double": 1}, (0, 3)),
])
def test_reduced_depth_sampled_rows(cuda, name, over, samples):
    from paper_2602_12529_gb300 import ffi
    cfg = synth.config(name, **over)
    W = {}
    model = ffi.Dit(cfg, _blob_from_synth(cfg, cuda, W))
    B = cfg["batch"]
    x, txt, t = _inputs(cfg, cuda, B)
    v = _run(cfg, model, x, txt, t, cuda).cpu().numpy()
    P = odit.widen_params(W)
    rng = np.random.default_rng(1)
    rows = np.sort(rng.choice(synth.n_img(cfg), 32, replace=False))
    xs = x.cpu().numpy()
    txs = synth.text_embeds(cfg, batch=B)
    ts = t.cpu().numpy().astype(np.float64)
    for b in samples:
        want = odit.velocity(P, cfg, xs[b:b + 1], odit.widen(txs[b:b + 1]), ts[b:b + 1], img_rows=rows)[0]
        err = rms_rel(v[b, rows], want)
        assert err <= V_TOL, (b, err)


@pytest.mark.parametrize("name,sub,batch", [("flux_8d16s", 3, None), ("qwen_image_60d", 1, None),
                                            ("wan_40", 1, 2)])
def test_full_depth_properties(cuda, name, sub, batch):
    import torch
    from paper_2602_12529_gb300 import ffi
    cfg = synth.config(name) if batch is None else synth.config(name, batch=batch)
    blob = _blob_on_device(cfg, cuda)
    model = ffi.Dit(cfg, blob)
    B = cfg["batch"]
    x, txt, t = _inputs(cfg, cuda, B)
    v1 = _run(cfg, model, x, txt, t, cuda)
    v2 = _run(cfg, model, x, txt, t, cuda)
    assert torch.isfinite(v1).all()
    assert torch.equal(v1, v2)
    assert float(v1.float().std()) > 1e-3
    tail = (x[B - sub:].contiguous(), txt[B - sub:].contiguous(), t[B - sub:].contiguous())
    # the last `sub` samples alone: with the attention split allowed (the
    # default) the split blocks depend on the batch, so the velocities agree
    # to rounding; without it they are bit-identical
    vs = _run(cfg, model, *tail, cuda)
    assert float((vs - v1[B - sub:]).norm() / v1[B - sub:].norm()) <= 1e-2
    model.set_attention_split(False)
    vb = _run(cfg, model, x, txt, t, cuda)
    vs = _run(cfg, model, *tail, cuda)
    model.set_attention_split(True)
    assert torch.equal(vs, vb[B - sub:])
    assert float((vb - v1).norm() / v1.norm()) <= 1e-2
    assert ffi.ff_check_device_status() == 0
    del model, blob
    torch.cuda.empty_cache()
