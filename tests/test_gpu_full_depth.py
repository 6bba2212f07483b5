"""Full-depth parity of ff_dit_velocity against the fp64 oracle at the large
workload shapes (the network of Eq. 1 / Eq. 3, Sec. 3.1-3.2, with the
architecture readings of the Flux / Qwen-Image / WAN stand-ins).

Every block of every model runs on all of its tokens on both sides; only the
last block and the final layer of the oracle are restricted to 32 sampled
image rows of one sample.  Error that builds up through depth (bf16 GEMM
operands, bf16 attention inputs, fp32 residual stream) is what these cases
see and the one-block cases cannot.

* Flux-shaped rollout model: 8 double + 16 single blocks, H 3072, 512 text +
  1024 image tokens, run at its batch of 32; the last sample is checked.
* Qwen-Image-shaped model: 60 double blocks, 256 text + 4096 image tokens,
  D_txt 3584, run at its batch of 4; the last sample is checked.
* WAN-shaped model: all 40 blocks at full width (H 5120, 40 x 128 heads, MLP
  13824) and 512 text tokens, on a 3 x 16 x 16 latent grid (768 tokens; the
  full 32760-token grid would take the oracle hours per call), batch 1.

Weights are drawn on the device (tests/device_params.py) and handed to the
oracle as the same bf16 values.  Tolerance: output RMS-relative error 2e-2
(the bound for the bf16 velocity).  These run the oracle for minutes on the
host cores, hence also marked slow.
"""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from device_params import DeviceParams, draw_blob_on_device
from oracle import dit as odit

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

V_TOL = 2e-2


def _velocity_gpu(ffi, cfg, blob, dev, B):
    import torch
    model = ffi.Dit(cfg, blob)
    x = torch.from_numpy(synth.initial_latent(cfg, batch=B)).to(dev)
    txt = torch.from_numpy(synth.text_embeds(cfg, batch=B).view(np.int16)).to(dev).view(torch.bfloat16)
    t = torch.from_numpy(np.linspace(1.0, 0.1, B).astype(np.float32)).to(dev)
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=dev)
    v = torch.empty_like(x)
    model.ff_dit_velocity(x, txt, t, v, ws)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    out = v.cpu().numpy()
    model.close()
    del ws
    return out, t.cpu().numpy().astype(np.float64)


@pytest.mark.parametrize("name,over", [
    ("flux_8d16s", {}),
    ("qwen_image_60d", {}),
    ("wan_40", {"grid": (3, 16, 16), "batch": 1}),
])
def test_full_depth_velocity_matches_oracle(cuda, name, over):
    import torch
    from paper_2602_12529_gb300 import ffi
    cfg = synth.config(name, **over)
    wan = cfg["arch"] == "wan"
    B = cfg["batch"]
    specs, total = ffi.ff_dit_weight_layout(cfg)
    blob = draw_blob_on_device(specs, total, cuda, seed=3)
    v, t = _velocity_gpu(ffi, cfg, blob, cuda, B)
    assert np.isfinite(v).all()
    b = B - 1
    rows = np.sort(np.random.default_rng(5).choice(synth.n_img(cfg), 32, replace=False))
    P = DeviceParams(blob, specs, slice_mod=not wan)
    x = synth.initial_latent(cfg, batch=B)[b:b + 1]
    txt = odit.widen(synth.text_embeds(cfg, batch=B)[b:b + 1])
    vel = odit.wan_velocity if wan else odit.velocity
    want = vel(P, cfg, x, txt, t[b:b + 1], img_rows=rows)[0]
    err = rms_rel(v[b, rows], want)
    print(f"{name}: {cfg['n_double']}+{cfg['n_single']} blocks, RMS-rel {err:.3e}")
    assert err <= V_TOL, err
    del blob, P
    torch.cuda.empty_cache()
