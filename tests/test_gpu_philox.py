"""GPU parity of the counter-based noise (ff_philox_normal) with the fp64
oracle (oracle/philox.py), and of the SDE step that draws it in the kernel
(ff_sde_step_logprob_philox) with the step fed the same noise from memory."""
import numpy as np
import pytest

from oracle import philox
from oracle import sde as osde

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("B,D,seed,stream", [(3, 4096 + 64, 0, 0), (2, 1 << 16, 12345, 7),
                                             (1, 8, (1 << 40) + 3, 4000000000), (5, 262144, 2024, 1),
                                             (32, 65536, 3, 9), (1, 2096640, 77, 1)])
def test_philox_normal_matches_oracle(cuda, B, D, seed, stream):
    import torch
    from paper_2602_12529_gb300 import ffi
    out = torch.empty((B, D), dtype=torch.float32, device=cuda)
    ffi.ff_philox_normal(out, seed, stream)
    torch.cuda.synchronize()
    got = out.cpu().numpy().astype(np.float64)
    want = philox.philox_normal(B, D, seed, stream)
    # fp32 log / sqrt / sincospi of the same exact uniforms: a few ulp
    err = np.abs(got - want) / np.maximum(1.0, np.abs(want))
    assert err.max() <= 4e-6, err.max()


@pytest.mark.parametrize("reduce", [0, 1])
def test_sde_step_with_in_kernel_noise_equals_the_step_fed_that_noise(cuda, reduce):
    import torch
    from paper_2602_12529_gb300 import ffi
    rng = np.random.default_rng(3)
    B, D = 4, 64 * 1024 + 64
    T = lambda a: torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(cuda)
    x, v = T(rng.standard_normal((B, D))), T(rng.standard_normal((B, D)))
    t = T([0.95, 0.7, 0.5, 0.3])
    tn = T([0.85, 0.6, 0.45, 0.1])
    sg = T([0.7, 0.7, 0.3, 0.9])
    seed, stream = 99, 2
    eps = torch.empty((B, D), dtype=torch.float32, device=cuda)
    ffi.ff_philox_normal(eps, seed, stream)
    xn_a, xn_b = torch.empty_like(x), torch.empty_like(x)
    lp_a, lp_b = torch.empty(B, device=cuda), torch.empty(B, device=cuda)
    ffi.ff_sde_step_logprob(x, v, eps, xn_a, t, tn, sg, lp_a, mode=ffi.FF_SDE_SAMPLE, reduce=reduce)
    ffi.ff_sde_step_logprob_philox(x, v, xn_b, t, tn, sg, lp_b, seed, stream, reduce=reduce)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    assert torch.equal(xn_a, xn_b) and torch.equal(lp_a, lp_b)
    # and against the oracle's step on the oracle's noise
    e64 = philox.philox_normal(B, D, seed, stream)
    h = lambda a: a.cpu().numpy().astype(np.float64)
    xn_ref, _ = osde.sde_step_logprob(h(x), h(v), h(t), h(tn), h(sg), eps=e64)
    got = h(xn_b)
    for b in range(B):
        assert np.sqrt(np.mean((got[b] - xn_ref[b]) ** 2)) <= 1e-5 * np.sqrt(np.mean(xn_ref[b] ** 2))


def test_rollout_with_device_noise_equals_the_rollout_fed_that_noise(cuda):
    import torch
    import synth
    from paper_2602_12529_gb300 import ffi, weights
    cfg = synth.config("tiny_mmdit")
    B, S = cfg["batch"], 4
    model = ffi.Dit(cfg, weights.pack(cfg, lambda n, s: synth.weight(n, s, synth.weight_kind(n), 0), cuda))
    x0 = torch.from_numpy(synth.initial_latent(cfg)).to(cuda)
    txt = torch.from_numpy(synth.text_embeds(cfg).view(np.int16)).to(cuda).view(torch.bfloat16)
    tg, sg = ffi.ff_sde_schedule(ffi.FF_SCHED_FLOW_SDE, S, 1.0, 0.7, 0.96)
    t = torch.tensor(tg, dtype=torch.float32, device=cuda)
    sigma = torch.tensor(sg, dtype=torch.float32, device=cuda)
    seed = 5150
    eps = torch.empty((S,) + tuple(x0.shape), dtype=torch.float32, device=cuda)
    for k in range(S):
        ffi.ff_philox_normal(eps[k], seed, k)
    xa, xb = x0.clone(), x0.clone()
    la, lb = torch.empty((B, S), device=cuda), torch.empty((B, S), device=cuda)
    ta = torch.empty((S + 1,) + tuple(x0.shape), device=cuda)
    tb = torch.empty_like(ta)
    model.ff_rollout(xa, txt, t, sigma, eps, la, traj=ta)
    model.ff_rollout_philox(xb, txt, t, sigma, seed, lb, traj=tb)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    assert torch.equal(ta, tb) and torch.equal(la, lb) and torch.equal(xa, xb)
    # another seed gives another trajectory
    xc = x0.clone()
    model.ff_rollout_philox(xc, txt, t, sigma, seed + 1, lb)
    torch.cuda.synchronize()
    assert not torch.equal(xc, xa)
