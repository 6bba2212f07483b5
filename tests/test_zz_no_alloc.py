"""GPU check of ff_sde_step_logprob_noalloc, the SDE step variant for callers
that cannot allocate device memory (for example a plug-in inside a host
application that owns every device allocation): its scratch is a fixed array
inside the library instead of a caller workspace.  Its results must match
the workspace entry point ff_sde_step_logprob on the same inputs, call after
call (the shared array keeps the previous call's contents).

Kept in a file of its own that pytest collects last."""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import sde as osde

pytestmark = pytest.mark.gpu


def _run_both(ffi, dev, B, D, seed, mode):
    import torch
    grid = osde.time_grid(10, 3.0)
    t = np.array([grid[(seed + b) % 10] for b in range(B)], np.float32)
    tn = np.array([grid[(seed + b) % 10 + 1] for b in range(B)], np.float32)
    sg = osde.sigma_flow_sde(t, 0.7, 0.96).astype(np.float32)
    f = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    x = f(synth.gaussian((B, D), seed, "x"))
    v = f(synth.gaussian((B, D), seed + 1, "v"))
    e = f(synth.gaussian((B, D), seed + 2, "e"))
    tt, ttn, tsg = f(t), f(tn), f(sg)
    if mode == ffi.FF_SDE_SAMPLE:
        xn_ref, xn_new = torch.empty_like(x), torch.empty_like(x)
    else:
        given = f(synth.gaussian((B, D), seed + 3, "xn"))
        xn_ref, xn_new = given.clone(), given.clone()
    lp_ref = torch.zeros(B, dtype=torch.float32, device=dev)
    lp_new = torch.full((B,), 123.0, dtype=torch.float32, device=dev)
    ffi.ff_sde_step_logprob(x, v, e, xn_ref, tt, ttn, tsg, lp_ref, mode=mode)
    ffi.ff_sde_step_logprob_noalloc(x, v, e, xn_new, tt, ttn, tsg, lp_new, mode=mode)
    torch.cuda.synchronize()
    return xn_ref.cpu().numpy(), lp_ref.cpu().numpy(), xn_new.cpu().numpy(), lp_new.cpu().numpy()


def test_noalloc_matches_workspace_entry_point_on_consecutive_calls(cuda):
    from paper_2602_12529_gb300 import ffi
    # two calls in a row per case; the second case is smaller than the first,
    # so it runs over scratch the previous call left behind
    cases = [(4, 262144, 11, ffi.FF_SDE_SAMPLE), (4, 262144, 12, ffi.FF_SDE_SAMPLE),
             (3, 12340, 13, ffi.FF_SDE_EVAL), (3, 12340, 14, ffi.FF_SDE_EVAL)]
    for B, D, seed, mode in cases:
        xr, lr, xn, ln = _run_both(ffi, cuda, B, D, seed, mode)
        assert rms_rel(xn, xr) <= 1e-5
        assert np.max(np.abs(xn - xr)) <= 1e-5 * np.max(np.abs(xr))
        np.testing.assert_allclose(ln, lr, rtol=1e-3)
    assert ffi.ff_check_device_status() == 0


def test_noalloc_rejects_sizes_beyond_its_scratch(cuda):
    from paper_2602_12529_gb300 import ffi
    lib = ffi.lib()
    # the scratch limits are checked before the pointers, so these calls pass
    # no pointers at all and can never reach a launch
    # 65536 partial sums at most, 1024 per sample once D >= 2^22: 128
    # samples of 2^23 elements need 131072
    rc = lib.ff_sde_step_logprob_noalloc(128, 1 << 23, None, None, None, None, None, None, None, 0, 0, None, 1, None)
    assert rc == 2
    assert b"scratch" in lib.ff_last_error()
    # 4096 ticket counters at most
    rc = lib.ff_sde_step_logprob_noalloc(4097, 4, None, None, None, None, None, None, None, 0, 0, None, 1, None)
    assert rc == 2
    assert b"scratch" in lib.ff_last_error()
