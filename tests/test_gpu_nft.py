"""GPU parity of the DiffusionNFT loss (Eq. 2, ff_nft_loss) against the fp64
oracle (oracle/nft.py)."""
import numpy as np
import pytest

import synth
from oracle import nft as onft

pytestmark = pytest.mark.gpu


def _t(a, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(a, dtype=np.float32)).to(dev)


@pytest.mark.parametrize("B,D,reduce,beta", [(4, 262144, 0, 0.1), (4, 262144, 1, 1.0), (5, 12340, 0, 0.5),
                                             (2, 4, 1, 0.1), (64, 4096, 0, 2.0)])
def test_nft_loss_parity(cuda, B, D, reduce, beta):
    import torch
    from paper_2602_12529_gb300 import ffi
    v, vo = synth.gaussian((B, D), 50, "v"), synth.gaussian((B, D), 51, "v_old")
    eps, x0 = synth.gaussian((B, D), 52, "eps"), synth.gaussian((B, D), 53, "x0")
    r = synth.uniform((B,), 54, "r")
    loss = torch.zeros(1, dtype=torch.float32, device=cuda)
    grad = torch.empty((B, D), dtype=torch.float32, device=cuda)
    err = torch.empty((B, 2), dtype=torch.float32, device=cuda)
    ffi.ff_nft_loss(_t(v, cuda), _t(vo, cuda), _t(eps, cuda), _t(x0, cuda), _t(r, cuda), beta, reduce, loss, grad, err)
    torch.cuda.synchronize()
    want, want_g, want_e = onft.nft_loss(v, vo, eps, x0, r, beta, "mean" if reduce else "sum")
    np.testing.assert_allclose(err.cpu().numpy(), want_e, rtol=2e-5)
    assert abs(float(loss.item()) - want) <= 2e-5 * float(np.mean(want_e))
    g = grad.cpu().numpy()
    assert np.max(np.abs(g - want_g)) <= 1e-5 * np.max(np.abs(want_g))
    first = float(loss.item())
    ffi.ff_nft_loss(_t(v, cuda), _t(vo, cuda), _t(eps, cuda), _t(x0, cuda), _t(r, cuda), beta, reduce, loss)
    torch.cuda.synchronize()
    assert float(loss.item()) == first


def test_nft_special_cases(cuda):
    """beta = 1, r = 1 is the plain flow-matching loss (AWM with A = 1);
    v = v_old leaves one error for both policies."""
    import torch
    from paper_2602_12529_gb300 import ffi
    B, D = 3, 8192
    v, vo = synth.gaussian((B, D), 55, "v"), synth.gaussian((B, D), 56, "v_old")
    eps, x0 = synth.gaussian((B, D), 57, "eps"), synth.gaussian((B, D), 58, "x0")
    loss, loss_a = torch.zeros(1, device=cuda), torch.zeros(1, device=cuda)
    ones = _t(np.ones(B), cuda)
    ffi.ff_nft_loss(_t(v, cuda), _t(vo, cuda), _t(eps, cuda), _t(x0, cuda), ones, 1.0, 0, loss)
    ffi.ff_awm_loss(_t(v, cuda), _t(eps, cuda), _t(x0, cuda), ones, 0, loss_a)
    err = torch.empty((B, 2), device=cuda)
    ffi.ff_nft_loss(_t(vo, cuda), _t(vo, cuda), _t(eps, cuda), _t(x0, cuda), _t(np.full(B, 0.3), cuda), 0.7, 1,
                    torch.zeros(1, device=cuda), None, err)
    torch.cuda.synchronize()
    assert float(loss.item()) == pytest.approx(float(loss_a.item()), rel=1e-5)
    e = err.cpu().numpy()
    np.testing.assert_allclose(e[:, 0], e[:, 1], rtol=1e-5)
