"""GPU parity of the attention backward (dq, dk, dv; head dim 64 and 128) and
of the forward's per-row log-sum-exp against the fp64 oracle, over joint
[segment 0; segment 1] sequences with ragged segment lengths."""
import math

import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import dit as odit

pytestmark = pytest.mark.gpu


def _bits(shape, seed, tag, std=1.0):
    return synth.bf16_bits(synth.gaussian(shape, seed, tag) * np.float32(std))


def _dev(bits, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(torch.bfloat16)


def _host(t):
    import torch
    return odit.widen(t.view(torch.int16).cpu().numpy().view(np.uint16))


@pytest.mark.parametrize("d,B,heads,n0,n1", [(128, 2, 2, 5, 70), (128, 1, 3, 32, 200), (128, 2, 2, 0, 130),
                                             (128, 1, 2, 300, 777), (128, 1, 2, 512, 4096), (128, 1, 8, 512, 4096),
                                             (64, 4, 4, 32, 64), (64, 2, 2, 5, 70), (64, 1, 3, 300, 777)])
def test_attention_backward_parity(cuda, d, B, heads, n0, n1):
    import torch
    from paper_2602_12529_gb300 import ffi
    H = heads * d
    q0 = _bits((max(B * n0, 1), 3 * H), 31, "bq0")
    q1 = _bits((B * n1, 3 * H), 32, "bq1")
    g0 = _bits((max(B * n0, 1), H), 33, "bg0")
    g1 = _bits((B * n1, H), 34, "bg1")
    L = ffi.lib().ff_attention_lse_rows(n0, n1)
    lse = torch.zeros(B * heads * L, dtype=torch.float32, device=cuda)
    o0 = torch.zeros((max(B * n0, 1), H), dtype=torch.bfloat16, device=cuda)
    o1 = torch.zeros((B * n1, H), dtype=torch.bfloat16, device=cuda)
    ffi.ff_attention_forward(B, heads, d, _dev(q0, cuda), o0, n0, _dev(q1, cuda), o1, n1, lse=lse)
    dq0 = torch.zeros((max(B * n0, 1), 3 * H + 64), dtype=torch.bfloat16, device=cuda)
    dq1 = torch.zeros((B * n1, 3 * H + 64), dtype=torch.bfloat16, device=cuda)
    ffi.ff_attention_backward(B, heads, d, (n0, _dev(q0, cuda), o0, _dev(g0, cuda), dq0),
                              (n1, _dev(q1, cuda), o1, _dev(g1, cuda), dq1), lse)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    w0, w1, gw0, gw1 = odit.widen(q0), odit.widen(q1), odit.widen(g0), odit.widen(g1)
    lse_h = lse.cpu().numpy().reshape(B, heads, L)
    d0, d1 = _host(dq0), _host(dq1)
    for b in range(B):
        rows = np.concatenate([w0[b * n0:(b + 1) * n0], w1[b * n1:(b + 1) * n1]])
        dout = np.concatenate([gw0[b * n0:(b + 1) * n0], gw1[b * n1:(b + 1) * n1]]).reshape(-1, heads, d)
        q = rows[:, :H].reshape(-1, heads, d)
        k = rows[:, H:2 * H].reshape(-1, heads, d)
        v = rows[:, 2 * H:].reshape(-1, heads, d)
        # forward log-sum-exp (base 2) of every real row
        want_lse = odit.attention_lse(q, k) / math.log(2.0)
        got_lse = np.concatenate([lse_h[b, :, :n0], lse_h[b, :, (n0 + 127) // 128 * 128:][:, :n1]], axis=1).T
        np.testing.assert_allclose(got_lse, want_lse, rtol=2e-4, atol=2e-4)
        # gradients
        dq, dk, dv = odit.attention_backward(q, k, v, dout)
        got = np.concatenate([d0[b * n0:(b + 1) * n0], d1[b * n1:(b + 1) * n1]])
        for name, want, c in (("dq", dq, 0), ("dk", dk, H), ("dv", dv, 2 * H)):
            err = rms_rel(got[:, c:c + H], want.reshape(-1, H))
            assert err <= 2e-2, (b, name, err)
    # columns past 3H are not written
    assert float(dq1[:, 3 * H:].float().abs().max()) == 0.0


@pytest.mark.parametrize("d,B,heads,nq,nk", [(128, 2, 2, 130, 77), (128, 1, 3, 300, 512), (64, 2, 4, 5, 200),
                                             (64, 1, 2, 777, 33), (128, 1, 2, 64, 3)])
def test_cross_attention_backward_parity(cuda, d, B, heads, nq, nk):
    """Latent queries against text keys / values (the WAN block's
    cross-attention): lse and dq, dk, dv against the fp64 definitions."""
    import torch
    from paper_2602_12529_gb300 import ffi
    H = heads * d
    qb = _bits((B * nq, H), 41, "cq")
    kvb = _bits((B * nk, 2 * H), 42, "ckv")
    gb = _bits((B * nq, H), 43, "cg")
    L = ffi.lib().ff_attention_lse_rows(nq, 0)
    lse = torch.zeros(B * heads * L, dtype=torch.float32, device=cuda)
    q, kv = _dev(qb, cuda), _dev(kvb, cuda)
    o = torch.zeros((B * nq, H), dtype=torch.bfloat16, device=cuda)
    ffi.ff_cross_attention_forward(B, heads, d, q, nq, kv, nk, o, lse=lse)
    dq = torch.zeros((B * nq, H), dtype=torch.bfloat16, device=cuda)
    dkv = torch.zeros((B * nk, 2 * H + 64), dtype=torch.bfloat16, device=cuda)
    ffi.ff_cross_attention_backward(B, heads, d, q, nq, o, _dev(gb, cuda), dq, kv, nk, dkv, lse)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    wq, wkv, wg = odit.widen(qb), odit.widen(kvb), odit.widen(gb)
    lse_h = lse.cpu().numpy().reshape(B, heads, L)
    gq, gkv = _host(dq), _host(dkv)
    for b in range(B):
        qh = wq[b * nq:(b + 1) * nq].reshape(nq, heads, d)
        kh = wkv[b * nk:(b + 1) * nk, :H].reshape(nk, heads, d)
        vh = wkv[b * nk:(b + 1) * nk, H:].reshape(nk, heads, d)
        gh = wg[b * nq:(b + 1) * nq].reshape(nq, heads, d)
        np.testing.assert_allclose(lse_h[b, :, :nq].T, odit.attention_lse(qh, kh) / math.log(2.0),
                                   rtol=2e-4, atol=2e-4)
        want_dq, want_dk, want_dv = odit.attention_backward(qh, kh, vh, gh)
        for name, got, want in (("dq", gq[b * nq:(b + 1) * nq], want_dq),
                                ("dk", gkv[b * nk:(b + 1) * nk, :H], want_dk),
                                ("dv", gkv[b * nk:(b + 1) * nk, H:2 * H], want_dv)):
            err = rms_rel(got, want.reshape(-1, H))
            assert err <= 2e-2, (b, name, err)
    assert float(dkv[:, 2 * H:].float().abs().max()) == 0.0
