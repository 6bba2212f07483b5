"""GPU parity of ff_gemm with every operand layout (the Linear forward, its
input gradient and its weight gradient) against the fp64 oracle, on shapes
that reach the single-CTA kernel (N 64 / 128 / 256 tiles) and the CTA-pair
kernel (N % 256 == 0, M >= 512), with ragged M, N and K."""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import dit as odit
from oracle import linalg

pytestmark = pytest.mark.gpu

LAYOUTS = [("MK", "NK"), ("MK", "KN"), ("KM", "NK"), ("KM", "KN")]


def _pad8(n):
    return (n + 7) // 8 * 8 + 8   # a leading dimension past the row, multiple of 8


def _operand(rows, cols, seed, tag):
    """bf16 bits of a [rows, cols] matrix stored with a padded row pitch."""
    ld = _pad8(cols)
    full = synth.bf16_bits(synth.gaussian((rows, ld), seed, tag))
    return full, ld


@pytest.mark.parametrize("al,bl", LAYOUTS)
@pytest.mark.parametrize("M,N,K,act,f32", [(300, 96, 72, 0, 1), (128, 64, 64, 1, 0), (1000, 256, 320, 0, 1),
                                           (512, 256, 192, 2, 0), (2048, 3072, 1024, 0, 1), (777, 512, 520, 1, 1)])
def test_gemm_layout_parity(cuda, al, bl, M, N, K, act, f32):
    import torch
    from paper_2602_12529_gb300 import ffi
    a_rows, a_cols = (M, K) if al == "MK" else (K, M)
    b_rows, b_cols = (N, K) if bl == "NK" else (K, N)
    A, lda = _operand(a_rows, a_cols, 1 + M, "ga")
    Bm, ldb = _operand(b_rows, b_cols, 2 + N, "gb")
    bias = synth.bf16_bits(synth.gaussian((N,), 3, "gbias"))
    dev = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(cuda).view(torch.bfloat16)
    Ag, Bg = dev(A)[:, :a_cols], dev(Bm)[:, :b_cols]
    out = torch.zeros((M, N + 32), dtype=torch.float32 if f32 else torch.bfloat16, device=cuda)[:, :N]
    ffi.ff_gemm(Ag, ffi.FF_A_MK if al == "MK" else ffi.FF_A_KM, Bg, ffi.FF_B_NK if bl == "NK" else ffi.FF_B_KN,
                out, bias=dev(bias), act=act)
    torch.cuda.synchronize()
    want = linalg.gemm(odit.widen(A)[:, :a_cols], odit.widen(Bm)[:, :b_cols], al, bl, odit.widen(bias),
                       {0: "none", 1: "gelu", 2: "silu"}[act])
    got = out.float().cpu().numpy()
    assert rms_rel(got, want) <= (2e-5 if f32 else 5e-3), rms_rel(got, want)


def test_linear_backward_products(cuda):
    """dx = dy W and dW = dy^T x for a Linear on 4096 tokens, 3072 -> 3072."""
    import torch
    from paper_2602_12529_gb300 import ffi
    T, Nin, Nout = 4096, 3072, 3072
    x = synth.bf16_bits(synth.gaussian((T, Nin), 11, "lx"))
    W = synth.bf16_bits(synth.gaussian((Nout, Nin), 12, "lw") * np.float32(0.02))
    dy = synth.bf16_bits(synth.gaussian((T, Nout), 13, "ldy"))
    dev = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(cuda).view(torch.bfloat16)
    dx = torch.empty((T, Nin), dtype=torch.float32, device=cuda)
    dW = torch.empty((Nout, Nin), dtype=torch.float32, device=cuda)
    ffi.ff_gemm(dev(dy), ffi.FF_A_MK, dev(W), ffi.FF_B_KN, dx)
    ffi.ff_gemm(dev(dy), ffi.FF_A_KM, dev(x), ffi.FF_B_KN, dW)
    torch.cuda.synchronize()
    rng = np.random.default_rng(0)
    rows = rng.choice(T, 64, replace=False)
    wrows = rng.choice(Nout, 64, replace=False)
    xw, Ww, dyw = odit.widen(x), odit.widen(W), odit.widen(dy)
    want_dx = dyw[rows] @ Ww
    want_dW = dyw[:, wrows].T @ xw
    assert rms_rel(dx.cpu().numpy()[rows], want_dx) <= 2e-5
    assert rms_rel(dW.cpu().numpy()[wrows], want_dW) <= 2e-5
