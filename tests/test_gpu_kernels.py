"""GPU parity of the velocity path's kernels one by one (tcgen05 GEMM and its
epilogues, joint attention, LN-modulate, QK-RMSNorm + RoPE) against the
fp64 oracle on identical bf16 inputs, through the exported debug entry
points."""
import numpy as np
import pytest

import synth
from conftest import rms_rel
from oracle import dit as odit

pytestmark = pytest.mark.gpu


def _bf(shape, seed, std=1.0, tag="m"):
    return synth.bf16_bits(synth.gaussian(shape, seed, tag) * np.float32(std))


def _dev_bf16(bits, dev):
    import torch
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(torch.bfloat16)


def _host_bf16(t):
    import torch
    return odit.widen(t.view(torch.int16).cpu().numpy().view(np.uint16))


@pytest.mark.parametrize("M,N,K,act,f32", [
    (256, 256, 256, 0, 0), (300, 96, 72, 0, 1), (128, 64, 64, 0, 1), (4, 768, 256, 2, 0),
    (1000, 1024, 320, 1, 0), (2048, 3072, 3072, 0, 1), (513, 512, 1024, 1, 1),
    # few-row (GEMV) path: ragged row counts, fp32 / bf16 outputs, activations
    (3, 992, 320, 1, 1), (1, 64, 8, 0, 1), (8, 4096, 3072, 2, 0), (5, 6144, 256, 0, 1),
    (9, 512, 256, 0, 1)])
def test_gemm_parity(cuda, M, N, K, act, f32):
    import torch
    from paper_2602_12529_gb300 import ffi
    a = _bf((M, K), 1, 1.0, "A")
    b = _bf((N, K), 2, 0.05, "B")
    bias = _bf((N,), 3, 0.1, "bias")
    out = torch.zeros((M, N), dtype=torch.float32 if f32 else torch.bfloat16, device=cuda)
    ffi.ff_debug_gemm(_dev_bf16(a, cuda), _dev_bf16(b, cuda), _dev_bf16(bias, cuda), out, act)
    torch.cuda.synchronize()
    want = odit.linear(odit.widen(a), odit.widen(b), odit.widen(bias))
    if act == 1:
        want = odit.gelu_tanh(want)
    elif act == 2:
        want = odit.silu(want)
    got = out.cpu().numpy() if f32 else _host_bf16(out)
    tol = 2e-5 if (f32 and act == 0) else 5e-3
    assert rms_rel(got, want) <= tol, rms_rel(got, want)


def test_gemm_repeated_launches_are_identical(cuda):
    import torch
    from paper_2602_12529_gb300 import ffi
    M, N, K = 1024, 2048, 1536
    a, b = _dev_bf16(_bf((M, K), 4), cuda), _dev_bf16(_bf((N, K), 5, 0.05), cuda)
    o1 = torch.empty((M, N), dtype=torch.float32, device=cuda)
    o2 = torch.empty_like(o1)
    ffi.ff_debug_gemm(a, b, None, o1)
    ffi.ff_debug_gemm(a, b, None, o2)
    torch.cuda.synchronize()
    assert torch.equal(o1, o2)
    assert ffi.ff_check_device_status() == 0


@pytest.mark.parametrize("M,N,K,rps", [(384, 256, 256, 96), (4096 * 2, 3072, 3072, 4096), (200, 64, 128, 50)])
def test_gemm_gated_residual_parity(cuda, M, N, K, rps):
    import torch
    from paper_2602_12529_gb300 import ffi
    B = (M + rps - 1) // rps
    a = _bf((M, K), 6)
    w = _bf((N, K), 7, 0.03)
    bias = _bf((N,), 8, 0.1)
    x0 = synth.gaussian((M, N), 9, "x")
    gate = synth.gaussian((B, 3 * N), 10, "g")
    xr = torch.from_numpy(x0).to(cuda)
    gt = torch.from_numpy(gate).to(cuda)
    ffi.ff_debug_gemm_gated(_dev_bf16(a, cuda), _dev_bf16(w, cuda), _dev_bf16(bias, cuda), xr, gt[:, N:2 * N].contiguous(), rps)
    torch.cuda.synchronize()
    y = odit.linear(odit.widen(a), odit.widen(w), odit.widen(bias))
    g = gate.astype(np.float64)[np.arange(M) // rps, N:2 * N]
    want = x0.astype(np.float64) + g * y
    got = xr.cpu().numpy()
    assert rms_rel(got - x0, want - x0) <= 2e-5


@pytest.mark.parametrize("B,heads,d,n0,n1", [(2, 2, 64, 5, 70), (1, 3, 128, 32, 200), (2, 2, 128, 0, 130),
                                             (1, 2, 128, 512, 1024),
                                             # d = 128 runs on CTA pairs owning 512 query rows: partial
                                             # blocks, a second pair tile past the segment end, ragged K/V
                                             (2, 2, 128, 300, 777), (1, 1, 128, 1000, 24), (3, 1, 128, 130, 513),
                                             # more 256-row query blocks than SMs: each persistent CTA
                                             # runs several blocks back to back (one K/V step per block,
                                             # ragged segments, d = 64)
                                             (8, 40, 128, 0, 256), (6, 40, 128, 0, 100), (3, 64, 64, 77, 300)])
@pytest.mark.parametrize("launch", [1, 2])
def test_attention_parity(cuda, B, heads, d, n0, n1, launch):
    """Both kernel variants (1: persistent CTAs over strided query blocks;
    2: one 256-row query block per CTA) against the fp64 attention."""
    import torch
    from paper_2602_12529_gb300 import ffi
    lib = ffi.lib()
    assert lib.ff_debug_attention_launch(launch) == 0
    try:
        _attention_case(ffi, cuda, B, heads, d, n0, n1)
    finally:
        lib.ff_debug_attention_launch(0)


def _attention_case(ffi, cuda, B, heads, d, n0, n1):
    import torch
    H = heads * d
    ld0, ld1, ldo = 3 * H + 64, 3 * H, H + 128    # non-trivial pitches
    q0 = _bf((max(B * n0, 1), ld0), 11, 1.0, "q0")
    q1 = _bf((B * n1, ld1), 12, 1.0, "q1")
    qg0, qg1 = _dev_bf16(q0, cuda), _dev_bf16(q1, cuda)
    o0 = torch.zeros((max(B * n0, 1), ldo), dtype=torch.bfloat16, device=cuda)
    o1 = torch.zeros((B * n1, ldo), dtype=torch.bfloat16, device=cuda)
    ffi.ff_debug_attention(B, heads, d, qg0, o0, n0, qg1, o1, n1)
    torch.cuda.synchronize()
    w0, w1 = odit.widen(q0), odit.widen(q1)
    g0, g1 = _host_bf16(o0), _host_bf16(o1)
    for b in range(B):
        rows = np.concatenate([w0[b * n0:(b + 1) * n0, :3 * H], w1[b * n1:(b + 1) * n1, :3 * H]])
        q = rows[:, :H].reshape(-1, heads, d)
        k = rows[:, H:2 * H].reshape(-1, heads, d)
        v = rows[:, 2 * H:].reshape(-1, heads, d)
        want = odit.attention(q, k, v).reshape(-1, H)
        got = np.concatenate([g0[b * n0:(b + 1) * n0, :H], g1[b * n1:(b + 1) * n1, :H]])
        assert rms_rel(got, want) <= 1e-2, (b, rms_rel(got, want))
    # columns beyond H of the outputs are untouched
    assert float(o1[:, H:].float().abs().max()) == 0.0


@pytest.mark.parametrize("d", [64, 128])
def test_attention_variants_bit_identical(cuda, d):
    """The persistent variant (one CTA per SM running several query blocks
    as one K/V stream) and the one-block-per-CTA variant compute every block
    the same way: O and lse agree bit for bit (400 query blocks, two ragged
    segments)."""
    import torch
    from paper_2602_12529_gb300 import ffi
    lib = ffi.lib()
    B, heads, n0, n1 = 2, 40, 77, 1000
    H = heads * d
    q0 = _dev_bf16(_bf((B * n0, 3 * H), 21, 1.0, "q0"), cuda)
    q1 = _dev_bf16(_bf((B * n1, 3 * H), 22, 1.0, "q1"), cuda)
    outs = []
    for launch in (1, 2):
        o0 = torch.zeros((B * n0, H), dtype=torch.bfloat16, device=cuda)
        o1 = torch.zeros((B * n1, H), dtype=torch.bfloat16, device=cuda)
        lse = torch.zeros(B * heads * lib.ff_attention_lse_rows(n0, n1), device=cuda)
        assert lib.ff_debug_attention_launch(launch) == 0
        try:
            ffi.ff_attention_forward(B, heads, d, q0, o0, n0, q1, o1, n1, lse=lse)
            torch.cuda.synchronize()
        finally:
            lib.ff_debug_attention_launch(0)
        outs.append((o0, o1, lse))
    assert ffi.ff_check_device_status() == 0
    for a, b in zip(*outs):
        assert torch.equal(a, b)


def _split_applies(items, sms):
    rest = items % sms
    return 0 < rest and 2 * rest <= sms


@pytest.mark.parametrize("B,heads,d,n0,n1", [
    (1, 52, 128, 0, 1024),    # 208 blocks: one full round, 56 blocks split in two halves of 4 steps
    (1, 20, 64, 77, 300),     # 60 blocks, all split; the halves meet inside segment 1
    (2, 12, 128, 100, 420),   # 72 blocks, 5 steps: halves of 2 and 3 steps
    (1, 30, 128, 0, 200),     # 2 steps: halves of one step each
])
def test_attention_split_parity(cuda, B, heads, d, n0, n1):
    """The persistent launch that runs its last round's query blocks as two
    halves of their K/V steps (launch 3, with a scratch): O and lse against
    the fp64 attention and its log-sum-exp, and against the unsplit launch."""
    import math
    import torch
    from paper_2602_12529_gb300 import ffi
    lib = ffi.lib()
    H = heads * d
    sms = torch.cuda.get_device_properties(cuda).multi_processor_count
    items = B * heads * ((n0 + 255) // 256 + (n1 + 255) // 256)
    assert _split_applies(items, sms), (items, sms)
    q0 = _bf((max(B * n0, 1), 3 * H), 31, 1.0, "q0")
    q1 = _bf((B * n1, 3 * H), 32, 1.0, "q1")
    qg0, qg1 = _dev_bf16(q0, cuda), _dev_bf16(q1, cuda)
    L = lib.ff_attention_lse_rows(n0, n1)
    ws = torch.full((ffi.ff_attention_forward_workspace_size(d),), 0xA5, dtype=torch.uint8, device=cuda)
    res = {}
    for launch in (3, 1):
        o0 = torch.zeros((max(B * n0, 1), H), dtype=torch.bfloat16, device=cuda)
        o1 = torch.zeros((B * n1, H), dtype=torch.bfloat16, device=cuda)
        lse = torch.zeros(B * heads * L, device=cuda)
        assert lib.ff_debug_attention_launch(launch) == 0
        try:
            for _ in range(2):   # a second call finds the tickets as the first left them
                ffi.ff_attention_forward(B, heads, d, qg0, o0, n0, qg1, o1, n1, lse=lse, ws=ws)
            torch.cuda.synchronize()
        finally:
            lib.ff_debug_attention_launch(0)
        res[launch] = (_host_bf16(o0), _host_bf16(o1), lse.cpu().numpy().reshape(B, heads, L))
    assert ffi.ff_check_device_status() == 0
    w0, w1 = odit.widen(q0), odit.widen(q1)
    g0, g1, lse_h = res[3]
    for b in range(B):
        rows = np.concatenate([w0[b * n0:(b + 1) * n0, :3 * H], w1[b * n1:(b + 1) * n1, :3 * H]])
        q = rows[:, :H].reshape(-1, heads, d)
        k = rows[:, H:2 * H].reshape(-1, heads, d)
        v = rows[:, 2 * H:].reshape(-1, heads, d)
        want = odit.attention(q, k, v).reshape(-1, H)
        got = np.concatenate([g0[b * n0:(b + 1) * n0], g1[b * n1:(b + 1) * n1]])
        assert rms_rel(got, want) <= 1e-2, (b, rms_rel(got, want))
        want_lse = odit.attention_lse(q, k) / math.log(2.0)
        got_lse = np.concatenate([lse_h[b, :, :n0], lse_h[b, :, (n0 + 127) // 128 * 128:][:, :n1]], axis=1).T
        np.testing.assert_allclose(got_lse, want_lse, rtol=2e-4, atol=2e-4)
    # split and unsplit: the same attention up to fp32 rounding before the bf16 output
    u0, u1, ulse = res[1]
    got = np.concatenate([g0[:B * n0], g1])
    ref = np.concatenate([u0[:B * n0], u1])
    assert rms_rel(got, ref) <= 4e-3
    np.testing.assert_allclose(lse_h, ulse, rtol=1e-5, atol=1e-5)


def test_attention_split_flux_block_sampled(cuda):
    """The Flux double-block shape (4 samples, 24 heads of 128, 512 text +
    4096 image tokens: 1728 query blocks) in the launch the velocity network
    takes (automatic choice, with a scratch): 56 blocks past the 11 full
    rounds run split on 152 SMs.  Sampled rows of split and unsplit blocks
    against the fp64 attention and log-sum-exp."""
    import math
    import torch
    from paper_2602_12529_gb300 import ffi
    lib = ffi.lib()
    B, heads, d, n0, n1 = 4, 24, 128, 512, 4096
    H = heads * d
    N = n0 + n1
    q0 = _bf((B * n0, 3 * H), 41, 1.0, "q0")
    q1 = _bf((B * n1, 3 * H), 42, 1.0, "q1")
    o0 = torch.zeros((B * n0, H), dtype=torch.bfloat16, device=cuda)
    o1 = torch.zeros((B * n1, H), dtype=torch.bfloat16, device=cuda)
    L = lib.ff_attention_lse_rows(n0, n1)
    lse = torch.zeros(B * heads * L, device=cuda)
    ffi.ff_attention_forward(B, heads, d, _dev_bf16(q0, cuda), o0, n0, _dev_bf16(q1, cuda), o1, n1, lse=lse)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    g0, g1 = _host_bf16(o0), _host_bf16(o1)
    lse_h = lse.cpu().numpy().reshape(B, heads, L)
    w0, w1 = odit.widen(q0), odit.widen(q1)
    qpairs = n0 // 256 + n1 // 256
    sms = torch.cuda.get_device_properties(cuda).multi_processor_count
    items = B * heads * qpairs
    split_first = items // sms * sms if _split_applies(items, sms) else items
    rng = np.random.default_rng(7)
    # (b, h, joint row): rows of the last (split) blocks, the first block and a middle one
    picks = []
    for it in (items - 1, items - 2, split_first, 0, items // 2):
        qp, bh = it % qpairs, it // qpairs
        b, h = bh // heads, bh % heads
        base = qp * 256 if qp < n0 // 256 else n0 + (qp - n0 // 256) * 256
        picks += [(b, h, base + int(r)) for r in rng.choice(256, 6, replace=False)]
    for b in sorted({p[0] for p in picks}):
        rows = np.concatenate([w0[b * n0:(b + 1) * n0, :3 * H], w1[b * n1:(b + 1) * n1, :3 * H]])
        for bb, h, r in picks:
            if bb != b:
                continue
            q = rows[r:r + 1, h * d:(h + 1) * d].reshape(1, 1, d)
            k = rows[:, H + h * d:H + (h + 1) * d].reshape(N, 1, d)
            v = rows[:, 2 * H + h * d:2 * H + (h + 1) * d].reshape(N, 1, d)
            want = odit.attention(q, k, v).reshape(d)
            got = (g0[b * n0 + r] if r < n0 else g1[b * n1 + r - n0])[h * d:(h + 1) * d]
            assert rms_rel(got, want) <= 1e-2, (b, h, r)
            want_lse = odit.attention_lse(q, k).reshape(()) / math.log(2.0)
            got_lse = lse_h[b, h, r if r < n0 else (n0 + 127) // 128 * 128 + r - n0]
            assert abs(got_lse - want_lse) <= 2e-4 * max(1.0, abs(want_lse)), (b, h, r)


@pytest.mark.parametrize("rows,H,tps", [(96, 256, 32), (1000, 3072, 250)])
def test_ln_modulate_parity(cuda, rows, H, tps):
    import torch
    from paper_2602_12529_gb300 import ffi
    B = (rows + tps - 1) // tps
    x = synth.gaussian((rows, H), 1, "x") * np.float32(3.0) + np.float32(0.5)
    mods = synth.gaussian((B, 4 * H), 2, "m") * np.float32(0.2)
    out = torch.zeros((rows, H), dtype=torch.bfloat16, device=cuda)
    ffi.ff_debug_ln_modulate(torch.from_numpy(x).to(cuda), torch.from_numpy(mods).to(cuda), H, 3 * H, tps, out)
    torch.cuda.synchronize()
    m = mods.astype(np.float64)[np.arange(rows) // tps]
    want = odit.modulate(odit.layer_norm(x.astype(np.float64)), m[:, H:2 * H], m[:, 3 * H:])
    assert rms_rel(_host_bf16(out), want) <= 5e-3


@pytest.mark.parametrize("d,axes,grid,rows_txt", [(64, (8, 28, 28), (1, 8, 8), 32), (128, (16, 56, 56), (1, 16, 16), 20),
                                                   (128, (44, 42, 42), (3, 5, 7), 0)])
def test_qk_norm_rope_parity(cuda, d, axes, grid, rows_txt):
    import torch
    from paper_2602_12529_gb300 import ffi
    heads = 3
    H = heads * d
    n_img = grid[0] * grid[1] * grid[2]
    B = 2
    rows = rows_txt + B * n_img
    qkv = _bf((rows, 3 * H), 3, 1.5, "qkv")
    qs = synth.bf16_bits(1.0 + synth.gaussian((d,), 4, "qs") * np.float32(0.1))
    ks = synth.bf16_bits(1.0 + synth.gaussian((d,), 5, "ks") * np.float32(0.1))
    g = _dev_bf16(qkv, cuda)
    ffi.ff_debug_qk_norm_rope(g, rows_txt, heads, d, _dev_bf16(qs, cuda), _dev_bf16(ks, cuda), grid, axes, 10000.0)
    torch.cuda.synchronize()
    got = _host_bf16(g)
    w = odit.widen(qkv)
    pos = np.zeros((rows, 3))
    img = odit.image_positions(grid)
    pos[rows_txt:] = img[(np.arange(rows - rows_txt)) % n_img]
    ang = odit.rope_angles(pos, axes)
    for part, sc in ((0, qs), (1, ks)):
        x = w[:, part * H:(part + 1) * H].reshape(rows, heads, d)
        want = odit.apply_rope(odit.rms_norm(x, odit.widen(sc)), ang).reshape(rows, H)
        assert rms_rel(got[:, part * H:(part + 1) * H], want) <= 6e-3
    np.testing.assert_array_equal(got[:, 2 * H:], w[:, 2 * H:])   # v untouched
