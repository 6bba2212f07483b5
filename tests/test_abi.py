"""CPU checks of the C ABI: the library builds and loads, exports every symbol
the headers declare, and its host-only entry points (schedule, weight layout,
workspace queries, argument validation) behave without a GPU."""
import ctypes as C
import os
import re

import numpy as np
import pytest

import synth
from oracle import dit as odit
from oracle import sde as osde
from paper_2602_12529_gb300 import build, ffi

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def L():
    build.build()
    return ffi.lib()


def _declared():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        src = open(os.path.join(ROOT, "include", h)).read()
        names |= set(re.findall(r"^\s*(?:const\s+char\s*\*|int)\s+(ff_\w+)\s*\(", src, re.M))
    return names


def test_exports_every_declared_symbol(L):
    declared = _declared()
    assert len(declared) >= 19
    for name in declared:
        assert hasattr(L, name), name
    assert set(ffi._SIGS) >= declared


def test_version_and_error_string(L):
    assert ffi.ff_version() >= 100
    assert isinstance(L.ff_last_error(), bytes)


@pytest.mark.parametrize("steps,shift", [(4, 1.0), (10, 3.0), (1, 3.0)])
def test_schedule_matches_oracle(L, steps, shift):
    t, s = ffi.ff_sde_schedule(ffi.FF_SCHED_FLOW_SDE, steps, shift, 0.7, 0.96)
    np.testing.assert_allclose(t, osde.time_grid(steps, shift), rtol=0, atol=1e-15)
    np.testing.assert_allclose(s, osde.sigma_flow_sde(np.array(t[:-1]), 0.7, 0.96), rtol=1e-15)
    _, s2 = ffi.ff_sde_schedule(ffi.FF_SCHED_DANCE_SDE, steps, shift, 0.3, 0.96)
    assert s2 == [0.3] * steps
    _, s3 = ffi.ff_sde_schedule(ffi.FF_SCHED_ODE, steps, shift, 0.3, 0.96)
    assert s3 == [0.0] * steps


def test_schedule_rejects_bad_arguments(L):
    with pytest.raises(ffi.FFError):
        ffi.ff_sde_schedule(7, 4)
    with pytest.raises(ffi.FFError):
        ffi.ff_sde_schedule(ffi.FF_SCHED_FLOW_SDE, 0)
    with pytest.raises(ffi.FFError):
        ffi.ff_sde_schedule(ffi.FF_SCHED_FLOW_SDE, 4, 1.0, 0.7, 1.0)


@pytest.mark.parametrize("name", list(synth.CONFIGS))
def test_weight_layout_matches_oracle_parameters(L, name):
    cfg = synth.config(name)
    specs, total = ffi.ff_dit_weight_layout(cfg)
    want = odit.wan_param_specs(cfg) if cfg["arch"] == "wan" else odit.param_specs(cfg)
    assert [(n, tuple(s)) for n, _, s in specs] == [(n, tuple(s)) for n, s in want]
    offs = [o for _, o, _ in specs]
    assert all(o % 64 == 0 for o in offs)
    assert offs == sorted(offs)
    last_n, last_o, last_s = specs[-1]
    assert total >= last_o + int(np.prod(last_s))


def test_workspace_queries(L):
    # SDE: a fixed 256 KiB ticket region, then one fp32 partial per
    # 4096-element chunk (at most 1024 per sample)
    n1 = ffi.ff_sde_workspace_size(4, 262144)
    assert n1 == 256 * 1024 + 4 * 64 * 4
    # loss: a 16-byte ticket, then one fp32 partial per block (at most 1216)
    assert ffi.ff_grpo_loss_workspace_size(32, 10) == 16 + 4
    assert ffi.ff_grpo_loss_workspace_size(1 << 20, 64) == 16 + 1216 * 4
    assert ffi.ff_sde_workspace_size(4, 1 << 26) == 256 * 1024 + 4 * 1024 * 4
    with pytest.raises(ffi.FFError):
        ffi.ff_sde_workspace_size(0, 16)
    # attention backward: -D and a copy of -lse, each fp32 [B, heads, L] with
    # L = pad128(n0) + pad128(n1)
    sz = ffi._SZ()
    assert L.ff_attention_backward_workspace_size(2, 3, 100, 200, C.byref(sz)) == 0
    assert sz.value == 2 * 2 * 3 * (128 + 256) * 4
    # attention forward's optional split scratch: per split query block (at
    # most 96) both halves' fp32 O of both 128-row tiles, their (m, l), 8 tickets
    for d in (64, 128):
        assert ffi.ff_attention_forward_workspace_size(d) == 96 * (2 * 2 * 128 * d * 4 + 2 * 2 * 128 * 8 + 8 * 4)
    with pytest.raises(ffi.FFError):
        ffi.ff_attention_forward_workspace_size(96)


def _plan(L, items, sms, steps, have_ws, mode=0):
    import ctypes as C
    pers, grid, first, n = C.c_int(), C.c_int64(), C.c_int64(), C.c_int64()
    rc = L.ff_debug_attention_plan(items, sms, steps, have_ws, mode, C.byref(pers), C.byref(grid), C.byref(first),
                                   C.byref(n))
    assert rc == 0, L.ff_last_error()
    return pers.value, grid.value, first.value, n.value


def test_attention_launch_plan(L):
    """The attention launcher's choice of variant, grid and split (host
    arithmetic, no GPU): persistent below 16 query blocks per SM or with at
    most 128 K/V steps per block, one block per CTA otherwise; a persistent
    launch with the scratch splits a last round that is at most half full."""
    # Flux block (B 4, 24 heads, 512 + 4096 tokens): 1728 blocks of 36 steps
    # on 152 SMs, 11 rounds + 56 -> 56 blocks split over CTAs 0 .. 111
    assert _plan(L, 1728, 152, 36, 1) == (1, 152, 1672, 56)
    assert _plan(L, 1728, 152, 36, 0) == (1, 152, 0, 0)           # no scratch: unsplit
    assert _plan(L, 1728, 152, 36, 1, mode=1) == (1, 152, 0, 0)   # forced unsplit
    assert _plan(L, 1728, 152, 36, 1, mode=2) == (0, 1728, 0, 0)  # forced one block per CTA
    # WAN self-attention (32760 tokens, 40 heads): 5120 blocks of 256 steps
    assert _plan(L, 5120, 152, 256, 1) == (0, 5120, 0, 0)
    # forced persistent with the split: 104 left over, more than half of 152
    assert _plan(L, 5120, 152, 256, 1, mode=3) == (1, 152, 0, 0)
    # WAN cross-attention (512 text keys): 4 steps, persistent, 104 left over
    assert _plan(L, 5120, 152, 4, 1) == (1, 152, 0, 0)
    # fewer blocks than SMs: every block split, two CTAs each
    assert _plan(L, 60, 152, 4, 1) == (1, 120, 0, 60)
    assert _plan(L, 76, 152, 4, 1) == (1, 152, 0, 76)
    assert _plan(L, 77, 152, 4, 1) == (1, 77, 0, 0)               # 154 halves do not fit
    # a single K/V step cannot be halved
    assert _plan(L, 60, 152, 1, 1) == (1, 60, 0, 0)
    # an exact number of rounds leaves nothing to split
    assert _plan(L, 304, 152, 36, 1) == (1, 152, 0, 0)
    # at most 96 split blocks (the scratch's capacity), even on a larger GPU
    assert _plan(L, 256 + 96, 256, 36, 1) == (1, 256, 256, 96)
    assert _plan(L, 256 + 100, 256, 36, 1) == (1, 256, 0, 0)
    # 16 blocks per SM and more than 128 steps: one block per CTA
    assert _plan(L, 16 * 152, 152, 129, 1) == (0, 16 * 152, 0, 0)
    assert _plan(L, 16 * 152 - 1, 152, 129, 1)[0] == 1
    import ctypes as C
    x = C.c_int(); y = C.c_int64()
    assert L.ff_debug_attention_plan(0, 152, 4, 1, 0, C.byref(x), C.byref(y), C.byref(y), C.byref(y)) == 1
    assert L.ff_debug_attention_plan(10, 152, 4, 1, 4, C.byref(x), C.byref(y), C.byref(y), C.byref(y)) == 1
    assert L.ff_debug_attention_plan(10, 152, 4, 1, 0, None, C.byref(y), C.byref(y), C.byref(y)) == 1


def test_attention_entries_reject_short_buffers(L):
    """Buffers too small for the launch are refused before anything runs:
    in the Python binding by shape (host tensors suffice, nothing reaches
    the library), and in the C entries by the output pitch (null pointers:
    nothing could be launched even past the check)."""
    import torch
    from paper_2602_12529_gb300 import ffi
    B, heads, d, n0, n1 = 2, 2, 64, 0, 100
    H = heads * d
    q1 = torch.zeros(B * n1, 3 * H, dtype=torch.bfloat16)
    o1 = torch.zeros(B * n1, H, dtype=torch.bfloat16)
    dummy = torch.zeros(1, 3 * H, dtype=torch.bfloat16)
    with pytest.raises(ValueError, match="out1"):
        ffi.ff_attention_forward(B, heads, d, dummy, dummy, n0, q1, o1[:B * n1 - 1], n1)
    with pytest.raises(ValueError, match="out1"):
        ffi.ff_attention_forward(B, heads, d, dummy, dummy, n0, q1, o1[:, :H - 8].contiguous(), n1)
    with pytest.raises(ValueError, match="qkv1"):
        ffi.ff_attention_forward(B, heads, d, dummy, dummy, n0, q1[:, :2 * H].contiguous(), o1, n1)
    with pytest.raises(ValueError, match="lse"):
        ffi.ff_attention_forward(B, heads, d, dummy, dummy, n0, q1, o1, n1, lse=torch.zeros(10))
    with pytest.raises(ValueError, match="kv"):
        ffi.ff_cross_attention_forward(B, heads, d, o1, n1, o1[:8], 8, o1)
    with pytest.raises(ValueError, match="dqkv1"):
        ffi.ff_attention_backward(B, heads, d, (0, None, None, None, None), (n1, q1, o1, o1, o1), torch.zeros(1))
    # C entries: an output pitch below heads * head_dim
    rc = L.ff_attention_forward(B, heads, d, 0, None, 0, None, 0, n1, None, 3 * H, None, H - 8, None, None, 0, None)
    assert rc == 1 and b"pitch" in L.ff_last_error()
    rc = L.ff_cross_attention_forward(B, heads, d, n1, None, H, 8, None, 2 * H, None, H - 8, None, None)
    assert rc == 1 and b"pitch" in L.ff_last_error()


def test_host_validation_without_gpu(L):
    # every one of these is rejected before any CUDA call is made
    assert L.ff_debug_attention_launch(4) == 1          # variants are 0 to 3
    assert L.ff_debug_attention_launch(3) == 0          # returns the previous setting
    assert L.ff_debug_attention_launch(0) == 3
    rc = L.ff_sde_step_logprob(0, 16, None, None, None, None, None, None, None, 0, 0, None, 1, None, 0, None)
    assert rc == 1
    rc = L.ff_sde_step_logprob(2, 18, 16, 16, 16, 16, 16, 16, 16, 0, 0, 16, 1, 16, 1 << 20, None)
    assert rc == 2   # D % 4 != 0
    rc = L.ff_sde_step_logprob(2, 16, 16, 16, 16, 16, 16, 16, 16, 5, 0, 16, 1, 16, 1 << 20, None)
    assert rc == 1   # bad mode
    rc = L.ff_sde_step_logprob(2, 16, 16, 16, 16, 16, 16, 16, 16, 0, 0, 16, 1, 16, 8, None)
    assert rc == 3   # workspace too small
    assert L.ff_group_advantage(0, 4, 16, 1e-4, 16, None) == 1
    assert L.ff_group_advantage(1, 5000, 16, 1e-4, 16, None) == 2
    assert L.ff_grpo_loss(4, 1, None, 16, 16, 0.2, 0.2, 16, None, 16, 64, None) == 1
    assert L.ff_grpo_loss(4, 1, 16, 16, 16, 1.5, 0.2, 16, None, 16, 64, None) == 1
    assert L.ff_grpo_loss(4, 1, 16, 16, 16, 0.2, 0.2, 16, None, 16, 0, None) == 3
    assert b"workspace" in L.ff_last_error()


def test_dit_handle_and_config_validation(L):
    cfg = synth.config("tiny_mmdit")
    c = ffi.make_config(cfg)
    h = C.c_void_p()
    assert L.ff_dit_create(C.byref(c), C.c_void_p(256), C.byref(h)) == 0
    n = C.c_size_t()
    assert L.ff_dit_workspace_size(h, 4, C.byref(n)) == 0
    R = 4 * (32 + 64)
    assert n.value >= R * 256 * (4 + 2 + 6 + 2) + R * (256 + 1024) * 2
    # a velocity call with a too-small workspace is rejected on the host
    assert L.ff_dit_velocity(h, 4, 16, 16, 16, 16, 256, 1024, None) == 3
    assert L.ff_dit_velocity(h, 4, 16, 16, 16, 16, 255, n.value, None) == 1
    assert L.ff_dit_destroy(h) == 0
    bad = ffi.make_config(dict(cfg, rope_axes=(8, 28, 30)))
    assert L.ff_dit_create(C.byref(bad), C.c_void_p(256), C.byref(h)) == 1
    bad = ffi.make_config(dict(cfg, head_dim=32, heads=8))
    assert L.ff_dit_create(C.byref(bad), C.c_void_p(256), C.byref(h)) == 2


def test_schedule_window_matches_oracle(L):
    t, s = ffi.ff_sde_schedule(ffi.FF_SCHED_FLOW_SDE, 10, 3.0, 0.7, 0.96)
    tw, sw = ffi.ff_sde_schedule_window(ffi.FF_SCHED_FLOW_SDE, 10, 3.0, 0.7, 0.96, 2, 3)
    assert tw == t
    np.testing.assert_array_equal(sw, osde.window_sigma(s, 2, 3))
    for bad in ((-1, 2), (9, 2), (0, 11)):
        with pytest.raises(ffi.FFError):
            ffi.ff_sde_schedule_window(ffi.FF_SCHED_FLOW_SDE, 10, 3.0, 0.7, 0.96, *bad)


def test_awm_and_multi_reward_host_validation(L):
    assert ffi.ff_awm_loss_workspace_size(4, 262144) == 4 * 65 * 8
    assert ffi.ff_awm_loss_workspace_size(2, 1 << 26) == 2 * 1025 * 8
    # rejected before any CUDA call
    assert L.ff_awm_loss(2, 18, 16, 16, 16, 16, 0, 16, None, None, 16, 1 << 20, None) == 2   # D % 4
    assert L.ff_awm_loss(2, 16, 16, 16, 16, 16, 3, 16, None, None, 16, 1 << 20, None) == 1   # bad reduce
    assert L.ff_awm_loss(2, 16, 16, 16, 16, 16, 0, 16, None, None, 16, 8, None) == 3         # workspace
    assert L.ff_awm_loss(2, 16, None, 16, 16, 16, 0, 16, None, None, 16, 1 << 20, None) == 1
    assert L.ff_forward_process(2, 18, 16, 16, 16, 16, None) == 2
    assert L.ff_forward_process(2, 16, 16, 16, None, 16, None) == 1
    assert L.ff_sample_timesteps(5, 4, 16, 0.0, 1.0, None, 0, 16, None) == 1
    assert L.ff_sample_timesteps(ffi.FF_TSAMPLE_DISCRETE, 4, 16, 0.0, 1.0, None, 0, 16, None) == 1
    assert L.ff_sample_timesteps(ffi.FF_TSAMPLE_LOGIT_NORMAL, 4, 16, 0.0, -1.0, None, 0, 16, None) == 1
    assert L.ff_group_advantage_multi(2, 4, 65, 16, 16, 0, 1e-4, 16, None) == 2
    assert L.ff_group_advantage_multi(2, 4, 2, 16, 16, 7, 1e-4, 16, None) == 1
    assert L.ff_grpo_loss_weighted(4, 2, 16, 16, 16, None, 0.2, 0.2, 16, None, 16, 64, None) == 1


def test_training_pass_host_validation(L):
    small = dict(synth.config("tiny_mmdit"), hidden=256, heads=2, head_dim=128, mlp=512, n_double=1, n_single=1,
                 txt_dim=128, n_txt=16, grid=(1, 4, 8), rope_axes=(16, 56, 56))
    c = ffi.make_config(small)
    h = C.c_void_p()
    assert L.ff_dit_create(C.byref(c), C.c_void_p(256), C.byref(h)) == 0
    n = C.c_size_t()
    assert L.ff_dit_train_workspace_size(h, 2, C.byref(n)) == 0
    H, F, R = 256, 512, 2 * (16 + 32)
    # at least the stored activations of one double- and one single-stream block
    assert n.value >= R * (30 * H + 4 * F) + R * (22 * H + 4 * F)
    # B N_t and B N_i must be multiples of 8 (token counts are the K of the weight gradients)
    odd = ffi.make_config(dict(small, n_txt=5))
    h5 = C.c_void_p()
    assert L.ff_dit_create(C.byref(odd), C.c_void_p(256), C.byref(h5)) == 0
    assert L.ff_dit_train_workspace_size(h5, 2, C.byref(n)) == 2
    assert L.ff_dit_train_workspace_size(h5, 8, C.byref(n)) == 0
    assert L.ff_dit_destroy(h5) == 0
    # rejected on the host: workspace too small, misaligned workspace, null gradient
    assert L.ff_dit_forward_train(h, 2, 16, 16, 16, 16, 256, 1024, None) == 3
    assert L.ff_dit_backward(h, 2, 16, 16, 16, None, 256, 1024, None) == 3
    assert L.ff_dit_backward(h, 2, 16, 16, None, None, 256, 1 << 40, None) == 1
    assert L.ff_dit_backward(h, 2, 16, 16, 16, None, 255, 1 << 40, None) == 1
    assert L.ff_dit_destroy(h) == 0
    # head_dim 64 models and WAN models have a training pass too
    c64 = ffi.make_config(synth.config("tiny_mmdit"))
    assert L.ff_dit_create(C.byref(c64), C.c_void_p(256), C.byref(h)) == 0
    assert L.ff_dit_train_workspace_size(h, 4, C.byref(n)) == 0
    assert L.ff_dit_destroy(h) == 0
    wcfg = dict(synth.config("wan_40"), hidden=256, heads=2, mlp=512, n_double=2, grid=(2, 4, 4),
                rope_axes=(44, 42, 42))
    wan = ffi.make_config(wcfg)
    assert L.ff_dit_create(C.byref(wan), C.c_void_p(256), C.byref(h)) == 0
    assert L.ff_dit_train_workspace_size(h, 4, C.byref(n)) == 0
    # per block: three fp32 residuals, nine bf16 [R_i, H] values, raw and
    # normalised qkv, the MLP's two [R_i, F] values, the text's raw and
    # normalised k | v
    Ri, Rt = 4 * 32, 4 * wcfg["n_txt"]
    assert n.value >= 2 * (Ri * (42 * 256 + 4 * 512) + Rt * 8 * 256)
    assert L.ff_dit_destroy(h) == 0
    # recompute mode 2 keeps only the block inputs: a smaller workspace; mode 1
    # also keeps the second block's self-attention O, its low part and lse
    full = n.value
    wan2 = ffi.make_config(wcfg)
    hr = C.c_void_p()
    assert L.ff_dit_create(C.byref(wan2), C.c_void_p(256), C.byref(hr)) == 0
    assert L.ff_dit_set_train_recompute(hr, 2) == 0
    assert L.ff_dit_train_workspace_size(hr, 4, C.byref(n)) == 0
    only_inputs = n.value
    assert only_inputs < full - Ri * (38 * 256 + 4 * 512)
    assert L.ff_dit_set_train_recompute(hr, 1) == 0
    assert L.ff_dit_train_workspace_size(hr, 4, C.byref(n)) == 0
    assert only_inputs + Ri * 4 * 256 <= n.value < full - Ri * (34 * 256 + 4 * 512)
    assert L.ff_dit_set_train_recompute(hr, 3) == 1
    assert L.ff_dit_set_train_recompute(hr, -1) == 1
    assert L.ff_dit_destroy(hr) == 0
    c64b = ffi.make_config(synth.config("tiny_mmdit"))                 # 2 double blocks
    assert L.ff_dit_create(C.byref(c64b), C.c_void_p(256), C.byref(hr)) == 0
    assert L.ff_dit_train_workspace_size(hr, 4, C.byref(n)) == 0
    stored = n.value
    assert L.ff_dit_set_train_recompute(hr, 1) == 0
    assert L.ff_dit_train_workspace_size(hr, 4, C.byref(n)) == 0
    assert n.value < stored
    assert L.ff_dit_set_train_recompute(None, 1) == 1
    # the backward runs only in the mode of the model's latest training forward
    assert L.ff_dit_destroy(hr) == 0
    assert L.ff_dit_create(C.byref(c64b), C.c_void_p(256), C.byref(hr)) == 0
    assert L.ff_dit_backward(hr, 4, 16, 16, 16, None, 256, 1 << 40, None) == 1       # no forward yet
    assert b"no ff_dit_forward_train" in L.ff_last_error()
    assert L.ff_dit_forward_train(hr, 4, 16, 16, 16, 16, 256, 1024, None) == 3        # workspace too small
    assert L.ff_dit_set_train_recompute(hr, 1) == 0
    assert L.ff_dit_backward(hr, 4, 16, 16, 16, None, 256, 1 << 40, None) == 1       # mode changed since
    assert b"recompute mode changed" in L.ff_last_error()
    assert L.ff_dit_set_train_recompute(hr, 0) == 0
    assert L.ff_dit_backward(hr, 4, 16, 16, 16, None, 256, 1024, None) == 3          # same mode: on to the workspace check
    assert L.ff_dit_destroy(hr) == 0
    wodd = ffi.make_config(dict(wcfg, n_txt=5))      # B N_t = 20: not a multiple of 8
    assert L.ff_dit_create(C.byref(wodd), C.c_void_p(256), C.byref(h)) == 0
    assert L.ff_dit_train_workspace_size(h, 4, C.byref(n)) == 2
    assert L.ff_dit_train_workspace_size(h, 8, C.byref(n)) == 0
    assert L.ff_dit_destroy(h) == 0
    # cross-attention (latent queries, text keys / values): rejected on the host
    assert L.ff_cross_attention_forward(1, 2, 128, 0, 16, 256, 8, 16, 512, 16, 256, None, None) == 1   # nq = 0
    assert L.ff_cross_attention_forward(1, 2, 128, 8, 16, 256, 0, 16, 512, 16, 256, None, None) == 1   # nk = 0
    assert L.ff_cross_attention_forward(1, 2, 128, 8, 16, 256, 8, 16, 512, 16, 256, 8, None) == 1      # lse misaligned
    assert L.ff_cross_attention_backward(1, 2, 128, 8, 16, 256, 16, 16, 256, 16, 256, 8, 16, 512, 16, 256,
                                         16, 16, 1 << 20, None) == 1                                     # lddkv < 2H
    assert L.ff_cross_attention_backward(1, 2, 96, 8, 16, 192, 16, 16, 192, 16, 192, 8, 16, 384, 16, 384,
                                         16, 16, 1 << 20, None) == 2                                     # head_dim 96
    # the counter-based noise and the SDE step that draws it
    assert L.ff_philox_normal(2, 18, 1, 0, 16, None) == 2                  # D % 4
    assert L.ff_philox_normal(2, 16, 1, 0, None, None) == 1                # null out
    assert L.ff_philox_normal(2, 16, 1, 0, 8, None) == 1                   # misaligned
    assert L.ff_sde_step_logprob_philox(2, 18, 16, 16, 16, 16, 16, 16, 1, 0, 0, 16, 1, 16, 1 << 20, None) == 2
    assert L.ff_sde_step_logprob_philox(2, 16, 16, 16, 16, 16, 16, 16, 1, 0, 0, 16, 1, 16, 8, None) == 3
    # the log-prob backward
    assert L.ff_sde_logprob_backward(2, 18, 16, 16, 16, 16, 16, 16, 0, 16, 1, 16, None) == 2   # D % 4
    assert L.ff_sde_logprob_backward(2, 16, 16, 16, 16, 16, 16, 16, 5, 16, 1, 16, None) == 1   # reduce
    assert L.ff_sde_logprob_backward(2, 16, 16, 16, None, 16, 16, 16, 0, 16, 1, 16, None) == 1
    assert L.ff_sde_logprob_backward(2, 16, 16, 16, 16, 16, 16, 16, 0, 16, 0, 16, None) == 1   # ld


def test_reduce_chunks_host_validation(L):
    I2 = C.c_int * 2
    I64 = C.c_int64 * 1
    I1 = C.c_int * 1
    # no jobs: nothing to do, no device needed
    assert L.ff_debug_reduce_chunks(0, 1, None, None, None, None, None, None, None, None, None, None, None) == 0
    assert L.ff_debug_reduce_chunks(-1, 1, None, None, None, None, None, None, None, None, None, None, None) == 1
    args = dict(part_off=I64(0), ld_part=I64(64), ncols=I1(64), first=I2(0, 0), count=I2(4, 0),
                per_sample=I1(1), out_off=I64(0), ld_out=I64(64))

    def call(B=2, part=16, out=16, **over):
        a = dict(args, **over)
        return L.ff_debug_reduce_chunks(1, B, part, out, a["part_off"], a["ld_part"], a["ncols"], a["first"],
                                        a["count"], a["per_sample"], a["out_off"], a["ld_out"], None)
    assert call(part=None) == 1
    assert call(count=I2(0, 0)) == 1          # empty span
    assert call(first=I2(-1, 0)) == 1         # negative first row
    assert call(ld_part=I64(32)) == 1         # pitch below ncols
    assert call(ld_out=I64(32)) == 1          # per-sample output pitch below ncols
    assert call(B=0) == 1                     # per-sample job without samples
    assert call(ncols=I1(0), ld_part=I64(0)) == 1


def test_nft_host_validation(L):
    assert ffi.ff_nft_loss_workspace_size(4, 262144) == 4 * 65 * 2 * 8
    assert L.ff_nft_loss(2, 18, 16, 16, 16, 16, 16, 0.1, 0, 16, None, None, 16, 1 << 20, None) == 2   # D % 4
    assert L.ff_nft_loss(2, 16, 16, 16, 16, 16, 16, 0.1, 3, 16, None, None, 16, 1 << 20, None) == 1   # reduce
    assert L.ff_nft_loss(2, 16, 16, 16, 16, 16, 16, 0.0, 0, 16, None, None, 16, 1 << 20, None) == 1   # beta
    assert L.ff_nft_loss(2, 16, 16, None, 16, 16, 16, 0.1, 0, 16, None, None, 16, 1 << 20, None) == 1
    assert L.ff_nft_loss(2, 16, 16, 16, 16, 16, 16, 0.1, 0, 16, None, None, 16, 8, None) == 3        # workspace
