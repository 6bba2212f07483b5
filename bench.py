#!/usr/bin/env python
"""Throughput of the rollout denoising step on GB300.

Headline workload (default): the WAN-shaped video model -- 40 blocks, H 5120,
40 x 128 heads, MLP 13824, self-attention over 32760 latent tokens (21 x 30
x 52 grid, 3-axis RoPE) plus cross-attention to 512 text tokens, batch 1 per
sample, groups of 8 rolled out one sample at a time.  One step = one
velocity call + one Flow-SDE step with its log-prob (noise drawn in the
kernel) + the group advantage over the 8 rewards + the clipped GRPO loss.

Prints ONE JSON line (rank 0).  Metric: latent tokens x denoise steps / s.
  value   -- inputs resident in HBM, K steps timed with CUDA events
  e2e     -- same metric through the public API with host (pinned) inputs
             copied in and results copied out inside the timed region
  roofline -- dominant kernel by device time: algorithmic work per launch
             divided by its CUDA-event launch duration in the timed region
  cpu_baseline -- the fp64 oracle on a bounded sample of the same workload
  other_workloads -- the Flux-shaped block (batch 4), the Flux-shaped
             rollout model (a full 10-step rollout of batch 32 per step) and
             the Qwen-Image-shaped 60-block model, each timed on its own

--impl reference times the oracle itself (the CPU reference of this path).
Multi-GPU (torchrun): every rank runs its own independent groups; no
collective touches the data path ("weak" scaling).
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "latent tokens x denoise steps/sec at 1 GB300; % bf16 TC peak (DiT), % HBM BW (SDE/loss)"
UNIT = "latent_tokens*steps/s"
WORKLOAD = "wan_40"
PROFILE_DIR = os.path.join(ROOT, "profiles")


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=20)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default=WORKLOAD)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--train-only", action="store_true",
                   help="of the extra measurements, only the training step (on this workload)")
    p.add_argument("--no-sweep", action="store_true",
                   help="skip the extra measurements (other workloads, training, sweeps)")
    p.add_argument("--profile-kernel", default=None,
                   choices=["sde_step", "sde_step_philox", "grpo_loss", "group_advantage", "ln_modulate",
                            "attention", "attention_backward", "velocity"],
                   help="launch only this kernel (a few times, no timing) for an ncu capture")
    p.add_argument("--elements", type=int, default=1 << 24, help="problem size of --profile-kernel's HBM kernels")
    return p.parse_args()


def workload_desc(cfg, rollout=False):
    f, h, w = cfg["grid"]
    if cfg.get("arch") == "wan":
        blocks = f"{cfg['n_double']} WAN blocks (self-attention + text cross-attention + FFN)"
        grid = f"{f}x{h}x{w} grid of 1x2x2 patches, 64-dim, 3-axis RoPE"
    else:
        blocks = f"{cfg['n_double']} double + {cfg['n_single']} single MMDiT blocks"
        grid = f"{h}x{w} grid of 2x2 patches, 64-dim"
    if rollout:
        per = (f"per step: a {cfg['steps_run']}-step SDE rollout of the whole batch (velocity + SDE step with "
               f"in-kernel noise + log-prob each step, every log-prob kept) + group advantage + clipped GRPO loss "
               f"over [batch, steps]")
    else:
        per = ("per step: 1 velocity call + 1 SDE step with log-prob + group advantage + clipped GRPO loss")
    return (f"{cfg['name']}: {blocks}, H {cfg['hidden']}, {cfg['heads']}x{cfg['head_dim']} heads, MLP {cfg['mlp']}, "
            f"{cfg['n_txt']} text + {f * h * w} latent tokens ({grid}), batch {cfg['batch']} (groups of "
            f"{cfg['group']}); {per}")


def device_blob(ffi, cfg, dev, seed=0):
    """Random-init weights drawn on the device (the large workloads hold up to
    about 20e9 parameters, too many to draw on the host): N(0, 0.02)
    matrices, zero biases, unit norm scales, as bf16."""
    import numpy as np
    import torch
    import synth
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


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(p) as f:
            d = json.load(f)
        return d["hbm_gbs"], d["bf16_tflops"], d.get("bf16_tflops_sustained"), "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


KERNEL_SOURCES = {"gemm_bf16": ["gemm.cu"], "attention": ["attention.cu"], "sde_step": ["sde.cu"]}


def profile_traffic(kernel, workload):
    """DRAM bytes per launch recorded from an ncu capture, if the kernel's
    source has not changed since (source hash recorded with the number)."""
    path = os.path.join(PROFILE_DIR, f"{kernel}_{workload}.md")
    try:
        txt = open(path).read()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", txt)
    h = re.search(r"source_sha256:\s*([0-9a-f]+)", txt)
    if not m or not h or kernel not in KERNEL_SOURCES:
        return None
    if h.group(1) != kernel_source_hash(kernel):
        return None
    return float(m.group(1))


def kernel_source_hash(kernel):
    """Hash of the files that define a kernel (its .cu plus the shared headers)."""
    d = os.path.join(ROOT, "paper_2602_12529_gb300", "csrc")
    sha = hashlib.sha256()
    for f in KERNEL_SOURCES[kernel] + ["ptx.cuh", "internal.h"]:
        with open(os.path.join(d, f), "rb") as fh:
            sha.update(f.encode() + fh.read())
    return sha.hexdigest()[:16]


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled every 100 ms."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
        try:
            self.p = subprocess.Popen(["nvidia-smi", "-i", str(gpu_index), f"--query-gpu={self.Q}",
                                       "--format=csv,noheader,nounits", "-lms", "100"], stdout=self.f,
                                      stderr=subprocess.DEVNULL)
        except OSError:
            self.p = None

    def stop(self):
        if self.p is not None:
            self.p.terminate()
            try:
                self.p.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.p.kill()
        self.f.flush()
        self.f.seek(0)
        rows = [l.strip().split(", ") for l in self.f.read().splitlines() if l.strip()]
        os.unlink(self.f.name)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            try:
                sm.append(float(r[1]))
                mx.append(float(r[2]))
            except (ValueError, IndexError):
                continue
            for n, v in zip(names, r[5:9]):
                if v.strip().lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# ---------------------------------------------------------------------------
# the oracle on a bounded sample (CPU baseline and the reference arm)
# ---------------------------------------------------------------------------

def velocity_flops(cfg, B=1):
    """Algorithmic FLOPs of one velocity call: 2 M N K per Linear, 4 N_q N_k d
    per head of attention (the accounting of the measurement section)."""
    H, F, P, L = cfg["hidden"], cfg["mlp"], cfg["patch_dim"], cfg["n_double"]
    Nt, Ni = cfg["n_txt"], synth_n_img(cfg)
    tf = cfg["time_freq_dim"]
    if cfg.get("arch") == "wan":
        per_block = 2.0 * Ni * (6 * H * H + 2 * H * F) + 2.0 * Nt * 2 * H * H \
            + 4.0 * H * Ni * Ni + 4.0 * H * Ni * Nt
        fixed = 2.0 * Ni * P * H * 2 + 2.0 * Nt * (cfg["txt_dim"] * H + H * H) + 2.0 * (tf * H + H * H + 6 * H * H)
        return B * (L * per_block + fixed)
    N = Nt + Ni
    Ls = cfg["n_single"]
    per_block = 2.0 * N * (4 * H * H + 2 * H * F) + 4.0 * H * N * N
    mod_w = L * 12 * H + Ls * 3 * H + 2 * H
    fixed = 2.0 * Ni * P * H * 2 + 2.0 * Nt * cfg["txt_dim"] * H + 2.0 * (tf * H + H * H + mod_w * H)
    return B * ((L + Ls) * per_block + fixed)


def oracle_sample(cfg):
    """(sample config, exact, description) of the oracle's bounded sample of a
    workload: the whole call for one sample where that takes seconds, else
    one block (one of each kind) of the same width, and for the video model a
    3 x 16 x 16 latent grid; the rate is then scaled to the whole call by
    the ratio of algorithmic FLOPs (an estimate)."""
    if cfg.get("arch") == "wan":
        s = dict(cfg, n_double=1, grid=(3, 16, 16), batch=1)
        return s, False, (f"1 of {cfg['n_double']} blocks on a 3x16x16 latent grid (768 of {synth_n_img(cfg)} "
                          f"tokens), 1 sample")
    if cfg["n_double"] + cfg["n_single"] <= 2 and synth_n_img(cfg) * cfg["hidden"] <= 4096 * 3072:
        return dict(cfg, batch=1), True, f"1 of {cfg['batch']} samples, whole velocity call"
    s = dict(cfg, n_double=min(cfg["n_double"], 1), n_single=min(cfg["n_single"], 1), batch=1)
    return s, False, (f"{s['n_double']} double + {s['n_single']} single of the {cfg['n_double']} + "
                      f"{cfg['n_single']} blocks at full width and sequence length, 1 sample")


class OracleStep:
    """fp64 oracle of one rollout step (velocity + SDE step + log-prob +
    advantage + loss) for one sample of a (sample) configuration."""

    def __init__(self, cfg):
        import numpy as np

        import synth
        from oracle import dit as odit
        self.np, self.odit, self.cfg = np, odit, cfg
        wan = cfg.get("arch") == "wan"
        self.vel = odit.wan_velocity if wan else odit.velocity
        specs = odit.wan_param_specs(cfg) if wan else odit.param_specs(cfg)
        self.P = odit.widen_params(synth.weights(specs, seed=0))
        self.x = synth.initial_latent(cfg, batch=1)
        self.txt = odit.widen(synth.text_embeds(cfg, batch=1))
        self.eps = synth.step_noise(cfg, 0, batch=1)
        self.rewards = synth.rewards(cfg["group"])

    def __call__(self):
        from oracle import grpo as ogrpo
        from oracle import sde as osde
        np, cfg = self.np, self.cfg
        grid = osde.time_grid(cfg["sde_steps"], cfg["shift"])
        t, tn = grid[0:1], grid[1:2]
        sg = osde.sigma_flow_sde(t, cfg["eta"], cfg["t_clamp"])
        v = self.vel(self.P, cfg, self.x, self.txt, t)
        xn, lp = osde.sde_step_logprob(self.x, v, t, tn, sg, eps=self.eps)
        adv = ogrpo.group_advantage(self.rewards, cfg["group"], cfg["eps_adv"])
        lpn = np.full((cfg["group"], 1), lp[0])
        ogrpo.grpo_loss(lpn, lpn + 0.01, adv, cfg["clip"], cfg["clip"])


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def oracle_scale(cfg, scfg):
    """Seconds of the whole call per second of the sample (FLOP ratio)."""
    return velocity_flops(cfg) / velocity_flops(scfg)


def oracle_rate(cfg):
    """(rate in latent-token-steps/s, seconds of the sample, description)."""
    scfg, exact, what = oracle_sample(cfg)
    step = OracleStep(scfg)
    t0 = time.perf_counter()
    step()
    dt = time.perf_counter() - t0
    scale = 1.0 if exact else oracle_scale(cfg, scfg)
    rate = synth_n_img(cfg) / (dt * scale)
    desc = (f"{what} + SDE step + log-prob + advantage + loss, fp64 numpy, {dt:.1f} s"
            + ("" if exact else f"; whole-call time estimated as {scale:.1f} x the sample's (algorithmic FLOP "
                                f"ratio)"))
    return rate, dt, desc


def run_reference(args):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import synth
    cfg = synth.config(args.workload)
    n_img = synth.n_img(cfg)
    scfg, exact, what = oracle_sample(cfg)
    scale = 1.0 if exact else oracle_scale(cfg, scfg)
    step = OracleStep(scfg)
    for _ in range(args.warmup):
        step()
    times = []
    for _ in range(args.steps):
        t0 = time.perf_counter()
        step()
        times.append(time.perf_counter() - t0)
    dt = sum(times) / len(times) * scale
    value = n_img / dt
    sample = (f"{what} + SDE step + log-prob + advantage + loss, fp64 numpy, {dt / scale:.2f} s per step"
              + ("" if exact else f"; whole-call time estimated as {scale:.1f} x the sample's (algorithmic FLOP "
                                  f"ratio)"))
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": workload_desc(cfg), "batch": cfg["batch"], "n_txt": cfg["n_txt"],
                       "n_img": n_img},
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "gpu_launches": 0}
    print(json.dumps(line), flush=True)
    return 0


# ---------------------------------------------------------------------------
# the CUDA path
# ---------------------------------------------------------------------------

def graph_time_us(dev, fns, reps):
    """Per-call microseconds of fns[0..] called round-robin `reps` times,
    captured in one CUDA graph (no host dispatch in the timed region) and
    replayed three times (median replay)."""
    import torch
    for f in fns[:2]:
        f()
    side = torch.cuda.Stream(dev)
    side.wait_stream(torch.cuda.current_stream(dev))
    with torch.cuda.stream(side):
        for f in fns[:2]:
            f()
    torch.cuda.current_stream(dev).wait_stream(side)
    torch.cuda.synchronize(dev)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        for i in range(reps):
            fns[i % len(fns)]()
    g.replay()
    torch.cuda.synchronize(dev)
    ts = []
    for _ in range(3):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record()
        g.replay()
        e1.record()
        torch.cuda.synchronize(dev)
        ts.append(e0.elapsed_time(e1))
    del g
    return sorted(ts)[1] * 1e3 / reps


def at_config_small_kernels(ffi, dev, hbm_peak, cfg, rank, reps=100):
    """Per-launch time of the memory-bound kernels at the workload's own sizes
    (inputs L2-resident): `reps` back-to-back calls captured in one CUDA
    graph.  These are launch- and L2-bound; the HBM sweep gives bandwidth."""
    import torch
    si = StepInputs(ffi, cfg, dev, rank)
    B, G = si.B, si.G
    D = si.x.numel() // B
    v = torch.randn_like(si.x)
    eps = torch.randn_like(si.x)
    x_next = torch.empty_like(si.x)
    logp = torch.empty((B, 1), dtype=torch.float32, device=dev)
    lp_old = logp + 0.01
    adv_all = torch.empty(si.n_r, dtype=torch.float32, device=dev)
    loss = torch.zeros(1, dtype=torch.float32, device=dev)
    grad = torch.empty((B, 1), dtype=torch.float32, device=dev)
    ws_sde = torch.zeros(ffi.ff_sde_workspace_size(B, D), dtype=torch.uint8, device=dev)
    ws_loss = torch.zeros(ffi.ff_grpo_loss_workspace_size(B, 1), dtype=torch.uint8, device=dev)
    cases = {
        "sde_step (SAMPLE, eps drawn in the kernel, log-prob)": (
            lambda: ffi.ff_sde_step_logprob_philox(si.x, v, x_next, si.t, si.tn, si.sg, logp, 7, 0, ws=ws_sde),
            12.0 * si.x.numel()),
        "sde_step (SAMPLE, eps read from memory, log-prob)": (
            lambda: ffi.ff_sde_step_logprob(si.x, v, eps, x_next, si.t, si.tn, si.sg, logp, ws=ws_sde),
            16.0 * si.x.numel()),
        "group_advantage": (lambda: ffi.ff_group_advantage(si.r, G, cfg["eps_adv"], adv_all), 8.0 * si.n_r),
        "grpo_loss (+ dL/dlp)": (lambda: ffi.ff_grpo_loss(logp, lp_old, adv_all[:B], cfg["clip"], cfg["clip"], loss,
                                                          grad, ws=ws_loss), 16.0 * logp.numel() + 4.0 * B),
    }
    out = {}
    for name, (fn, nbytes) in cases.items():
        us = graph_time_us(dev, [fn], reps)
        out[name] = {"us_per_call": us, "bytes": nbytes, "gbs": nbytes / us / 1e3,
                     "frac_of_hbm": nbytes / us / 1e3 / hbm_peak, "calls_per_graph": reps}
    return out


def hbm_sweep(ffi, dev, hbm_peak, l2_bytes=129 * 2 ** 20):
    """Bandwidth of the memory-bound kernels at sizes well beyond L2, with
    enough rotating buffer sets that every launch reads from HBM; each point
    is a CUDA graph of back-to-back calls over the sets (no host dispatch
    inside the timed region)."""
    import torch

    def timeit(fns, reps=12):
        return graph_time_us(dev, fns, reps) / 1e6

    def nsets(nbytes):
        return max(2, -(-4 * l2_bytes // nbytes))

    def row(n, per, sets, sec, **kw):
        return dict({"elements": n, "bytes": per, "gbs": per / sec / 1e9, "frac": per / sec / 1e9 / hbm_peak,
                     "sets": sets}, **kw)

    out = {}
    B = 4
    t = torch.full((B,), 0.75, device=dev)
    tn = torch.full((B,), 0.5, device=dev)
    sg = torch.full((B,), 0.7, device=dev)
    lp = torch.empty(B, device=dev)
    rows = []
    for n in (1 << 24, 1 << 26, 1 << 28):
        D = n // B
        per = 16 * n
        sets = []
        for _ in range(nsets(per)):
            x = torch.randn(B, D, device=dev)
            sets.append((x, torch.randn_like(x), torch.randn_like(x), torch.empty_like(x)))
        ws = torch.zeros(ffi.ff_sde_workspace_size(B, D), dtype=torch.uint8, device=dev)
        fns = [lambda s_=s_: ffi.ff_sde_step_logprob(s_[0], s_[1], s_[2], s_[3], t, tn, sg, lp, ws=ws) for s_ in sets]
        rows.append(row(n, per, len(sets), timeit(fns)))
        del sets
    out["sde_step"] = rows
    rows = []
    for n in (1 << 24, 1 << 26, 1 << 28):
        D = n // B
        per = 12 * n
        sets = []
        for _ in range(nsets(per)):
            x = torch.randn(B, D, device=dev)
            sets.append((x, torch.randn_like(x), torch.empty_like(x)))
        ws = torch.zeros(ffi.ff_sde_workspace_size(B, D), dtype=torch.uint8, device=dev)
        fns = [lambda s_=s_: ffi.ff_sde_step_logprob_philox(s_[0], s_[1], s_[2], t, tn, sg, lp, 7, 0, ws=ws)
               for s_ in sets]
        rows.append(row(n, per, len(sets), timeit(fns)))
        del sets
    out["sde_step_device_noise"] = rows
    rows = []
    for n in (1 << 22, 1 << 24, 1 << 26):
        Bq, T = n // 16, 16
        per = 12 * n + 4 * Bq
        sets = []
        for _ in range(nsets(per)):
            a = torch.randn(Bq, T, device=dev)
            sets.append((a, a + 0.01 * torch.randn_like(a), torch.randn(Bq, device=dev), torch.empty_like(a)))
        loss = torch.empty(1, device=dev)
        ws = torch.zeros(ffi.ff_grpo_loss_workspace_size(Bq, T), dtype=torch.uint8, device=dev)
        fns = [lambda s_=s_: ffi.ff_grpo_loss(s_[0], s_[1], s_[2], 0.2, 0.2, loss, s_[3], ws=ws) for s_ in sets]
        rows.append(row(n, per, len(sets), timeit(fns)))
        del sets
    out["grpo_loss"] = rows
    rows = []
    for n in (1 << 22, 1 << 24, 1 << 26):
        per = 8 * n
        sets = [(torch.rand(n, device=dev), torch.empty(n, device=dev)) for _ in range(nsets(per))]
        fns = [lambda s_=s_: ffi.ff_group_advantage(s_[0], 16, 1e-4, s_[1]) for s_ in sets]
        rows.append(row(n, per, len(sets), timeit(fns), group=16))
        del sets
    out["group_advantage"] = rows
    for name, per_elem in (("forward_process", 12), ("awm_loss", 16)):
        rows = []
        for n in (1 << 24, 1 << 26, 1 << 28):
            D = n // B
            per = per_elem * n
            sets = []
            for _ in range(nsets(per)):
                x = torch.randn(B, D, device=dev)
                sets.append((x, torch.randn_like(x), torch.randn_like(x), torch.empty_like(x)))
            tt = torch.full((B,), 0.6, device=dev)
            adv = torch.randn(B, device=dev)
            loss = torch.empty(1, device=dev)
            if name == "forward_process":
                fns = [lambda s_=s_: ffi.ff_forward_process(s_[0], s_[1], tt, s_[3]) for s_ in sets]
            else:
                ws = torch.empty(ffi.ff_awm_loss_workspace_size(B, D), dtype=torch.uint8, device=dev)
                fns = [lambda s_=s_: ffi.ff_awm_loss(s_[0], s_[1], s_[2], adv, ffi.FF_AWM_MEAN, loss, s_[3], ws=ws)
                       for s_ in sets]
            rows.append(row(n, per, len(sets), timeit(fns)))
            del sets
        out[name] = rows
    rows = []
    for n in (1 << 24, 1 << 26, 1 << 28):
        D = n // B
        per = 20 * n
        sets = []
        for _ in range(nsets(per)):
            x = torch.randn(B, D, device=dev)
            sets.append((x, torch.randn_like(x), torch.randn_like(x), torch.randn_like(x), torch.empty_like(x)))
        r = torch.rand(B, device=dev)
        loss = torch.empty(1, device=dev)
        ws = torch.empty(ffi.ff_nft_loss_workspace_size(B, D), dtype=torch.uint8, device=dev)
        fns = [lambda s_=s_: ffi.ff_nft_loss(s_[0], s_[1], s_[2], s_[3], r, 0.1, ffi.FF_AWM_MEAN, loss, s_[4], ws=ws)
               for s_ in sets]
        rows.append(row(n, per, len(sets), timeit(fns)))
        del sets
    out["nft_loss"] = rows
    torch.cuda.empty_cache()
    return out


def awm_step(args, ffi, model, cfg, dev, x0, txt, eps, rewards, timed, world):
    """The AWM training step of Eq. 3 on the same workload and batch: training
    times from the logit-normal sampler, x_t by the forward process, the
    velocity, and the advantage-weighted loss with its gradient w.r.t. v.
    Timed like the main step (CUDA events, K steps), and once more with the
    per-launch events for the two memory-bound kernels' rooflines."""
    import torch
    B = x0.shape[0]
    D = x0.numel() // B
    z = torch.linspace(-1.5, 1.5, B, device=dev)
    tt = torch.empty(B, device=dev)
    xt = torch.empty_like(x0)
    v = torch.empty_like(x0)
    gv = torch.empty_like(x0)
    adv_all = torch.empty(rewards.numel(), device=dev)
    ffi.ff_group_advantage(rewards, rewards.numel(), 1e-4, adv_all)
    adv = adv_all[:B]
    loss = torch.empty(1, device=dev)
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=dev)
    ws_awm = torch.empty(ffi.ff_awm_loss_workspace_size(B, D), dtype=torch.uint8, device=dev)

    def step():
        ffi.ff_sample_timesteps(ffi.FF_TSAMPLE_LOGIT_NORMAL, z, 0.0, 1.0, tt)
        ffi.ff_forward_process(x0, eps, tt, xt)
        model.ff_dit_velocity(xt, txt, tt, v, ws)
        ffi.ff_awm_loss(v, eps, x0, adv, ffi.FF_AWM_MEAN, loss, gv, ws=ws_awm)

    for _ in range(args.warmup):
        step()
    ms = timed(step, args.steps) / args.steps
    ffi.ff_prof_enable((16 * (cfg["n_double"] + cfg["n_single"]) + 64) * args.steps + 64)
    timed(step, args.steps)
    recs = ffi.ff_prof_records()
    ffi.ff_prof_disable()
    _, _, _, peak_src = load_peaks()
    hbm = load_peaks()[0]
    roofs = {}
    for name in ("forward_process", "awm_loss"):
        r = [(ms_, by) for n_, ms_, fl, by in recs if n_ == name]
        if r:
            ach = sum(b for _, b in r) / len(r) / (sum(m for m, _ in r) / len(r) / 1e3) / 1e9
            roofs[name] = {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm,
                           "launches": len(r), "algorithmic_per_launch": r[0][1], "peak_source": f"{peak_src} HBM copy"}
    n_img = synth_n_img(cfg)
    return {"ms_per_step": ms, "value": world * B * n_img / (ms / 1e3), "unit": UNIT,
            "what": "logit-normal t + forward process + velocity + Eq. 3 loss with dL/dv, batch of the main step",
            "rooflines": roofs}


def backward_kernels(args, ffi, cfg, dev):
    """The training-backward building blocks at the workload's shapes (one
    block's attention over the joint sequence, the QKV Linear's three
    products), CUDA-event timed; algorithmic FLOPs: attention backward
    10 B h N^2 d (recomputed S, dP, dV, dK, dQ), each GEMM 2 M N K."""
    import numpy as np
    import torch
    B, heads, d = cfg["batch"], cfg["heads"], cfg["head_dim"]
    if d != 128 or cfg.get("arch") == "wan":
        return None
    n0, n1 = cfg["n_txt"], synth_n_img(cfg)
    H = heads * d
    g = torch.Generator(device=dev)
    g.manual_seed(5)
    rnd = lambda *shape: torch.randn(*shape, generator=g, device=dev).to(torch.bfloat16)
    q0, q1 = rnd(B * n0, 3 * H), rnd(B * n1, 3 * H)
    o0, o1 = torch.empty(B * n0, H, device=dev, dtype=torch.bfloat16), torch.empty(B * n1, H, device=dev,
                                                                                   dtype=torch.bfloat16)
    g0, g1 = rnd(B * n0, H), rnd(B * n1, H)
    dq0, dq1 = torch.empty_like(q0), torch.empty_like(q1)
    lse = torch.empty(B * heads * ffi.lib().ff_attention_lse_rows(n0, n1), device=dev)
    aws = torch.empty(ffi.ff_attention_forward_workspace_size(d), dtype=torch.uint8, device=dev)
    ffi.ff_attention_forward(B, heads, d, q0, o0, n0, q1, o1, n1, lse=lse, ws=aws)
    T = B * (n0 + n1)
    x, W, dy = rnd(T, H), rnd(3 * H, H), rnd(T, 3 * H)
    y = torch.empty(T, 3 * H, device=dev, dtype=torch.bfloat16)
    dx = torch.empty(T, H, device=dev, dtype=torch.bfloat16)
    dW = torch.empty(3 * H, H, device=dev, dtype=torch.float32)
    N = n0 + n1
    cases = {
        "attention_forward_lse": (lambda: ffi.ff_attention_forward(B, heads, d, q0, o0, n0, q1, o1, n1, lse=lse,
                                                                   ws=aws),
                                  4.0 * B * heads * N * N * d),
        "attention_backward": (lambda: ffi.ff_attention_backward(B, heads, d, (n0, q0, o0, g0, dq0),
                                                                 (n1, q1, o1, g1, dq1), lse),
                               10.0 * B * heads * N * N * d),
        "qkv_forward": (lambda: ffi.ff_gemm(x, ffi.FF_A_MK, W, ffi.FF_B_NK, y), 2.0 * T * 3 * H * H),
        "qkv_input_grad": (lambda: ffi.ff_gemm(dy, ffi.FF_A_MK, W, ffi.FF_B_KN, dx), 2.0 * T * 3 * H * H),
        "qkv_weight_grad": (lambda: ffi.ff_gemm(dy, ffi.FF_A_KM, x, ffi.FF_B_KN, dW), 2.0 * T * 3 * H * H),
    }
    _, tc_burst, _, src = load_peaks()
    out = {}
    for name, (f, fl) in cases.items():
        for _ in range(max(3, args.warmup)):
            f()
        torch.cuda.synchronize(dev)
        ts = []
        for _ in range(max(3, args.steps)):
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            f()
            e1.record()
            torch.cuda.synchronize(dev)
            ts.append(e0.elapsed_time(e1))
        ms = float(np.median(ts))
        out[name] = {"ms": ms, "tflops": fl / ms / 1e9, "frac": fl / ms / 1e9 / tc_burst}
    out["peak"] = f"{tc_burst} TFLOP/s ({src} bf16 dense burst)"
    return out


def train_step(args, ffi, model, cfg, dev, x, txt, t, tn, sg, x_next, lp_old, adv, fwd_flops, timed, world):
    """One Flow-GRPO training step on the batch of the main step: re-score
    the rollout's x_next under the current velocity (training forward, SDE
    log-prob in EVAL mode), the clipped loss with dL/dlp, then dL/dv through
    the log-prob backward and dL/dtheta for every weight through the DiT
    backward.  Algorithmic FLOPs: the forward's (GEMM 2 M N K, attention
    4 B h N^2 d), plus twice the GEMM FLOPs (input and weight gradients) and
    10 B h N^2 d per attention backward (recomputed S, dP, dV, dK, dQ)."""
    import torch
    B = x.shape[0]
    D = x.numel() // B
    need = model.train_workspace_size(B)
    _, total = ffi.ff_dit_weight_layout(cfg)
    free, _ = torch.cuda.mem_get_info(dev)
    recompute = 0
    if need + 4 * total > 0.9 * free:
        # keep the block inputs (mode 1: and the attention outputs) and re-run
        # each block in the backward
        for recompute in (1, 2):
            model.set_train_recompute(recompute)
            need = model.train_workspace_size(B)
            if need + 4 * total <= 0.9 * free:
                break
        else:
            model.set_train_recompute(False)
            return {"skipped": f"training workspace {need / 1e9:.1f} GB (recompute mode 2) + fp32 gradients "
                               f"{4 * total / 1e9:.1f} GB exceed the free device memory ({free / 1e9:.1f} GB)"}
    ws_t = torch.empty(need, dtype=torch.uint8, device=dev)
    grad = torch.empty(total, dtype=torch.float32, device=dev)
    v = torch.empty_like(x)
    dv = torch.empty_like(x)
    lp = torch.empty((B, 1), dtype=torch.float32, device=dev)
    glp = torch.empty((B, 1), dtype=torch.float32, device=dev)
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    ws_sde = torch.zeros(ffi.ff_sde_workspace_size(B, D), dtype=torch.uint8, device=dev)
    ws_loss = torch.zeros(ffi.ff_grpo_loss_workspace_size(B, 1), dtype=torch.uint8, device=dev)

    def step():
        model.ff_dit_forward_train(x, txt, t, v, ws_t)
        ffi.ff_sde_step_logprob(x, v, None, x_next, t, tn, sg, lp, mode=ffi.FF_SDE_EVAL, ws=ws_sde)
        ffi.ff_grpo_loss(lp, lp_old, adv, cfg["clip"], cfg["clip"], loss, glp, ws=ws_loss)
        ffi.ff_sde_logprob_backward(x, v, x_next, t, tn, sg, glp, dv)
        model.ff_dit_backward(txt, dv, grad, ws_t)

    for _ in range(args.warmup):
        step()
    ms = timed(step, args.steps) / args.steps
    # recompute mode runs each block forward twice before its backward: room for every launch
    ffi.ff_prof_enable((200 * (cfg["n_double"] + cfg["n_single"]) + 256) * args.steps + 64)
    timed(step, args.steps)
    recs = ffi.ff_prof_records()
    ffi.ff_prof_disable()
    if recompute:
        model.set_train_recompute(False)
    kern = {}
    for name, ms_, fl, by in recs:
        k = kern.setdefault(name, [0, 0.0])
        k[0] += 1
        k[1] += ms_
    tot = sum(k[1] for k in kern.values())
    Ni = synth_n_img(cfg)
    L = cfg["n_double"] + cfg["n_single"]
    if cfg.get("arch") == "wan":   # self-attention over the latents + cross-attention to the text
        attn_fwd = 4.0 * B * cfg["hidden"] * Ni * (Ni + cfg["n_txt"]) * L
    else:                          # joint attention over text + latents
        N = cfg["n_txt"] + Ni
        attn_fwd = 4.0 * B * cfg["heads"] * N * N * cfg["head_dim"] * L
    gemm_fwd = fwd_flops - attn_fwd
    flops = 3.0 * gemm_fwd + attn_fwd + 2.5 * attn_fwd
    _, tc_burst, tc_sust, src = load_peaks()
    return {"ms_per_step": ms, "value": world * B * synth_n_img(cfg) / (ms / 1e3), "unit": UNIT,
            "what": "training forward (activations kept) + SDE EVAL log-prob + clipped loss and dL/dlp + "
                    "log-prob backward + DiT backward to every weight (fp32 gradients), batch of the main step",
            "tflops": flops / (ms / 1e3) / 1e12, "frac": flops / (ms / 1e3) / 1e12 / tc_burst,
            "frac_vs_sustained": flops / (ms / 1e3) / 1e12 / tc_sust if tc_sust else None,
            "algorithmic_flops": flops, "workspace_gb": need / 1e9, "recompute": recompute,
            "gpu_launches": len(recs) // args.steps,
            "kernels": {k: {"launches": v_[0] // args.steps, "ms_per_step": v_[1] / args.steps, "share": v_[1] / tot}
                        for k, v_ in sorted(kern.items(), key=lambda kv: -kv[1][1])},
            "peak": f"{tc_burst} TFLOP/s ({src} bf16 dense burst)"}


def synth_n_img(cfg):
    import synth
    return synth.n_img(cfg)


# ---- multi-rank host logic (one process per GPU; weak scaling) ----------
# The path shards by whole groups: every rank rolls out its own B samples
# (B / G prompts) with its own seeds, so no collective touches the data path.
# Timing is the slowest rank's, and the reported value counts every rank's
# units.

def rank_seed(rank: int) -> int:
    """Seed offset of a rank's inputs (distinct prompts, noise and rewards)."""
    return 1000 * rank


def max_over_ranks(ms: float, world: int, device=None) -> float:
    """Slowest rank's elapsed time (all-reduce MAX); the identity at N = 1."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    m = torch.tensor([ms], device=device)
    dist.all_reduce(m, op=dist.ReduceOp.MAX)
    return float(m.item())


def whole_job_rate(world: int, units_per_rank_step: float, ms_step: float) -> float:
    """Units all ranks processed per second, at the slowest rank's step time."""
    return world * units_per_rank_step / (ms_step / 1e3)


def make_model(ffi, cfg, dev):
    """(handle, weight blob, parameter count) of a random-init model."""
    import synth
    from paper_2602_12529_gb300 import weights
    _, n_params = ffi.ff_dit_weight_layout(cfg)
    if n_params > 2e9:
        blob = device_blob(ffi, cfg, dev)
    else:
        blob = weights.pack(cfg, lambda n, s: synth.weight(n, s, synth.weight_kind(n), 0), dev)
    return ffi.Dit(cfg, blob), blob, n_params


def kernel_table(ffi, step, steps, timed, cfg):
    """Per-kernel CUDA-event durations of `steps` calls of step():
    {name: [launches, ms, flops, bytes]} and the launch count."""
    per_step = 16 * (cfg["n_double"] + cfg["n_single"]) * max(1, cfg.get("steps_run", 1)) + 64
    ffi.ff_prof_enable(per_step * steps + 64)
    timed(step, steps)
    recs = ffi.ff_prof_records()
    ffi.ff_prof_disable()
    kern = {}
    for name, ms, fl, by in recs:
        k = kern.setdefault(name, [0, 0.0, 0.0, 0.0])
        k[0] += 1
        k[1] += ms
        k[2] += fl
        k[3] += by
    return kern, len(recs)


# A kernel timed inside a run at least this long (device time of the timed
# launches) runs under the power cap: its tensor roofline takes the sustained
# peak, a shorter run's the burst peak.
SUSTAINED_RUN_MS = 500.0


def roofline_of(kern, name, workload):
    """Roofline object of one kernel from its per-launch algorithmic work and
    CUDA-event durations (tensor-bound if it counts FLOPs, else HBM)."""
    n, ms, fl, by = kern[name]
    total = sum(k[1] for k in kern.values())
    hbm, tc_burst, tc_sust, peak_src = load_peaks()
    if fl > 0:
        ach = fl / n / (ms / n / 1e3) / 1e12
        sustained = tc_sust is not None and total >= SUSTAINED_RUN_MS
        peak = tc_sust if sustained else tc_burst
        return {"bound": "tensor", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                "frac": ach / peak, "frac_vs_burst": ach / tc_burst,
                "frac_vs_sustained": ach / tc_sust if tc_sust else None,
                "traffic": profile_traffic(name, workload), "kernel": name, "launches": n,
                "share_of_device_time": ms / total, "algorithmic_per_launch": fl / n,
                "peak_source": (f"{peak_src} bf16 dense, sustained (timed inside {total / 1e3:.1f} s of "
                                f"device time under the power cap)") if sustained
                               else f"{peak_src} bf16 dense (burst)"}
    ach = by / n / (ms / n / 1e3) / 1e9
    return {"bound": "hbm", "achieved": ach, "peak": hbm, "unit": "GB/s", "frac": ach / hbm,
            "traffic": profile_traffic(name, workload), "kernel": name, "launches": n,
            "share_of_device_time": ms / total, "algorithmic_per_launch": by / n,
            "peak_source": f"{peak_src} HBM copy"}


def breakdown_of(kern, steps):
    total = sum(k[1] for k in kern.values())
    return {k: {"launches": v[0] // steps, "ms_per_step": v[1] / steps, "share": v[1] / total}
            for k, v in sorted(kern.items(), key=lambda kv: -kv[1][1])}


class StepInputs:
    """Device inputs of one rollout step of a workload (seeded, synthetic) and
    the host copies they came from."""

    def __init__(self, ffi, cfg, dev, rank):
        import numpy as np
        import torch

        import synth
        B, G = cfg["batch"], cfg["group"]
        self.B, self.G = B, G
        tgrid, sig = ffi.ff_sde_schedule(ffi.FF_SCHED_FLOW_SDE, cfg["sde_steps"], cfg["shift"], cfg["eta"],
                                         cfg["t_clamp"])
        self.tgrid, self.sig = tgrid, sig
        seed = rank_seed(rank)
        self.noise_seed = 100 + seed
        self.h = {
            "x": synth.initial_latent(cfg, seed=2 + seed),
            "txt": synth.text_embeds(cfg, seed=1 + seed).view(np.int16),
            "t": np.full(B, tgrid[0], np.float32),
            "tn": np.full(B, tgrid[1], np.float32),
            "sg": np.full(B, sig[0], np.float32),
        }
        # rewards of whole groups (a WAN group of 8 is rolled out one sample
        # at a time, so it can be larger than the batch)
        self.n_r = -(-B // G) * G
        self.h["r"] = synth.rewards(self.n_r, seed=7 + seed)
        self.h_jitter = synth.logprob_jitter((B, 1), seed=9 + seed)

        def dev_t(a):
            return torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        self.x, self.t, self.tn, self.sg, self.r = (dev_t(self.h[k]) for k in ("x", "t", "tn", "sg", "r"))
        self.txt = dev_t(self.h["txt"]).view(torch.bfloat16)
        self.jitter = dev_t(self.h_jitter)


def measure_step_workload(args, ffi, cfg, dev, rank, world, timed, steps, warmup, keep_model=False):
    """One rollout step of `cfg` (velocity + SDE step with in-kernel noise and
    its log-prob + group advantage + clipped GRPO loss with dL/dlp): time per
    step, kernel breakdown and the dominant kernel's roofline."""
    import torch
    import synth
    model, blob, n_params = make_model(ffi, cfg, dev)
    si = StepInputs(ffi, cfg, dev, rank)
    B, G = si.B, si.G
    D = si.x.numel() // B
    v = torch.empty_like(si.x)
    x_next = torch.empty_like(si.x)
    logp = torch.empty((B, 1), dtype=torch.float32, device=dev)
    lp_old = torch.empty((B, 1), dtype=torch.float32, device=dev)
    adv_all = torch.empty(si.n_r, dtype=torch.float32, device=dev)
    adv = adv_all[:B]
    loss = torch.zeros(1, dtype=torch.float32, device=dev)
    grad = torch.empty((B, 1), dtype=torch.float32, device=dev)
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=dev)
    ws_sde = torch.zeros(ffi.ff_sde_workspace_size(B, D), dtype=torch.uint8, device=dev)
    ws_loss = torch.zeros(ffi.ff_grpo_loss_workspace_size(B, 1), dtype=torch.uint8, device=dev)
    # old log-probs of the (synthetic) rollout policy: new + N(0, 0.01^2)
    model.ff_dit_velocity(si.x, si.txt, si.t, v, ws)
    ffi.ff_sde_step_logprob_philox(si.x, v, x_next, si.t, si.tn, si.sg, logp, si.noise_seed, 0, ws=ws_sde)
    torch.add(logp, si.jitter, out=lp_old)

    def step(xi=si.x, txti=si.txt, ti=si.t, tni=si.tn, sgi=si.sg, ri=si.r, lpo=lp_old, xo=x_next, lpn=logp,
             lo=loss):
        model.ff_dit_velocity(xi, txti, ti, v, ws)
        ffi.ff_sde_step_logprob_philox(xi, v, xo, ti, tni, sgi, lpn, si.noise_seed, 0, ws=ws_sde)
        ffi.ff_group_advantage(ri, G, cfg["eps_adv"], adv_all)
        ffi.ff_grpo_loss(lpn, lpo, adv, cfg["clip"], cfg["clip"], lo, grad, ws=ws_loss)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize(dev)
    ms_step = timed(step, steps) / steps
    n_img = synth.n_img(cfg)
    prof_steps = max(1, min(steps, 5))
    kern, launches = kernel_table(ffi, step, prof_steps, timed, cfg)
    dominant = max(kern, key=lambda k: kern[k][1])
    dit_flops = sum(k[2] for k in kern.values()) / prof_steps
    _, tc_burst, _, _ = load_peaks()
    out = {"workload": workload_desc(cfg), "ms_per_step": ms_step,
           "value": whole_job_rate(world, B * n_img, ms_step), "unit": UNIT, "steps": steps, "warmup": warmup,
           "dit_tflops": dit_flops / (ms_step / 1e3) / 1e12,
           "dit_frac_of_burst": dit_flops / (ms_step / 1e3) / 1e12 / tc_burst,
           "roofline": roofline_of(kern, dominant, cfg["name"]),
           "secondary_rooflines": {k: roofline_of(kern, k, cfg["name"]) for k in ("gemm_bf16", "attention",
                                                                                   "sde_step", "grpo_loss")
                                   if k in kern and k != dominant},
           "kernel_breakdown": breakdown_of(kern, prof_steps),
           "gpu_launches_per_step": launches // prof_steps,
           "weights_gb": 2 * n_params / 1e9, "workspace_gb": ws.numel() / 1e9}
    ctx = {"model": model, "blob": blob, "si": si, "step": step, "v": v, "x_next": x_next, "logp": logp,
           "lp_old": lp_old, "loss": loss, "adv": adv, "adv_all": adv_all, "grad": grad, "ws": ws,
           "ws_sde": ws_sde, "ws_loss": ws_loss, "launches_per_step": launches // prof_steps,
           "dit_flops": dit_flops, "n_params": n_params}
    if not keep_model:
        model.close()
        del ctx, blob
        torch.cuda.empty_cache()
        return out, None
    return out, ctx


def measure_rollout_workload(ffi, cfg, dev, rank, world, timed, steps=3, warmup=1):
    """The configured trajectory sampling of a workload: S denoise steps
    (velocity + SDE step with in-kernel noise + log-prob, all S log-probs
    kept) from x_T for the whole batch (ff_rollout_philox), then the group
    advantage and the clipped GRPO loss over [B, S] with dL/dlp."""
    import torch
    import synth
    model, blob, n_params = make_model(ffi, cfg, dev)
    si = StepInputs(ffi, cfg, dev, rank)
    B, G, S = si.B, si.G, cfg["steps_run"]
    t = torch.tensor(si.tgrid[:S + 1], dtype=torch.float32, device=dev)
    sg = torch.tensor(si.sig[:S], dtype=torch.float32, device=dev)
    x = torch.empty_like(si.x)
    logp = torch.empty((B, S), dtype=torch.float32, device=dev)
    lp_old = torch.empty_like(logp)
    adv = torch.empty(si.n_r, dtype=torch.float32, device=dev)
    loss = torch.zeros(1, dtype=torch.float32, device=dev)
    grad = torch.empty_like(logp)
    ws = torch.empty(model.rollout_workspace_size(B, S), dtype=torch.uint8, device=dev)
    ws_loss = torch.zeros(ffi.ff_grpo_loss_workspace_size(B, S), dtype=torch.uint8, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(9 + rank_seed(rank))
    x.copy_(si.x)
    model.ff_rollout_philox(x, si.txt, t, sg, si.noise_seed, logp, ws=ws)
    torch.add(logp, 0.01 * torch.randn(logp.shape, generator=g, device=dev), out=lp_old)

    def step():
        x.copy_(si.x)                       # every rollout starts from x_T
        model.ff_rollout_philox(x, si.txt, t, sg, si.noise_seed, logp, ws=ws)
        ffi.ff_group_advantage(si.r, G, cfg["eps_adv"], adv)
        ffi.ff_grpo_loss(logp, lp_old, adv[:B], cfg["clip"], cfg["clip"], loss, grad, ws=ws_loss)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize(dev)
    ms = timed(step, steps) / steps
    kern, launches = kernel_table(ffi, step, 1, timed, cfg)
    dominant = max(kern, key=lambda k: kern[k][1])
    dit_flops = sum(k[2] for k in kern.values())
    _, tc_burst, _, _ = load_peaks()
    n_img = synth.n_img(cfg)
    out = {"workload": workload_desc(cfg, rollout=True), "ms_per_step": ms,
           "value": whole_job_rate(world, B * n_img * S, ms), "unit": UNIT, "steps": steps, "warmup": warmup,
           "denoise_steps_per_rollout": S,
           "dit_tflops": dit_flops / (ms / 1e3) / 1e12, "dit_frac_of_burst": dit_flops / (ms / 1e3) / 1e12 / tc_burst,
           "roofline": roofline_of(kern, dominant, cfg["name"]),
           "kernel_breakdown": breakdown_of(kern, 1), "gpu_launches_per_step": launches,
           "weights_gb": 2 * n_params / 1e9}
    model.close()
    del blob, ws
    torch.cuda.empty_cache()
    return out


def run_ours(args):
    import numpy as np
    import torch
    import torch.distributed as dist

    import synth
    from paper_2602_12529_gb300 import build, ffi

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        dist.init_process_group("nccl", device_id=dev)
    if rank == 0 or not os.path.exists(build.LIB):
        build.build()
    if world > 1:
        dist.barrier()
    ffi.lib()
    stream = torch.cuda.current_stream(dev)

    def timed(fn, k):
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(k):
            fn()
        e1.record(stream)
        torch.cuda.synchronize(dev)
        ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
        if world > 1:
            dist.barrier()
        return ms

    cfg = synth.config(args.workload)
    B, G, Nt, Ni = cfg["batch"], cfg["group"], cfg["n_txt"], synth.n_img(cfg)
    clocks = ClockSampler(local) if rank == 0 else None
    head, ctx = measure_step_workload(args, ffi, cfg, dev, rank, world, timed, args.steps, args.warmup,
                                      keep_model=True)
    model, si, step = ctx["model"], ctx["si"], ctx["step"]
    ms_step = head["ms_per_step"]

    # ---- end to end through the public API with host inputs: every step
    # copies its inputs in from pinned host memory and its results (x_next,
    # log-probs, loss) out; HostFedPipeline overlaps step k + 1's copies in
    # and step k's copies out with step k's kernels (two device buffer sets,
    # a copy stream, events).  The serial form (copies on the compute stream)
    # is reported beside it.
    from paper_2602_12529_gb300.pipeline import HostFedPipeline
    pin = lambda a: torch.from_numpy(np.ascontiguousarray(a)).pin_memory()
    h_in = {k: pin(si.h[k]) for k in ("x", "txt", "t", "tn", "sg", "r")}
    h_in["lpo"] = ctx["lp_old"].cpu().pin_memory()
    h_out = [{"x_next": torch.empty(si.x.shape, dtype=torch.float32).pin_memory(),
              "logp": torch.empty((B, 1), dtype=torch.float32).pin_memory(),
              "loss": torch.empty(1, dtype=torch.float32).pin_memory()} for _ in range(2)]
    h2d = sum(a.numel() * a.element_size() for a in h_in.values())
    d2h = sum(a.numel() * a.element_size() for a in h_out[0].values())

    def e2e_body(i, o):
        step(i["x"], i["txt"].view(torch.bfloat16), i["t"], i["tn"], i["sg"], i["r"], i["lpo"],
             o["x_next"], o["logp"], o["loss"])

    like_in = {"x": si.x, "txt": si.txt.view(torch.int16), "t": si.t, "tn": si.tn, "sg": si.sg, "r": si.r,
               "lpo": ctx["lp_old"]}
    pipe = HostFedPipeline(dev, like_in, {"x_next": ctx["x_next"], "logp": ctx["logp"], "loss": ctx["loss"]},
                           e2e_body)
    K_e2e = args.steps if ms_step < 200 else max(3, min(args.steps, 8))
    pipe.run([h_in] * 2, h_out)
    ms_e2e = timed(lambda: pipe.run([h_in] * K_e2e, [h_out[k % 2] for k in range(K_e2e)]), 1) / K_e2e
    e2e_value = whole_job_rate(world, B * Ni, ms_e2e)

    def e2e_serial():
        i = pipe.ins[0]
        for name, h_ in h_in.items():
            i[name].copy_(h_, non_blocking=True)
        e2e_body(i, pipe.outs[0])
        for name, h_ in h_out[0].items():
            h_.copy_(pipe.outs[0][name], non_blocking=True)

    e2e_serial()
    K_ser = min(K_e2e, 3)
    ms_e2e_serial = timed(e2e_serial, K_ser) / K_ser
    del pipe

    want_train = (not args.no_sweep or args.train_only) and rank == 0 and world == 1
    extras = want_train and not args.train_only
    light = argparse.Namespace(steps=min(args.steps, 3), warmup=min(args.warmup, 2))
    awm = awm_step(light, ffi, model, cfg, dev, si.x, si.txt, torch.randn_like(si.x), si.r, timed, world) \
        if extras else None
    train = train_step(argparse.Namespace(steps=2, warmup=1) if ms_step > 200 else light, ffi, model, cfg, dev,
                       si.x, si.txt, si.t, si.tn, si.sg, ctx["x_next"], ctx["lp_old"], ctx["adv"], ctx["dit_flops"],
                       timed, world) if want_train else None
    model.close()
    del ctx, model, step
    torch.cuda.empty_cache()

    # ---- the other workloads, each timed on its own (rank 0, one GPU)
    others = {}
    if extras:
        for name in ("flux_double_block", "flux_8d16s", "qwen_image_60d", "wan_40"):
            if name == args.workload:
                continue
            ocfg = synth.config(name)
            if name == "flux_8d16s":
                others[name] = measure_rollout_workload(ffi, ocfg, dev, rank, world, timed)
            elif name == "wan_40":
                others[name], _ = measure_step_workload(args, ffi, ocfg, dev, rank, world, timed, 3, 2)
            else:
                others[name], _ = measure_step_workload(args, ffi, ocfg, dev, rank, world, timed,
                                                        10 if name == "flux_double_block" else 5, 3)
            torch.cuda.empty_cache()
    bwd = backward_kernels(args, ffi, synth.config("flux_double_block"), dev) if extras else None
    at_cfg = at_config_small_kernels(ffi, dev, load_peaks()[0], cfg, rank) if extras else None
    sweep = hbm_sweep(ffi, dev, load_peaks()[0]) if extras else None
    clk = clocks.stop() if clocks else None
    status = ffi.ff_check_device_status()

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        rate, secs, sample = oracle_rate(cfg)
        cpu = {"value": rate, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle", "sample": sample}

    if rank == 0:
        line = {"metric": METRIC, "value": head["value"], "unit": UNIT, "n_gpus": world, "steps": args.steps,
                "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
                "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
                "config": {"workload": head["workload"], "batch": B, "group": G, "n_txt": Nt, "n_img": Ni,
                           "hidden": cfg["hidden"], "parallelism": f"dp{world} (independent groups per GPU)",
                           "l2": f"no flush: per-step working set ({head['weights_gb']:.2f} GB weights + "
                                 f"{head['workspace_gb']:.2f} GB activation workspace) > 129 MB L2"},
                "roofline": head["roofline"],
                "dit_tflops": head["dit_tflops"],
                "dit_frac_of_burst": head["dit_frac_of_burst"],
                "secondary_rooflines": head["secondary_rooflines"],
                "kernel_breakdown": head["kernel_breakdown"],
                "cpu_baseline": cpu,
                "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                        "ms_per_step": ms_e2e, "steps": K_e2e,
                        "copies": "overlapped with the previous / next step's kernels "
                                  "(HostFedPipeline: copy stream, two device buffer sets)",
                        "serial_ms_per_step": ms_e2e_serial},
                "other_workloads": others,
                "hbm_sweep": sweep,
                "small_kernels_at_config": at_cfg,
                "awm_step": awm,
                "train_step": train,
                "backward_kernels": bwd,
                "gpu_launches": head["gpu_launches_per_step"] * args.steps,
                "clocks": clk,
                "device_status": status}
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def profile_kernel(args):
    """Launch one kernel `reps` times on rotating inputs, for an ncu capture
    (`-k regex:<kernel> -s <skip> -c <count>`); prints what it launched.
    HBM kernels run at --elements elements (two input sets, each larger
    than L2 at the default 2^24); attention and LN-modulate at the
    workload's own shapes; velocity is one whole velocity call."""
    import torch

    import synth
    from paper_2602_12529_gb300 import build, ffi
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    build.build()
    ffi.lib()
    n, k, reps = args.elements, args.profile_kernel, 4
    cfg = synth.config(args.workload)
    g = torch.Generator(device=dev)
    g.manual_seed(3)
    rnd = lambda *shape: torch.randn(*shape, generator=g, device=dev)
    if k in ("sde_step", "sde_step_philox"):
        B, D = 4, n // 4
        sets = [tuple(rnd(B, D) for _ in range(4)) for _ in range(2)]
        t, tn, sg = torch.full((B,), 0.75, device=dev), torch.full((B,), 0.5, device=dev), torch.full((B,), 0.7,
                                                                                                      device=dev)
        lp = torch.empty(B, device=dev)
        ws = torch.zeros(ffi.ff_sde_workspace_size(B, D), dtype=torch.uint8, device=dev)
        for i in range(reps):
            x, v, e, o = sets[i % 2]
            if k == "sde_step":
                ffi.ff_sde_step_logprob(x, v, e, o, t, tn, sg, lp, ws=ws)
            else:
                ffi.ff_sde_step_logprob_philox(x, v, o, t, tn, sg, lp, 7, 0, ws=ws)
        what = f"{k}: B 4 x D {D} fp32 ({(16 if k == 'sde_step' else 12) * n / 1e6:.0f} MB per launch)"
    elif k == "grpo_loss":
        Bq, T = n // 16, 16
        sets = []
        for _ in range(2):
            a = rnd(Bq, T)
            sets.append((a, a + 0.01 * rnd(Bq, T), rnd(Bq), torch.empty_like(a)))
        loss = torch.empty(1, device=dev)
        ws = torch.zeros(ffi.ff_grpo_loss_workspace_size(Bq, T), dtype=torch.uint8, device=dev)
        for i in range(reps):
            a, b, adv, gr = sets[i % 2]
            ffi.ff_grpo_loss(a, b, adv, 0.2, 0.2, loss, gr, ws=ws)
        what = f"grpo_loss with dL/dlp: B {Bq} x T {T} ({(12 * n + 4 * Bq) / 1e6:.0f} MB per launch)"
    elif k == "group_advantage":
        sets = [(torch.rand(n, generator=g, device=dev), torch.empty(n, device=dev)) for _ in range(2)]
        for i in range(reps):
            ffi.ff_group_advantage(sets[i % 2][0], 16, 1e-4, sets[i % 2][1])
        what = f"group_advantage: {n} rewards in groups of 16 ({8 * n / 1e6:.0f} MB per launch)"
    elif k == "ln_modulate":
        rows, H = cfg["batch"] * (synth.n_img(cfg) + cfg["n_txt"]), cfg["hidden"]
        x = rnd(rows, H)
        mods = rnd(cfg["batch"], 2 * H)
        out = torch.empty(rows, H, dtype=torch.bfloat16, device=dev)
        for _ in range(reps):
            ffi.ff_debug_ln_modulate(x, mods, 0, H, rows // cfg["batch"], out)
        what = f"ln_modulate: {rows} rows x {H} fp32 -> bf16 ({6 * rows * H / 1e6:.0f} MB per launch)"
    elif k in ("attention", "attention_backward"):
        B, heads, d = cfg["batch"], cfg["heads"], cfg["head_dim"]
        H = heads * d
        if cfg.get("arch") == "wan":
            n0, n1 = 0, synth.n_img(cfg)
        else:
            n0, n1 = cfg["n_txt"], synth.n_img(cfg)
        q0 = rnd(max(B * n0, 1), 3 * H).to(torch.bfloat16)
        q1 = rnd(B * n1, 3 * H).to(torch.bfloat16)
        o0 = torch.empty(max(B * n0, 1), H, dtype=torch.bfloat16, device=dev)
        o1 = torch.empty(B * n1, H, dtype=torch.bfloat16, device=dev)
        aws = torch.empty(ffi.ff_attention_forward_workspace_size(d), dtype=torch.uint8, device=dev)
        if k == "attention":
            for _ in range(reps):
                ffi.ff_attention_forward(B, heads, d, q0, o0, n0, q1, o1, n1, ws=aws)
        else:   # the backward (D, dQ, dK / dV kernels) after one forward that keeps lse
            lse = torch.empty(B * heads * ffi.lib().ff_attention_lse_rows(n0, n1), device=dev)
            ffi.ff_attention_forward(B, heads, d, q0, o0, n0, q1, o1, n1, lse=lse, ws=aws)
            g0, g1 = rnd(max(B * n0, 1), H).to(torch.bfloat16), rnd(B * n1, H).to(torch.bfloat16)
            dq0, dq1 = torch.empty_like(q0), torch.empty_like(q1)
            for _ in range(reps):
                ffi.ff_attention_backward(B, heads, d, (n0, q0, o0, g0, dq0), (n1, q1, o1, g1, dq1), lse)
        what = f"{k}: B {B}, {heads} x {d} heads, {n0} + {n1} tokens"
    else:
        model, blob, _ = make_model(ffi, cfg, dev)
        si = StepInputs(ffi, cfg, dev, 0)
        v = torch.empty_like(si.x)
        ws = torch.empty(model.workspace_size(si.B), dtype=torch.uint8, device=dev)
        for _ in range(2):
            model.ff_dit_velocity(si.x, si.txt, si.t, v, ws)
        what = f"velocity: {workload_desc(cfg)} (2 calls)"
        reps = 2
    torch.cuda.synchronize(dev)
    print(json.dumps({"profile_kernel": k, "launches": reps, "what": what,
                      "device_status": ffi.ff_check_device_status()}), flush=True)
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.profile_kernel:
        return profile_kernel(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
