"""The N > 1 host path of bench.py on CPU: two gloo ranks, each with its own
seeds and its own groups, the slowest rank's time taken by an all-reduce
MAX, and the whole-job rate counting both ranks.  Also checks that the
per-rank inputs differ and that a rank's groups need nothing from the other
rank (its advantages equal the ones computed from its own rewards alone)."""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    import sys
    import torch
    import torch.distributed as dist
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    sys.path.insert(0, root)
    import bench
    import synth
    from oracle import grpo as ogrpo
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    cfg = synth.config("tiny_mmdit")
    seed = bench.rank_seed(rank)
    r = synth.rewards(cfg["batch"], seed=7 + seed)
    x = synth.initial_latent(cfg, seed=2 + seed)
    adv_local = ogrpo.group_advantage(r, cfg["group"], cfg["eps_adv"])
    # gather everything on every rank only to check it, not as part of the path
    gathered = [None] * world
    dist.all_gather_object(gathered, (r, float(x[0, 0, 0])))
    ms = bench.max_over_ranks(10.0 + 5.0 * rank, world)
    rate = bench.whole_job_rate(world, cfg["batch"] * synth.n_img(cfg), ms)
    out[rank] = (ms, rate, adv_local, gathered)
    dist.destroy_process_group()


def test_two_gloo_ranks_shard_by_groups_and_time_by_the_slowest():
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    procs = [ctx.Process(target=_rank, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    import synth
    from oracle import grpo as ogrpo
    cfg = synth.config("tiny_mmdit")
    ms0, rate0, adv0, g0 = out[0]
    ms1, rate1, adv1, g1 = out[1]
    assert ms0 == ms1 == 15.0                      # the slowest rank's time on every rank
    tokens = cfg["batch"] * synth.n_img(cfg)
    assert rate0 == rate1 == pytest.approx(2 * tokens / 0.015)
    (r0, x0), (r1, x1) = g0
    assert not np.array_equal(r0, r1) and x0 != x1  # distinct prompts / noise / rewards per rank
    # a rank's advantages come from its own groups only
    np.testing.assert_array_equal(adv0, ogrpo.group_advantage(r0, cfg["group"], cfg["eps_adv"]))
    np.testing.assert_array_equal(adv1, ogrpo.group_advantage(r1, cfg["group"], cfg["eps_adv"]))


def test_single_rank_is_the_identity():
    import bench
    assert bench.max_over_ranks(12.5, 1) == 12.5
    assert bench.whole_job_rate(1, 1000.0, 2.0) == pytest.approx(5e5)
