"""The host-fed pipeline (copies of the next batch in and of the previous
batch's results out overlapping each batch's kernels) gives, batch by batch,
bit for bit the results of running the same batches one at a time."""
import numpy as np
import pytest

import synth

pytestmark = pytest.mark.gpu


def test_host_fed_pipeline_matches_serial_steps(cuda):
    import torch
    from paper_2602_12529_gb300 import ffi, weights
    from paper_2602_12529_gb300.pipeline import HostFedPipeline
    cfg = synth.config("tiny_mmdit")
    B, G = cfg["batch"], cfg["batch"]
    model = ffi.Dit(cfg, weights.pack(cfg, lambda n, s: synth.weight(n, s, synth.weight_kind(n), 0), cuda))
    D = synth.n_img(cfg) * cfg["patch_dim"]
    v = torch.empty((B, synth.n_img(cfg), cfg["patch_dim"]), dtype=torch.float32, device=cuda)
    ws = torch.empty(model.workspace_size(B), dtype=torch.uint8, device=cuda)
    ws_sde = torch.zeros(ffi.ff_sde_workspace_size(B, D), dtype=torch.uint8, device=cuda)
    ws_loss = torch.zeros(ffi.ff_grpo_loss_workspace_size(B, 1), dtype=torch.uint8, device=cuda)
    adv = torch.empty(B, dtype=torch.float32, device=cuda)
    grad = torch.empty((B, 1), dtype=torch.float32, device=cuda)

    def body(i, o):
        model.ff_dit_velocity(i["x"], i["txt"].view(torch.bfloat16), i["t"], v, ws)
        ffi.ff_sde_step_logprob(i["x"], v, i["eps"], o["x_next"], i["t"], i["tn"], i["sg"], o["logp"], ws=ws_sde)
        ffi.ff_group_advantage(i["r"], G, 1e-4, adv)
        ffi.ff_grpo_loss(o["logp"], i["lpo"], adv, 0.2, 0.2, o["loss"], grad, ws=ws_loss)

    n = 5
    host_in = []
    for k in range(n):
        rng = np.random.default_rng(40 + k)
        host_in.append({k_: torch.from_numpy(np.ascontiguousarray(a)).pin_memory() for k_, a in {
            "x": synth.initial_latent(cfg, seed=2 + k),
            "txt": synth.text_embeds(cfg, seed=1 + k).view(np.int16),
            "eps": synth.step_noise(cfg, 0, seed=100 + k),
            "t": np.full(B, 0.9 - 0.1 * k, np.float32), "tn": np.full(B, 0.7 - 0.1 * k, np.float32),
            "sg": np.full(B, 0.7, np.float32), "r": rng.uniform(0, 1, B).astype(np.float32),
            "lpo": rng.standard_normal((B, 1)).astype(np.float32)}.items()})
    like_in = {k_: torch.empty(h.shape, dtype=h.dtype, device=cuda) for k_, h in host_in[0].items()}
    like_out = {"x_next": torch.empty_like(v), "logp": torch.empty((B, 1), device=cuda),
                "loss": torch.empty(1, device=cuda)}
    out_p = [{k_: torch.empty(t.shape, dtype=t.dtype).pin_memory() for k_, t in like_out.items()} for _ in range(n)]
    pipe = HostFedPipeline(cuda, like_in, like_out, body)
    pipe.run(host_in, out_p)
    torch.cuda.synchronize()
    assert ffi.ff_check_device_status() == 0
    # the same batches one at a time, copies on the compute stream
    for k in range(n):
        i = {k_: h.to(cuda) for k_, h in host_in[k].items()}
        o = {k_: torch.empty_like(t) for k_, t in like_out.items()}
        body(i, o)
        torch.cuda.synchronize()
        for k_ in like_out:
            assert torch.equal(o[k_].cpu(), out_p[k][k_]), (k, k_)
    # distinct batches gave distinct results (the pipeline did not reuse a set)
    assert not torch.equal(out_p[0]["x_next"], out_p[1]["x_next"])
