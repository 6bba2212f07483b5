"""GPU checks of the batched fixed-order chunk reductions behind every
gradient sum of the training pass (bias, gate, shift / scale and norm-scale
gradients): against the fp64 sums of the same fp32 partials, and batching
against one job per launch, bit for bit."""
import numpy as np
import pytest

from paper_2602_12529_gb300 import ffi

pytestmark = pytest.mark.gpu

B = 3


def _jobs():
    """Eleven jobs (two launches of up to eight): per-sample and total sums,
    one and two spans, ragged column counts, different pitches."""
    J = []
    off = 0
    for i, (ncols, ld, spans, per) in enumerate([
            (64, 64, [(0, 5)], True), (37, 40, [(2, 9)], False), (3072, 6144, [(0, 8), (24, 32)], True),
            (1, 4, [(1, 3)], False), (300, 304, [(0, 64), (192, 64)], False), (128, 256, [(0, 17)], True),
            (33, 36, [(4, 1)], True), (96, 96, [(0, 2), (6, 7)], True), (2048, 2048, [(0, 72)], False),
            (5, 8, [(0, 1), (1, 1)], False), (640, 640, [(3, 33)], True)]):
        rows = max(f + (B if per else 1) * c for f, c in spans)
        J.append(dict(part_off=off, ld_part=ld, ncols=ncols, spans=spans, per_sample=per, rows=rows))
        off += rows * ld + 4
    return J, off


def _want(part, j):
    base = part[j["part_off"]:j["part_off"] + j["rows"] * j["ld_part"]].reshape(j["rows"], j["ld_part"])
    base = base[:, :j["ncols"]].astype(np.float64)
    if j["per_sample"]:
        return np.stack([sum(base[f + b * c:f + (b + 1) * c].sum(0) for f, c in j["spans"]) for b in range(B)])
    return sum(base[f:f + c].sum(0) for f, c in j["spans"])[None, :]


def test_batched_reductions_match_fp64_sums_and_single_job_launches(cuda):
    import torch
    J, n_part = _jobs()
    rng = np.random.default_rng(7)
    part_h = (rng.standard_normal(n_part) * 10.0 ** rng.integers(-3, 4, n_part)).astype(np.float32)
    out_off = 0
    for j in J:
        j["out_off"] = out_off
        j["ld_out"] = j["ncols"] + 3
        out_off += (B if j["per_sample"] else 1) * j["ld_out"]
    part = torch.from_numpy(part_h).to(cuda)
    out = torch.full((out_off,), float("nan"), dtype=torch.float32, device=cuda)
    ffi.ff_debug_reduce_chunks(part, out, J, B)
    single = torch.full_like(out, float("nan"))
    for j in J:
        ffi.ff_debug_reduce_chunks(part, single, [j], B)
    torch.cuda.synchronize()
    got = out.cpu().numpy()
    for j in J:
        nr = B if j["per_sample"] else 1
        g = np.stack([got[j["out_off"] + b * j["ld_out"]:j["out_off"] + b * j["ld_out"] + j["ncols"]] for b in range(nr)])
        want = _want(part_h, j).astype(np.float32)
        # an fp64 sum of a few hundred fp32 terms rounds to fp32 like the exact sum, bar double rounding
        assert np.all(np.abs(g - want) <= np.spacing(np.abs(want))), j
    # unwritten gaps stay untouched, and batching changes no bit
    assert torch.equal(torch.isnan(out), torch.isnan(single))
    m = ~torch.isnan(out)
    assert torch.equal(out[m], single[m])
    assert ffi.ff_check_device_status() == 0
