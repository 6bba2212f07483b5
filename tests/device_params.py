"""Oracle parameters read from a bf16 weight blob that lives on the GPU.

The full-depth models hold up to 20e9 parameters: too many to draw on the
host or to keep in fp64.  Their weights are drawn on the device (torch's
seeded generator, N(0, 0.02) matrices, zero biases, unit norm scales) and
this mapping hands the oracle the same bf16 values, widened exactly to
fp64, one tensor at a time: the tensors of the block the oracle asked for
last are kept, earlier blocks are dropped.  With slice_mod, ``mod.w`` (the
MMDiT's all-block modulation matrix) is handed out as a row slicer, read
12H rows at a time.
Test infrastructure only: no arithmetic of the method is here.
"""
from __future__ import annotations

from collections.abc import Mapping

import numpy as np

from oracle import dit as odit

BLOCK_PREFIXES = ("double", "single", "blocks")


def draw_blob_on_device(specs, total, dev, seed=0, kind_of=None):
    """bf16 weight blob [total] on `dev`: N(0, 0.02) matrices, zero biases,
    unit norm scales (synth.weight_kind's naming)."""
    import torch

    import synth
    kind_of = kind_of or synth.weight_kind
    blob = torch.zeros(total, dtype=torch.bfloat16, device=dev)
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    for name, off, shape in specs:
        n = int(np.prod(shape))
        kind = kind_of(name)
        if kind == "matrix":
            for i in range(0, n, 1 << 28):          # no fp32 copy of a whole large matrix
                m = min(1 << 28, n - i)
                blob[off + i:off + i + m] = (torch.randn(m, generator=g, device=dev) * 0.02).to(torch.bfloat16)
        elif kind == "scale":
            blob[off:off + n] = 1.0
    return blob


class _RowSlicer:
    """Rows of a [R, C] parameter, fetched and widened on indexing."""

    def __init__(self, owner, off, shape):
        self.owner, self.off, self.shape = owner, off, tuple(shape)

    def __getitem__(self, rows):
        if not isinstance(rows, slice) or rows.step not in (None, 1):
            raise TypeError("row slices only")
        r0, r1, _ = rows.indices(self.shape[0])
        C = self.shape[1]
        return self.owner.fetch(self.off + r0 * C, (r1 - r0) * C).reshape(r1 - r0, C)


class DeviceParams(Mapping):
    def __init__(self, blob, specs, slice_mod=True):
        self.blob = blob
        self.slice_mod = slice_mod
        self.specs = {name: (off, tuple(shape)) for name, off, shape in specs}
        self.fixed = {}
        self.block = None
        self.block_cache = {}

    def fetch(self, off, n):
        import torch
        bits = self.blob[off:off + n].view(torch.int16).cpu().numpy().view(np.uint16)
        return odit.widen(bits)

    def __getitem__(self, name):
        off, shape = self.specs[name]
        if name == "mod.w" and self.slice_mod:
            return _RowSlicer(self, off, shape)
        parts = name.split(".")
        if parts[0] in BLOCK_PREFIXES:
            blk = parts[0] + "." + parts[1]
            if blk != self.block:
                self.block, self.block_cache = blk, {}
            cache = self.block_cache
        else:
            cache = self.fixed
        if name not in cache:
            cache[name] = self.fetch(off, int(np.prod(shape))).reshape(shape)
        return cache[name]

    def __iter__(self):
        return iter(self.specs)

    def __len__(self):
        return len(self.specs)
