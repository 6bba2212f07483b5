"""Packs named bf16 parameter tensors into the single device blob whose layout
ff_dit_weight_layout defines (every tensor at a 64-element aligned offset)."""
from __future__ import annotations

import numpy as np

from . import ffi


def layout(cfg: dict):
    return ffi.ff_dit_weight_layout(cfg)


def pack(cfg: dict, get_tensor, device="cuda"):
    """Allocate the blob on `device` and fill it tensor by tensor.

    get_tensor(name, shape) -> numpy uint16 array (bf16 bit patterns) of that
    shape.  Tensors are copied one at a time, so host memory stays bounded by
    the largest single tensor.  Returns a torch.bfloat16 tensor.
    """
    import torch
    specs, total = layout(cfg)
    blob = torch.zeros(total, dtype=torch.int16, device=device)
    for name, off, shape in specs:
        a = np.ascontiguousarray(get_tensor(name, shape), dtype=np.uint16)
        if a.shape != tuple(shape):
            raise ValueError(f"{name}: got shape {a.shape}, layout wants {shape}")
        blob[off:off + a.size].copy_(torch.from_numpy(a.ravel().view(np.int16)))
    return blob.view(torch.bfloat16)
