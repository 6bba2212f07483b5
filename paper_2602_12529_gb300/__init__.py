"""GB300 (sm_103a) rollout denoising step of Flow-GRPO-style RL on flow-matching
DiTs: DiT velocity, SDE step + log-prob, group advantage and clipped policy
loss, as hand-written CUDA kernels behind the C ABI of include/ff.h.

``ffi`` is the ctypes binding (same names as the C functions); ``build`` compiles
libff.so in-tree; ``weights`` packs named bf16 tensors into the library's blob.
"""
from . import build, ffi  # noqa: F401

__all__ = ["build", "ffi"]
