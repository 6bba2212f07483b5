"""fp64 CPU oracle of the rollout denoising step (test infrastructure only).

This package is the plain, slow, obviously-correct statement of what the CUDA
path computes, written from the paper and checked against closed forms,
invariants and brute force in ``tests/test_oracle_*.py``.  It is test
infrastructure: only ``tests/``, ``__graft_entry__.smoke()`` and the CPU
baseline leg of ``bench.py`` may import it.  The CUDA library never calls it,
and it shares no code with the CUDA path (only the seeded inputs of
``synth/``).

Modules:
  sde   -- time grids, noise schedules (Table 1), the Flow-SDE update (Eq. 1)
           and its Gaussian transition log-probability.
  grpo  -- group-normalised advantage (one or several rewards) and the
           clipped-ratio policy loss (optionally with per-step weights).
  awm   -- training-time sampling, the forward process x_t and the
           advantage-weighted matching loss of Eq. 3.
  nft   -- the DiffusionNFT loss of Eq. 2 (implicit positive / negative
           policies read from the cited method).
  dit   -- the flow-matching DiT velocity v_theta(x_t, t): MMDiT double- and
           single-stream blocks (adaLN modulation, QK-RMSNorm, RoPE, joint
           attention, GELU MLP) and the final projection, and the WAN-style
           network (self-attention, text cross-attention, FFN).
  dit_grad -- the gradient of <dv, v_theta> with respect to every weight and
           x_t: the training pass's vector-Jacobian product, one elementary
           backward per forward step.
  linalg -- the three dense products of a Linear's backward.
  philox -- counter-based Gaussian noise for SAMPLE steps: Philox4x32-10 and
           the Box-Muller transform.

Every array is float64; bf16 weights and inputs are widened exactly.  Nothing
is rounded between steps.

Parity status: sde, grpo and awm are pinned by closed forms; the DiT pieces are
pinned one by one (attention, RoPE, norms, GELU, modulation identity) and the
whole velocity only through those pieces plus invariants ("parity unpinned" as
a whole: no printed outputs exist for a random-init network).  dit_grad is
pinned by central differences of that velocity, per tensor.  philox is pinned
by an independent library implementation of the generator and by the
Gaussian statistics of its output.
"""
