"""Counter-based Gaussian noise for the rollout's SAMPLE steps, drawn where it
is used instead of on the host (fp64 numpy, exact integer arithmetic).

Test infrastructure only (see oracle/__init__.py).  The Flow-SDE step of
Eq. 1 needs one standard-normal eps per latent element and step.  The paper
does not say where the noise comes from; reading: a counter-based generator,
so any element of any step can be drawn independently, on any device, and
reproduced from (seed, step) alone.

Generator: Philox4x32 with 10 rounds (Salmon, Moraes, Dror and Shaw,
"Parallel random numbers: as easy as 1, 2, 3", SC 2011).  It maps a 128-bit
counter (c0, c1, c2, c3) and a 64-bit key (k0, k1) to four 32-bit words.  One
round, with the 64-bit products split into high and low words:
    (hi0, lo0) = M0 c0,   (hi1, lo1) = M1 c2
    (c0, c1, c2, c3) <- (hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0)
and between rounds the key advances by (W0, W1) modulo 2^32:
    M0 = 0xD2511F53, M1 = 0xCD9E8D57, W0 = 0x9E3779B9, W1 = 0xBB67AE85.

Layout (ours): element i of sample b in stream s (the step index) under seed
K uses counter (i // 4, b, s, 0) and key (K mod 2^32, K div 2^32); words
w0..w3 of that call give elements 4g .. 4g + 3.  Each word becomes a
uniform u = (floor(w / 512) + 1/2) 2^-23: 24 significant bits, so exact in
fp32, within [2^-24, 1 - 2^-24]; the Box-Muller transform turns the pairs
(u0, u1), (u2, u3) into
    z0, z1 = sqrt(-2 ln u0) (cos 2 pi u1, sin 2 pi u1)
    z2, z3 = sqrt(-2 ln u2) (cos 2 pi u3, sin 2 pi u3).
"""
from __future__ import annotations

import numpy as np

M0, M1 = 0xD2511F53, 0xCD9E8D57
W0, W1 = 0x9E3779B9, 0xBB67AE85
ROUNDS = 10
_MASK = np.uint64(0xFFFFFFFF)


def philox4x32(c0, c1, c2, c3, k0, k1, rounds: int = ROUNDS):
    """Philox4x32-R of arrays of counters (uint32-valued) under a key;
    returns the four output words as uint64 arrays holding 32-bit values."""
    c = [np.asarray(v, dtype=np.uint64) & _MASK for v in (c0, c1, c2, c3)]
    k0, k1 = np.uint64(int(k0) & 0xFFFFFFFF), np.uint64(int(k1) & 0xFFFFFFFF)
    for r in range(rounds):
        if r:
            k0 = np.uint64((int(k0) + W0) & 0xFFFFFFFF)
            k1 = np.uint64((int(k1) + W1) & 0xFFFFFFFF)
        p0 = np.uint64(M0) * c[0]
        p1 = np.uint64(M1) * c[2]
        hi0, lo0 = p0 >> np.uint64(32), p0 & _MASK
        hi1, lo1 = p1 >> np.uint64(32), p1 & _MASK
        c = [hi1 ^ c[1] ^ k0, lo1, hi0 ^ c[3] ^ k1, lo0]
    return c


def uniforms(words):
    """(floor(w / 512) + 1/2) 2^-23 for 32-bit words: in (0, 1), exact in fp32."""
    return ((np.asarray(words, dtype=np.uint64) >> np.uint64(9)).astype(np.float64) + 0.5) * 2.0 ** -23


def box_muller(u_a, u_b):
    """The pair (sqrt(-2 ln u_a) cos 2 pi u_b, sqrt(-2 ln u_a) sin 2 pi u_b)."""
    r = np.sqrt(-2.0 * np.log(u_a))
    return r * np.cos(2.0 * np.pi * u_b), r * np.sin(2.0 * np.pi * u_b)


def philox_normal(B: int, D: int, seed: int, stream: int) -> np.ndarray:
    """fp64 [B, D] standard normals of the layout above (D a multiple of 4)."""
    if D % 4:
        raise ValueError("D must be a multiple of 4")
    g = np.arange(D // 4, dtype=np.uint64)
    out = np.empty((B, D), dtype=np.float64)
    for b in range(B):
        w = philox4x32(g, np.full_like(g, b), np.full_like(g, stream), np.zeros_like(g),
                       seed & 0xFFFFFFFF, (seed >> 32) & 0xFFFFFFFF)
        u = [uniforms(x) for x in w]
        z0, z1 = box_muller(u[0], u[1])
        z2, z3 = box_muller(u[2], u[3])
        out[b] = np.stack([z0, z1, z2, z3], axis=1).reshape(D)
    return out
