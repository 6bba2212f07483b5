"""Pins of the counter-based noise (oracle/philox.py): the generator against
an independent library implementation of Philox4x32-10 (Triton's, run on the
CPU by its interpreter), the uniforms' grid, and the Gaussian statistics of
the Box-Muller output."""
import os

import numpy as np
import pytest
from scipy import stats

from oracle import philox


_TRITON_SCRIPT = r"""
import json, sys
import torch
import triton
import triton.language as tl


@triton.jit
def k(out_ptr, seed, n: tl.constexpr):
    offs = tl.arange(0, n)
    a, b, c, d = tl.randint4x(seed, offs)
    tl.store(out_ptr + offs * 4 + 0, a)
    tl.store(out_ptr + offs * 4 + 1, b)
    tl.store(out_ptr + offs * 4 + 2, c)
    tl.store(out_ptr + offs * 4 + 3, d)


seed, n = int(sys.argv[1]), int(sys.argv[2])
out = torch.zeros(n * 4, dtype=torch.int32)
k[(1,)](out, seed, n)
print(json.dumps([int(v) & 0xFFFFFFFF for v in out.tolist()]))
"""


def _triton_words(seed, n):
    """Triton's Philox4x32-10 (counter (offset, 0, 0, 0), key = the seed's two
    32-bit halves) for offsets 0 .. n - 1, run by its CPU interpreter in a
    fresh process (the interpreter is chosen when Triton is first imported)."""
    import json
    import subprocess
    import sys
    pytest.importorskip("triton")
    env = dict(os.environ, TRITON_INTERPRET="1")
    r = subprocess.run([sys.executable, "-c", _TRITON_SCRIPT, str(seed), str(n)], env=env, capture_output=True,
                       text=True, timeout=300)
    if r.returncode != 0:
        pytest.skip(f"triton interpreter unavailable: {r.stderr.strip().splitlines()[-1:]}")
    return np.array(json.loads(r.stdout.strip().splitlines()[-1]), dtype=np.int64).reshape(n, 4)


@pytest.mark.parametrize("seed", [0, 12345, 0x7FFFFFFF])
def test_philox_matches_an_independent_library_implementation(seed):
    n = 256
    want = _triton_words(seed, n)
    g = np.arange(n, dtype=np.uint64)
    got = philox.philox4x32(g, 0 * g, 0 * g, 0 * g, seed & 0xFFFFFFFF, seed >> 32)
    np.testing.assert_array_equal(np.stack([w.astype(np.int64) for w in got], axis=1), want)


def test_philox_rounds_and_key_matter():
    g = np.arange(64, dtype=np.uint64)
    base = philox.philox4x32(g, g, g, g, 1, 2)
    for other in (philox.philox4x32(g, g, g, g, 1, 2, rounds=9), philox.philox4x32(g, g, g, g, 2, 2),
                  philox.philox4x32(g, g, g, g, 1, 3), philox.philox4x32(g, g + 1, g, g, 1, 2)):
        assert all(np.mean(a != b) > 0.99 for a, b in zip(base, other))


def test_uniforms_lie_on_the_24_bit_grid_inside_the_unit_interval():
    w = np.array([0, 511, 512, 0xFFFFFFFF, 0x80000000], dtype=np.uint64)
    u = philox.uniforms(w)
    np.testing.assert_array_equal(u, np.array([0.5, 0.5, 1.5, 2 ** 23 - 0.5, 2 ** 22 + 0.5]) * 2.0 ** -23)
    assert np.all(u > 0) and np.all(u < 1)
    assert np.array_equal(u.astype(np.float32).astype(np.float64), u)


def test_normals_are_standard_normal():
    z = philox.philox_normal(4, 1 << 18, seed=7, stream=3).ravel()
    n = z.size
    assert abs(z.mean()) < 5 / np.sqrt(n)
    assert abs(z.var() - 1) < 5 * np.sqrt(2 / n)
    assert abs(stats.kurtosis(z, fisher=False) - 3) < 5 * np.sqrt(24 / n)
    assert stats.kstest(z, "norm").pvalue > 1e-3


def test_streams_samples_and_seeds_are_independent_and_reproducible():
    a = philox.philox_normal(2, 1 << 16, seed=11, stream=0)
    np.testing.assert_array_equal(a, philox.philox_normal(2, 1 << 16, seed=11, stream=0))
    others = (philox.philox_normal(2, 1 << 16, seed=11, stream=1), philox.philox_normal(2, 1 << 16, seed=12, stream=0))
    n = a[0].size
    for o in others:
        for b in range(2):
            assert abs(np.corrcoef(a[b], o[b])[0, 1]) < 5 / np.sqrt(n)
    assert abs(np.corrcoef(a[0], a[1])[0, 1]) < 5 / np.sqrt(n)
    # the Box-Muller pair of one call is uncorrelated too (even / odd elements)
    assert abs(np.corrcoef(a[0][0::2], a[0][1::2])[0, 1]) < 5 / np.sqrt(n / 2)
