"""Pins of the oracle's counter-based Gumbel noise (CPU only).

The generator is pinned by the published known-answer vectors of Philox4x32-10
(tests/golden/philox4x32_10_kat.txt); the noise built on it by the moments of
the standard Gumbel distribution (mean = the Euler-Mascheroni constant,
variance = pi^2 / 6), by a chi-square test of the uniforms, by the bounds of
u, and by an element-wise check of the counter layout against single calls."""
import math
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "philox4x32_10_kat.txt")


def _kat():
    out = []
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        ctr, key, res = (tuple(int(w, 16) for w in part.split()) for part in line.split("|"))
        out.append((ctr, key, res))
    return out


def test_known_answer_vectors():
    cases = _kat()
    assert len(cases) == 3
    for ctr, key, res in cases:
        got = oracle.philox4x32_10(np.array(ctr, dtype=np.uint32), np.array(key, dtype=np.uint32))
        assert tuple(int(x) for x in got) == res


def test_vectorised_calls_match_single_calls():
    rng = np.random.default_rng(0)
    ctr = rng.integers(0, 2 ** 32, (50, 4), dtype=np.uint64).astype(np.uint32)
    key = rng.integers(0, 2 ** 32, (50, 2), dtype=np.uint64).astype(np.uint32)
    many = oracle.philox4x32_10(ctr, key)
    for i in range(50):
        assert np.array_equal(many[i], oracle.philox4x32_10(ctr[i], key[i]))


def test_counter_layout_of_the_noise():
    rows, V, seed, offset = [3, 17, 0], 37, 0x1234_5678_9ABC_DEF0, (7 << 32) + 5
    g, x = oracle.philox_gumbel(rows, V, seed, offset)
    for r, n in enumerate(rows):
        for v in range(V):
            ctr = np.array([v // 4, n, offset & 0xFFFFFFFF, offset >> 32], dtype=np.uint32)
            key = np.array([seed & 0xFFFFFFFF, seed >> 32], dtype=np.uint32)
            word = int(oracle.philox4x32_10(ctr, key)[v % 4])
            assert int(x[r, v]) == word
            u = ((word >> 9) + 0.5) / 2 ** 23
            assert g[r, v] == pytest.approx(-math.log(-math.log(u)), rel=1e-14, abs=1e-15)


def test_uniforms_and_bounds():
    g, x = oracle.philox_gumbel(np.arange(64), 8192, seed=99)
    u = ((x >> 9).astype(np.float64) + 0.5) * 2.0 ** -23
    assert u.min() >= 2.0 ** -24 and u.max() <= 1.0 - 2.0 ** -24
    # every u is an fp32 value (24 significant bits), so the kernel's is exact
    assert np.array_equal(u.astype(np.float32).astype(np.float64), u)
    # chi-square of 256 equal bins over 2^19 uniforms
    counts = np.bincount((x >> 24).ravel(), minlength=256)
    expected = x.size / 256
    chi2 = float(((counts - expected) ** 2 / expected).sum())
    assert chi2 < 255 + 5 * math.sqrt(2 * 255)         # ~5 sigma of a chi-square(255)
    assert np.isfinite(g).all()


def test_gumbel_moments():
    g, _ = oracle.philox_gumbel(np.arange(128), 8192, seed=5, offset=11)   # 2^20 samples
    n = g.size
    euler_gamma = 0.5772156649015329
    assert abs(g.mean() - euler_gamma) < 5 * math.sqrt(math.pi ** 2 / 6 / n)
    assert abs(g.var() - math.pi ** 2 / 6) < 0.02


def test_streams_differ_by_row_seed_and_offset():
    a, _ = oracle.philox_gumbel([0, 1], 4096, seed=1, offset=0)
    b, _ = oracle.philox_gumbel([0, 1], 4096, seed=2, offset=0)
    c, _ = oracle.philox_gumbel([0, 1], 4096, seed=1, offset=1)
    for x, y in ((a[0], a[1]), (a[0], b[0]), (a[0], c[0])):
        assert abs(np.corrcoef(x, y)[0, 1]) < 0.1
