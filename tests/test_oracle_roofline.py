"""Pins of the oracle's theoretical timing model (CPU only).

Every cell of the paper's printed slowdown and speedup tables (Sec. "Timing
analysis", transcribed in tests/golden/roofline_tables.txt) must come out of
the model rounded to the printed three decimals; plus the model's limits
(time(1) ratios of 1, speedup equal to the NFE speedup when a block forward
costs what a one-token forward does); and the linear-layer GEMM of the
measured forwards against its explicit triple sum."""
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "roofline_tables.txt")


def _cells():
    out = []
    for line in open(GOLDEN):
        if line.startswith("#") or not line.strip():
            continue
        kind, b, nfe, L, blk, v = line.split()
        out.append((kind, int(b), int(nfe), int(L), int(blk), float(v)))
    return out


def test_every_printed_cell():
    cells = _cells()
    assert len(cells) == 512
    bad = []
    for kind, b, nfe, L, blk, v in cells:
        if kind == "slowdown":
            got = oracle.block_slowdown(blk, L, b)
        else:
            got = oracle.sbd_speedup(blk, blk // nfe, lambda n: oracle.roofline_forward(n, L, b))
        # half a printed unit, plus 2e-5 for cells on a rounding boundary
        # (the batch-8, NFE-8, k = 64 column sits at 3.73651)
        if abs(got - v) > 0.0005 + 2e-5:
            bad.append((kind, b, nfe, L, blk, v, round(got, 4)))
    assert not bad, bad[:10]


def test_limits():
    assert oracle.block_slowdown(1, 4096, 8) == 1.0
    flat = lambda n: 1.0                                    # a block costs one forward
    for k, l in ((8, 2), (16, 4), (32, 1)):
        assert oracle.sbd_speedup(k, l, flat) == pytest.approx(k / l)   # = the NFE speedup
    # k forwards of one token against one forward of 2k: the (l - 1) term vanishes at l = 1
    lin = lambda n: float(n)
    assert oracle.sbd_speedup(16, 1, lin) == pytest.approx(16 / 32)


def test_gemm_roofline_regimes():
    c = oracle.ROOFLINE_H100
    t, f = oracle.roofline_gemm(1, 4096, 4096)
    assert f == 2 * 4096 * 4096
    assert t == pytest.approx((4096 + 4096 * 4096 + 4096) / c["bandwidth"])   # memory-bound
    t, f = oracle.roofline_gemm(8192, 8192, 8192)
    assert t == pytest.approx(2 * 8192 ** 3 / c["peak_flops"])                 # compute-bound


def test_linear_is_the_explicit_triple_sum():
    rng = np.random.default_rng(0)
    x, w = rng.standard_normal((3, 5)), rng.standard_normal((4, 5))
    y = oracle.linear(x, w)
    for t in range(3):
        for n in range(4):
            assert y[t, n] == pytest.approx(sum(x[t, k] * w[n, k] for k in range(5)), abs=1e-12)
    assert oracle.linear(np.zeros((2, 5)), w).shape == (2, 4)
