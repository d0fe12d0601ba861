"""The multi-layer block-step loop of the sweep (Algorithm 3), run through
the bench's own SweepLoop at reduced sizes and replayed step by step through
the oracle: every layer's attention output (Eq. 5), every step's entropies
and sampled tokens (Eqs. 6-7), unmask sets (Eq. 3), committed tokens and
the number of steps per block.

The loop draws its inputs on the device; the test copies them back and
hands the oracle exactly those values."""
import numpy as np
import pytest

import gen
import oracle
from tests.helpers import (BF16_ATTN_TOL, ENTROPY_TOL, GAMMA_MARGIN, compare_unmask,
                           token_tolerance, top2_gap)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sbd():
    import paper_2509_04185_gb300 as m
    return m


def _bits(t) -> np.ndarray:
    """A device bf16 tensor as its raw uint16 bit patterns on the host."""
    import torch
    return t.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def _replay(loop, trace, noise, tau, gamma):
    """Returns (token exemptions, unmask exemptions, oracle steps)."""
    w = loop.w
    B, k = w.batch, w.block_k
    for L_, out in zip(loop.layers, loop.outs):
        f = {x: oracle.widen(_bits(L_[x]), "bf16") for x in ("q", "kc", "vc", "kb", "vb")}
        ref = oracle.block_attention(f["q"], f["kc"], f["vc"], loop.lens.cpu().numpy(), f["kb"],
                                     f["vb"])
        got = out.float().cpu().numpy()
        assert np.isfinite(got).all()
        assert float(np.abs(got - ref).max()) <= BF16_ATTN_TOL
    W = _bits(loop.W)
    g_buf = loop.gumbel.cpu().numpy() if noise == "buffer" else None
    tok_exempt = set_exempt = 0
    # the oracle's own loop, fed the same per-step inputs
    o_masked = np.ones((B, k), dtype=np.uint8)
    o_bt = np.full((B, k), -1, dtype=np.int32)
    o_steps = 0
    for t in trace:
        s = t["step"]
        m_before = t["masked_before"]
        assert np.array_equal(m_before, o_masked), ("state diverged before step", s)
        if noise == "buffer":
            g = g_buf
        else:
            g = oracle.philox_gumbel(list(range(B * k)), w.vocab, loop.seed, s)[0].reshape(
                B, k, w.vocab)
        hid = oracle.widen(_bits(loop.hidden[min(s, k - 1)]), "bf16")
        rent, rtok, zs = oracle.head_entropy_sample(hid, W, "bf16", m_before, g, tau)
        sel = m_before.astype(bool)
        ent, tok = t["entropy"], t["token"]
        assert np.abs(ent[sel] - rent[sel]).max() <= ENTROPY_TOL
        # tokens: equal, except where the oracle's top-2 scores are a tie at
        # the kernel's precision (+ the fp32 rounding of in-kernel noise)
        tied = set()
        for (b, i), z in zs.items():
            if tok[b, i] != rtok[b, i]:
                gap = top2_gap(z, None if g is None else g[b, i], tau)
                slack = 2e-5 * tau if noise == "philox" else 0.0
                assert gap < token_tolerance(z, w.hidden // 16) + slack, (s, b, i, gap)
                tied.add((b, i))
        tok_exempt += len(tied)
        # unmask set: the oracle's EB set on its own entropies
        m_after = t["masked_after"]
        set_exempt += compare_unmask(m_before, rent, gamma, m_after, tie_tol=GAMMA_MARGIN)
        newly = sel & ~m_after.astype(bool)
        assert np.array_equal(t["n_unmasked"], newly.sum(axis=1))
        assert np.all(t["n_unmasked"][sel.any(axis=1)] >= 1)
        # committed tokens: the GPU's samples at exactly the unmasked
        # positions, the oracle's samples unless that row was a tie
        bt = t["bt_after"]
        assert np.array_equal(bt[newly], tok[newly])
        assert np.array_equal(bt[~newly], t["bt_before"][~newly])
        for b, i in zip(*np.nonzero(newly)):
            if (b, i) not in tied:
                assert bt[b, i] == rtok[b, i], (s, b, i)
        # the oracle's step on its own state
        o_masked, o_bt, _, _, _ = oracle.eb_select(rent, rtok, o_masked, o_bt, float(np.float32(gamma)))
        if not np.array_equal(o_masked, m_after):      # an exempted decision: follow the GPU
            o_masked = m_after.copy()
        o_bt = np.where(newly, bt, o_bt)
        o_steps += 1
    assert not o_masked.any()
    final = trace[-1]["bt_after"]
    assert (final >= 0).all() and (final < w.vocab).all()
    return tok_exempt, set_exempt, o_steps


@pytest.mark.parametrize("noise", ["buffer", "philox"])
@pytest.mark.parametrize("gamma", [0.1, 1.0])
def test_reduced_sweep_loop_matches_the_oracle(sbd, noise, gamma):
    """2 layers, batch 2, k = 32, cache 512, vocab 4096, hidden 4096: the
    sweep's code path (bench.SweepLoop) with every block starting fully
    masked, replayed through the oracle."""
    import torch

    import bench
    w = gen.shrink(gen.sweep_workload(32), n_layers=2, batch=2, cache_len=512, vocab=4096)
    stream = torch.cuda.current_stream()
    loop = bench.SweepLoop(w, seed=3, noise=noise, tau=1.0, gamma=gamma,
                           dev=torch.device("cuda"), stream=stream)
    trace = []
    steps = loop.block(trace=trace)
    assert sbd.sbd_device_error() == 0
    assert steps == len(trace) and 1 <= steps <= w.block_k
    tok_ex, set_ex, o_steps = _replay(loop, trace, noise, 1.0, gamma)
    print(f"steps {steps}, token exemptions {tok_ex}, unmask exemptions {set_ex}")
    assert o_steps == steps
    assert tok_ex <= 1 and set_ex <= 1
    # a second block from the same inputs repeats the first exactly
    trace2 = []
    assert loop.block(trace=trace2) == steps
    assert np.array_equal(trace2[-1]["bt_after"], trace[-1]["bt_after"])


def test_reduced_sweep_small_blocks(sbd):
    """k = 4 (the attention's register path) and k = 8, batch 3, 3 layers."""
    import torch

    import bench
    for k in (4, 8):
        w = gen.shrink(gen.sweep_workload(k), n_layers=3, batch=3, cache_len=300, vocab=3000,
                       hidden=1024)
        loop = bench.SweepLoop(w, seed=k, noise="buffer", tau=1.0, gamma=0.1,
                               dev=torch.device("cuda"), stream=torch.cuda.current_stream())
        trace = []
        steps = loop.block(trace=trace)
        tok_ex, set_ex, o_steps = _replay(loop, trace, "buffer", 1.0, 0.1)
        assert o_steps == steps and tok_ex <= 1 and set_ex <= 1
        assert sbd.sbd_device_error() == 0


@pytest.mark.parametrize("noise", ["buffer", "philox"])
def test_graphed_sweep_loop_matches_eager(sbd, noise):
    """The bench times the loop with one CUDA graph per step index; those
    graphs take the same number of steps and commit the same tokens as the
    eager loop (whose steps the test above replays through the oracle)."""
    import torch

    import bench
    w = gen.shrink(gen.sweep_workload(16), n_layers=2, batch=2, cache_len=512, vocab=4096)
    stream = torch.cuda.Stream()
    loop = bench.SweepLoop(w, seed=5, noise=noise, tau=1.0, gamma=0.1,
                           dev=torch.device("cuda"), stream=stream)
    torch.cuda.synchronize()
    eager_steps = loop.block()
    bt_eager = loop.bt.cpu()
    loop.capture()
    for _ in range(2):
        graph_steps = loop.block()
        torch.cuda.synchronize()
        assert graph_steps == eager_steps
        assert torch.equal(loop.bt.cpu(), bt_eager)
    assert sbd.sbd_device_error() == 0
