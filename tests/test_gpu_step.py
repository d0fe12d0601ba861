"""The whole block step loop (Algorithm 3): attention -> LM head with
entropy and Gumbel-max sampling -> EB select, repeated until the block has
no masks.  At every step the oracle evaluates the same state; unmask sets
must match except for the exemptions of the comparison rules."""
import numpy as np
import pytest

import gen
import oracle
from tests.helpers import (ENTROPY_TOL, GAMMA_MARGIN, compare_unmask, step_inputs, to_dev,
                           token_tolerance, top2_gap)

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sbd():
    import paper_2509_04185_gb300 as m
    return m


def _loop(sbd, w, gamma, seed=0, max_steps=None):
    import torch
    d = step_inputs(w, seed)
    dt = w.dtype
    att = {x: to_dev(d[x], dt) for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    lens = torch.from_numpy(d["cache_len"]).cuda()
    W = to_dev(d["w"], dt)
    masked = torch.from_numpy(d["masked"]).cuda()
    bt = torch.from_numpy(d["block_tokens"]).cuda()
    m_host = d["masked"].copy()
    bt_host = d["block_tokens"].copy()
    steps, exempt, tok_exempt = 0, 0, 0
    while m_host.any():
        sbd.sbd_block_attention(att["q"], att["k_cache"], att["v_cache"], lens, att["k_blk"],
                                att["v_blk"])
        hidden = gen.hidden_states(w, seed, steps)
        gumbel = gen.gumbel_noise(w, seed, steps)
        ent, tok = sbd.sbd_head_entropy_sample(to_dev(hidden, dt), W, masked,
                                               torch.from_numpy(gumbel).cuda(), 1.0)
        n_un = sbd.sbd_eb_select(ent, tok, gamma, masked, bt)
        new_m = masked.cpu().numpy()
        # oracle on the same state
        rent, rtok, zs = oracle.head_entropy_sample(oracle.widen(hidden, dt), d["w"], dt, m_host,
                                                    gumbel, 1.0)
        e = ent.cpu().numpy()
        t = tok.cpu().numpy()
        sel = m_host.astype(bool)
        assert np.abs(e[sel] - rent[sel]).max() <= ENTROPY_TOL
        # the order-tie rule of the comparison: oracle entropies closer
        # than GAMMA_MARGIN may be taken in either order
        exempt += compare_unmask(m_host, rent, gamma, new_m, tie_tol=GAMMA_MARGIN)
        nu = n_un.cpu().numpy()
        assert np.all(nu[m_host.any(axis=1)] >= 1)
        assert np.array_equal(nu, (m_host.astype(int) - new_m.astype(int)).sum(axis=1))
        # committed tokens: the sampled token at exactly the newly unmasked
        # positions, equal to the oracle's except at a score tie
        bt_now = bt.cpu().numpy()
        newly = sel & ~new_m.astype(bool)
        assert np.array_equal(bt_now[newly], t[newly])
        assert np.array_equal(bt_now[~newly], bt_host[~newly])
        acc = w.hidden // (16 if dt == "bf16" else 1)
        for b, i in zip(*np.nonzero(newly)):
            if bt_now[b, i] != rtok[b, i]:
                z = zs[(b, i)]
                assert top2_gap(z, gumbel[b, i], 1.0) < token_tolerance(z, acc), (steps, b, i)
                tok_exempt += 1
        bt_host = bt_now
        m_host = new_m
        steps += 1
        assert steps <= w.block_k
    final = bt.cpu().numpy()
    assert (final >= 0).all() and (final < w.vocab).all()
    assert sbd.sbd_device_error() == 0
    print(f"{w.name}: {steps} steps, unmask exemptions {exempt}, token exemptions {tok_exempt}")
    assert tok_exempt <= 1
    return steps, exempt


@pytest.mark.parametrize("gamma", [0.0, 0.1, 1.0])
def test_tiny_f32_loop(sbd, gamma):
    w = gen.get_workload("tiny_f32")
    steps, exempt = _loop(sbd, w, gamma)
    assert exempt == 0
    assert 1 <= steps <= 3


@pytest.mark.parametrize("gamma", [0.01, 0.1, 1.0])
def test_llama_small_vocab_loop(sbd, gamma):
    w = gen.shrink(gen.get_workload("llama8b_k16"), vocab=4096, cache_len=512)
    steps, exempt = _loop(sbd, w, gamma)
    assert exempt <= 1


def test_llama8b_full_loop(sbd):
    steps, exempt = _loop(sbd, gen.get_workload("llama8b_k16"), 0.1)
    assert exempt <= 1


def test_ragged_full_loop(sbd):
    steps, exempt = _loop(sbd, gen.get_workload("ragged_b32_k8"), 0.1)
    assert exempt <= 2
