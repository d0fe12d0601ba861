"""Pins of the oracle's LM-head logits, entropy and Gumbel-max token (CPU).

Closed forms (uniform -> log V, one-hot -> 0, two-point -> binary entropy,
small-variance random energy -> log V - sigma^2/2), SciPy's entropy routine,
PyTorch's linear layer for the logits, hand-built argmax cases and a
chi-square frequency test of the Gumbel-max sampler against softmax."""
import math

import numpy as np
import pytest
import scipy.stats
import torch

import gen
import oracle


@pytest.mark.parametrize("V", [512, 128256, 151936])
def test_uniform_logits_entropy_is_log_v(V):
    z = np.full(V, 3.25)
    assert abs(oracle.entropy(z) - math.log(V)) < 1e-9


def test_uniform_reference_values():
    # log 512, log 128256, log 151936 to 4 decimals
    assert abs(oracle.entropy(np.zeros(512)) - 6.2383) < 1e-4
    assert abs(oracle.entropy(np.zeros(128256)) - 11.7618) < 1e-4
    assert abs(oracle.entropy(np.zeros(151936)) - 11.9312) < 1e-4


def test_one_hot_entropy_is_zero():
    z = np.zeros(1000)
    z[17] = 1e4
    assert oracle.entropy(z) == 0.0


@pytest.mark.parametrize("a,b", [(0.0, 0.0), (1.0, -0.5), (-3.0, 2.0), (10.0, 0.0)])
def test_two_point_binary_entropy(a, b):
    p = 1.0 / (1.0 + math.exp(b - a))
    h = -(p * math.log(p) + (1 - p) * math.log(1 - p))
    assert abs(oracle.entropy(np.array([a, b])) - h) < 1e-12


def test_entropy_matches_scipy_and_is_shift_invariant():
    rng = np.random.default_rng(0)
    for _ in range(5):
        z = rng.standard_normal(4096) * rng.uniform(0.1, 8)
        p = np.exp(z - z.max())
        p /= p.sum()
        ref = scipy.stats.entropy(p)
        assert abs(oracle.entropy(z) - ref) < 1e-9
        assert abs(oracle.entropy(z + 123.0) - ref) < 1e-9


def test_random_energy_small_sigma():
    # V iid N(0, sigma^2) logits: H = log V - sigma^2/2 + O(sigma^3, V^-1/2)
    rng = np.random.default_rng(1)
    V, sigma = 400000, 0.1
    z = rng.standard_normal(V) * sigma
    assert abs(oracle.entropy(z) - (math.log(V) - sigma**2 / 2)) < 5e-4


def test_logits_match_torch_linear_and_widening():
    rng = np.random.default_rng(2)
    R, H, V = 3, 40, 70
    h = rng.standard_normal((R, H))
    w32 = rng.standard_normal((V, H)).astype(np.float32)
    z = oracle.logits(h, w32, "f32", vocab_chunk=16)
    ref = torch.nn.functional.linear(torch.from_numpy(h), torch.from_numpy(w32.astype(np.float64)))
    np.testing.assert_allclose(z, ref.numpy(), atol=1e-12)
    wb = gen.f32_to_bf16_bits(w32)
    zb = oracle.logits(h, wb, "bf16", vocab_chunk=7)
    wt = torch.from_numpy(wb.view(np.int16)).view(torch.bfloat16).double()
    ref = torch.nn.functional.linear(torch.from_numpy(h), wt)
    np.testing.assert_allclose(zb, ref.numpy(), atol=1e-12)


def test_greedy_and_ties():
    z = np.array([0.0, 2.0, -1.0, 2.0, 1.0])
    assert oracle.sample_token(z, None, 0.0) == 1          # tie -> lowest id
    g = np.array([0.0, 0.0, 5.0, 0.5, 0.0])
    assert oracle.sample_token(z, g, 0.0) == 1             # tau 0 ignores noise
    assert oracle.sample_token(z, g, 1.0) == 2             # -1 + 5 = 4
    assert oracle.sample_token(z, g, 0.2) == 3             # 2.1 beats 2.0 and 0
    assert oracle.sample_token(z, np.zeros(5), 1.0) == 1   # g = 0 -> argmax


@pytest.mark.parametrize("tau", [1.0, 0.5])
def test_gumbel_max_is_softmax_sampling(tau):
    """argmax(z + tau g) ~ softmax(z / tau): chi-square test on V = 8."""
    V, n = 8, 40000
    z = np.array([0.3, -1.0, 2.0, 0.0, 1.1, -0.4, 0.7, 1.5])
    g = gen.gumbel_f32((n, V), 0, "pin", "gumbel_chi2", int(tau * 10)).astype(np.float64)
    counts = np.bincount([oracle.sample_token(z, g[t], tau) for t in range(n)], minlength=V)
    p = np.exp(z / tau - (z / tau).max())
    p /= p.sum()
    chi2, pval = scipy.stats.chisquare(counts, p * n)
    assert pval > 1e-4, (chi2, pval, counts, p * n)


def test_head_entropy_sample_rows_and_unmasked():
    w = gen.shrink(gen.WORKLOADS["tiny_f32"], vocab=64, hidden=16)
    d = gen.step_inputs(w, seed=3)
    h = oracle.widen(d["hidden"], w.dtype)
    ent, tok, zs = oracle.head_entropy_sample(h, d["w"], w.dtype, d["masked"], d["gumbel"], 1.0)
    for b in range(w.batch):
        for i in range(w.block_k):
            if d["masked"][b, i]:
                z = h[b, i] @ oracle.widen(d["w"], w.dtype).T
                assert abs(ent[b, i] - oracle.entropy(z)) < 1e-12
                assert tok[b, i] == int(np.argmax(z + d["gumbel"][b, i].astype(np.float64)))
            else:
                assert ent[b, i] == np.inf and tok[b, i] == -1


def test_noise_dominates_at_large_tau():
    """argmax(z + tau g): for tau far above the logit range the sampled token
    is the argmax of the noise alone, which pins that tau scales the noise,
    not the logits."""
    rng = np.random.default_rng(3)
    z = rng.standard_normal(50)
    for t in range(20):
        g = rng.gumbel(size=50)
        assert oracle.sample_token(z, g, 1e9) == int(np.argmax(g))
