"""Pins of the oracle's confidence and of the other selection rules (CPU only).

Appendix "Sampling algorithm" of arXiv 2509.04185: the EB-Sampler with the
confidence error proxy (general EB bound) and the Factor rule.  Pinned by
closed forms of the confidence, by the identity of the general bound with
Eq. 3 under the entropy order, by a brute force over every subset, by
hand-worked cases whose arithmetic is written out below, and by the rules'
invariants."""
import itertools
import math

import numpy as np
import pytest
from scipy.special import softmax

import oracle

GAMMA_GRID = [0.0, 0.01, 0.1, 0.2, 0.4, 0.8, 1.5]


# ------------------------------------------------------------- confidence

@pytest.mark.parametrize("V", [1, 7, 512, 128256])
def test_uniform_logits_confidence_is_one_over_v(V):
    assert oracle.confidence(np.full(V, 0.37)) == pytest.approx(1.0 / V, rel=1e-12)


def test_one_hot_confidence_is_one():
    z = np.zeros(1000)
    z[3] = 1e4
    assert oracle.confidence(z) == 1.0


@pytest.mark.parametrize("a,b", [(0.0, 0.0), (1.0, -1.0), (-3.0, 2.5), (10.0, 9.99)])
def test_two_point_confidence_is_logistic(a, b):
    # max(p, 1 - p) with p = 1 / (1 + e^(b - a)): the logistic of |a - b|
    assert oracle.confidence(np.array([a, b])) == pytest.approx(
        1.0 / (1.0 + math.exp(-abs(a - b))), rel=1e-12)


def test_confidence_matches_softmax_and_bounds_entropy():
    rng = np.random.default_rng(11)
    for _ in range(50):
        V = int(rng.integers(2, 3000))
        z = rng.normal(0.0, float(rng.uniform(0.1, 8.0)), V) + float(rng.normal(0, 50))
        c = oracle.confidence(z)
        assert c == pytest.approx(float(softmax(z).max()), rel=1e-12)
        assert 1.0 / V - 1e-15 <= c <= 1.0
        # min-entropy <= Shannon entropy <= log V
        H = oracle.entropy(z)
        assert -math.log(c) <= H + 1e-12
        assert H <= math.log(V) + 1e-12


def test_head_returns_confidence_of_masked_rows():
    rng = np.random.default_rng(3)
    B, k, H, V = 2, 3, 8, 50
    hid = rng.normal(0, 1, (B, k, H))
    w = rng.normal(0, 1, (V, H)).astype(np.float32)
    masked = np.array([[1, 0, 1], [0, 1, 1]], dtype=np.uint8)
    ent, tok, zs, conf = oracle.head_entropy_sample(hid, w, "f32", masked, None, 0.0,
                                                    with_confidence=True)
    for b in range(B):
        for i in range(k):
            if masked[b, i]:
                z = hid[b, i] @ w.astype(np.float64).T
                assert conf[b, i] == pytest.approx(float(softmax(z).max()), rel=1e-12)
            else:
                assert conf[b, i] == 0.0


# ------------------------------------------------------- general EB bound

def _brute_force_general(H, gamma):
    """max |A| over every subset A with sum_A H - max_A H <= gamma."""
    best = 0
    for size in range(1, len(H) + 1):
        for A in itertools.combinations(range(len(H)), size):
            vals = sorted(H[a] for a in A)
            rest = 0.0
            for v in vals[:-1]:
                rest += v
            if rest <= gamma:
                best = max(best, size)
    return best


def test_general_bound_under_entropy_order_is_eq3():
    rng = np.random.default_rng(21)
    for _ in range(400):
        n = int(rng.integers(1, 17))
        H = rng.exponential(float(rng.uniform(0.01, 1.0)), n)
        gamma = float(rng.uniform(0.0, 1.0))
        asc = sorted(H)
        assert oracle.eb_general_accept_count(asc, gamma) == oracle.eb_accept_count(asc, gamma)


@pytest.mark.parametrize("gamma", GAMMA_GRID)
def test_confidence_order_against_brute_force(gamma):
    rng = np.random.default_rng(int(gamma * 1000) + 7)
    for _ in range(150):
        n = int(rng.integers(1, 10))
        H = rng.exponential(0.15, n)
        # any order is a candidate subset family: never above the brute force
        order = rng.permutation(n)
        s = oracle.eb_general_accept_count([H[i] for i in order], gamma)
        assert 1 <= s <= _brute_force_general(list(H), gamma)
        # confidences decreasing in entropy: the confidence order is the
        # ascending-entropy order and the prefix reaches the brute force
        conf = np.exp(-H)
        conf_order = sorted(range(n), key=lambda i: (-conf[i], i))
        s2 = oracle.eb_general_accept_count([H[i] for i in conf_order], gamma)
        assert s2 == _brute_force_general(list(H), gamma)


def _select(rule, H, C, thr, masked=None):
    k = len(H)
    if masked is None:
        masked = np.ones(k, dtype=np.uint8)
    mk = masked.astype(bool)
    ent = np.where(mk, np.asarray(H, dtype=np.float64), np.inf)[None, :]
    conf = np.where(mk, np.asarray(C, dtype=np.float64), 0.0)[None, :]
    tok = (np.arange(k, dtype=np.int32) + 100)[None, :]
    bt = np.where(mk, -1, np.arange(k) + 500).astype(np.int32)[None, :]
    nm, nbt, nun, acc, order = oracle.select_step(ent, conf, tok, masked[None, :], bt, rule, thr)
    return nm[0], nbt[0], int(nun[0]), acc[0], order[0]


def test_confidence_proxy_worked_example():
    # confidence order: pos 3 (0.99), 0 (0.9), 2 (0.8), 1 (0.5); entropies in
    # that order 0.05, 0.2, 0.5, 2.0.  Sum minus max of the prefixes:
    #   s=1: 0;  s=2: 0.25 - 0.2 = 0.05;  s=3: 0.75 - 0.5 = 0.25;  s=4: 2.75 - 2.0 = 0.75
    H = [0.2, 2.0, 0.5, 0.05]
    C = [0.9, 0.5, 0.8, 0.99]
    for gamma, s_exp, acc_exp in ((0.3, 3, {3, 0, 2}), (0.2, 2, {3, 0}), (0.0, 1, {3}),
                                  (0.75, 4, {0, 1, 2, 3})):
        nm, nbt, s, acc, order = _select("eb_confidence", H, C, gamma)
        assert order == [3, 0, 2, 1]
        assert s == s_exp and acc == acc_exp, gamma
        for i in range(4):
            assert nm[i] == (0 if i in acc_exp else 1)
            assert nbt[i] == (100 + i if i in acc_exp else -1)


def test_running_max_matters():
    # entropies in confidence order 1.0, 0.1, 0.1 with gamma = 0.25:
    # s=2: 1.1 - 1.0 = 0.1;  s=3: 1.2 - 1.0 = 0.2 -> all three (the sum of the
    # ones before the last, 1.0 and 1.1, would stop at s = 1)
    assert oracle.eb_general_accept_count([1.0, 0.1, 0.1], 0.25) == 3


def test_general_bound_invariants():
    rng = np.random.default_rng(8)
    for _ in range(200):
        n = int(rng.integers(1, 17))
        H = list(rng.exponential(0.3, n))
        prev = 0
        for gamma in GAMMA_GRID:
            s = oracle.eb_general_accept_count(H, gamma)
            assert 1 <= s <= n
            assert s >= prev                               # monotone in gamma
            prev = s
        assert oracle.eb_general_accept_count(H, sum(H) - max(H)) == n
        assert oracle.eb_general_accept_count(H, 0.0) == 1  # all H > 0
    assert oracle.eb_general_accept_count([], 0.5) == 0


# ------------------------------------------------------------ Factor rule

def test_factor_worked_examples():
    c = [0.99, 0.9, 0.8, 0.5]                    # already descending
    # (n + 1) c^n for n = 1..4: 1.98, 2.7, 3.2, 2.5
    assert oracle.factor_accept_count(c, 2.0) == 1
    assert oracle.factor_accept_count(c, 2.4) == 1
    assert oracle.factor_accept_count(c, 2.6) == 4   # the last count qualifies again
    assert oracle.factor_accept_count(c, 3.0) == 4
    assert oracle.factor_accept_count(c, 1.5) == 1   # none qualifies: one token
    # complement: (n + 1)(1 - c^n) = 0.02, 0.3, 0.8, 2.5
    assert oracle.factor_accept_count(c, 1.0, complement=True) == 3
    assert oracle.factor_accept_count(c, 0.5, complement=True) == 2
    assert oracle.factor_accept_count(c, 0.01, complement=True) == 1
    assert oracle.factor_accept_count(c, 2.6, complement=True) == 4
    assert oracle.factor_accept_count([], 2.0) == 0


@pytest.mark.parametrize("c,f", [(0.3, 1.0), (0.9, 5.0), (0.05, 0.31), (0.6, 10.0)])
def test_factor_constant_confidence_closed_form(c, f):
    # (n + 1) c < f  <=>  n < f / c - 1: the largest such n is ceil(f / c) - 2
    for n_m in range(1, 20):
        exp_n = min(n_m, max(1, math.ceil(f / c) - 2))
        assert oracle.factor_accept_count([c] * n_m, f) == exp_n
        exp_c = min(n_m, max(1, math.ceil(f / (1.0 - c)) - 2))
        assert oracle.factor_accept_count([c] * n_m, f, complement=True) == exp_c


def test_factor_select_takes_a_confidence_prefix():
    rng = np.random.default_rng(4)
    for _ in range(100):
        k = int(rng.integers(1, 33))
        masked = (rng.uniform(size=k) < 0.7).astype(np.uint8)
        C = rng.uniform(0.0, 1.0, k)
        H = rng.exponential(1.0, k)
        f = float(rng.uniform(0.5, 6.0))
        for rule in ("factor", "factor_complement"):
            nm, nbt, s, acc, order = _select(rule, H, C, f, masked)
            n_m = int(masked.sum())
            assert order == sorted([i for i in range(k) if masked[i]], key=lambda i: (-C[i], i))
            assert s == (0 if n_m == 0 else len(acc)) and acc == set(order[:s])
            assert (n_m == 0 and s == 0) or 1 <= s <= n_m
            assert all(nm[i] == 0 for i in acc)


def test_entropy_rule_of_select_step_is_eb_select():
    rng = np.random.default_rng(9)
    for _ in range(50):
        k = int(rng.integers(1, 33))
        masked = (rng.uniform(size=k) < 0.8).astype(np.uint8)
        H = rng.exponential(0.2, k)
        C = rng.uniform(size=k)
        a = _select("eb_entropy", H, C, 0.1, masked)
        ent = np.where(masked.astype(bool), H, np.inf)[None, :]
        tok = (np.arange(k, dtype=np.int32) + 100)[None, :]
        bt = np.where(masked.astype(bool), -1, np.arange(k) + 500).astype(np.int32)[None, :]
        b = oracle.eb_select(ent, tok, masked[None, :], bt, 0.1)
        assert np.array_equal(a[0], b[0][0]) and a[2] == int(b[2][0]) and a[3] == b[3][0]


def test_unknown_rule_is_rejected():
    with pytest.raises(ValueError):
        _select("top_k", [0.1], [0.5], 1.0)
