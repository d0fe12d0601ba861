"""Pins of the oracle's entropy-bounded (EB) selection (CPU only).

The main pin is a brute force over every subset A of the masked positions
using the general form of the EB bound (Appendix B, Eq. 9):
    s* = max { |A| : sum_{i in A} H_i - max_{i in A} H_i <= gamma },
which for the entropy proxy equals Eq. 3; plus hand-worked cases and the
invariants of the rule (at least one unmask, monotone in gamma, ...)."""
import itertools

import numpy as np
import pytest

import oracle

GAMMA_GRID = [0.0, 0.01, 0.1, 0.2, 0.4, 0.8, 1.5]       # Fig. 5 ablation grid


def _brute_force_s(H, gamma):
    n = len(H)
    best = 0
    for size in range(1, n + 1):
        for A in itertools.combinations(range(n), size):
            # sum minus the max = the sum of the others; summed ascending so
            # that values on a decimal grid round as in a prefix sum
            vals = sorted(H[a] for a in A)
            rest = 0.0
            for v in vals[:-1]:
                rest += v
            if rest <= gamma:
                best = max(best, size)
    return best


def _select_one(H, gamma, masked=None):
    k = len(H)
    if masked is None:
        masked = np.ones(k, dtype=np.uint8)
    ent = np.where(masked.astype(bool), np.asarray(H, dtype=np.float64), np.inf)[None, :]
    tok = (np.arange(k, dtype=np.int32) + 100)[None, :]
    bt = np.where(masked.astype(bool), -1, np.arange(k) + 500).astype(np.int32)[None, :]
    nm, nbt, nun, acc, order = oracle.eb_select(ent, tok, masked[None, :], bt, gamma)
    return nm[0], nbt[0], int(nun[0]), acc[0], order[0]


def test_worked_example():
    # H sorted: 0.01, 0.02, 0.5, 3.0; S_1 = 0.01, S_2 = 0.03 <= 0.1, S_3 = 0.53 > 0.1
    nm, nbt, s, acc, _ = _select_one([0.5, 0.01, 3.0, 0.02], 0.1)
    assert s == 3 and acc == {0, 1, 3}
    assert list(nm) == [0, 0, 1, 0]
    assert list(nbt) == [100, 101, -1, 103]


@pytest.mark.parametrize("gamma", GAMMA_GRID)
def test_brute_force_subsets(gamma):
    rng = np.random.default_rng(int(gamma * 1000) + 1)
    for trial in range(150):
        n = int(rng.integers(1, 10))
        kind = trial % 3
        if kind == 0:
            H = rng.exponential(0.1, n)
        elif kind == 1:
            H = rng.uniform(0, 1.0, n)
        else:
            H = np.round(rng.uniform(0, 0.5, n), 1)          # many ties
        s = oracle.eb_accept_count(sorted(H), gamma)
        assert s == _brute_force_s(list(H), gamma), (H, gamma)
        _, _, s2, acc, _ = _select_one(H, gamma)
        assert s2 == s
        # accepted set is an entropy-lower set
        rej = set(range(n)) - acc
        if rej:
            assert max(H[a] for a in acc) <= min(H[r] for r in rej)


def test_at_least_one_and_monotone_in_gamma():
    rng = np.random.default_rng(5)
    for _ in range(200):
        n = int(rng.integers(1, 17))
        H = rng.exponential(0.3, n)
        prev = 0
        for gamma in GAMMA_GRID + [3.0, 100.0]:
            s = oracle.eb_accept_count(sorted(H), gamma)
            assert 1 <= s <= n
            assert s >= prev
            prev = s
        all_but_max = 0.0
        for v in np.sort(H)[:-1]:
            all_but_max += float(v)
        assert oracle.eb_accept_count(sorted(H), all_but_max) == n


def test_gamma_zero_unmasks_the_argmin_when_all_positive():
    rng = np.random.default_rng(8)
    for _ in range(50):
        H = rng.uniform(0.01, 5, 12)
        _, _, s, acc, _ = _select_one(H, 0.0)
        assert s == 1 and acc == {int(np.argmin(H))}


def test_gamma_zero_literal_reading_with_zero_entropy():
    # <= as printed: a zero-entropy first position lets the second through
    _, _, s, acc, _ = _select_one([0.7, 0.0, 0.3], 0.0)
    assert s == 2 and acc == {1, 2}


def test_ties_ordered_by_position():
    _, _, s, acc, order = _select_one([0.4, 0.2, 0.2, 0.2], 0.25)
    assert order == [1, 2, 3, 0]
    assert s == 2 and acc == {1, 2}


def test_only_masked_positions_are_considered():
    masked = np.array([1, 0, 1, 0, 1], dtype=np.uint8)
    nm, nbt, s, acc, order = _select_one([0.9, 0.0, 0.5, 0.0, 0.1], 0.2, masked)
    assert order == [4, 2, 0]
    assert s == 2 and acc == {4, 2}
    assert list(nm) == [1, 0, 0, 0, 0]
    assert list(nbt) == [-1, 501, 102, 503, 104]


def test_empty_mask_is_noop():
    masked = np.zeros(4, dtype=np.uint8)
    nm, nbt, s, acc, _ = _select_one([0.1] * 4, 0.5, masked)
    assert s == 0 and acc == set() and not nm.any()
    assert list(nbt) == [500, 501, 502, 503]


def test_steps_per_block_bounds():
    """Iterating the rule to an empty mask takes between 1 and |M| steps."""
    rng = np.random.default_rng(12)
    for _ in range(100):
        k = int(rng.integers(1, 33))
        masked = np.ones((1, k), dtype=np.uint8)
        bt = np.full((1, k), -1, dtype=np.int32)
        steps = 0
        while masked.any():
            ent = np.where(masked.astype(bool), rng.exponential(0.2, (1, k)), np.inf)
            tok = rng.integers(0, 1000, (1, k)).astype(np.int32)
            masked, bt, n_un, _, _ = oracle.eb_select(ent, tok, masked, bt, 0.1)
            assert n_un[0] >= 1
            steps += 1
        assert 1 <= steps <= k
        assert (bt >= 0).all()


# ------------------------------------------------------ margins to gamma

def test_prefix_margins_worked_example():
    """Sorted H = 0.01, 0.02, 0.5, 3.0 at gamma = 0.1: the decision on rank
    j >= 2 compares S_{j-1} (the sum of the j-1 smallest) with gamma, so the
    margins are |0.01 - 0.1|, |0.03 - 0.1|, |0.53 - 0.1| (by hand)."""
    m = oracle.eb_prefix_margins([0.01, 0.02, 0.5, 3.0], 0.1)
    assert np.allclose(m, [0.09, 0.07, 0.43], rtol=0, atol=1e-15)
    # S_j and S_{j-1} differ: with S_j the first margin would be 0.07
    m2 = oracle.eb_prefix_margins([0.2, 0.05], 0.1)
    assert np.allclose(m2, [0.1], rtol=0, atol=1e-15)
    assert oracle.eb_prefix_margins([0.7], 0.1) == []
    assert oracle.eb_prefix_margins([], 0.1) == []


def test_prefix_margins_equal_brute_force_thresholds():
    """The margin of rank j is the distance from gamma to the smallest gamma
    at which Eq. 9's bound admits j positions: min over subsets A with
    |A| = j of (sum_A H - max_A H), found by enumeration."""
    rng = np.random.default_rng(31)
    for trial in range(60):
        n = int(rng.integers(1, 8))
        H = sorted(rng.exponential(0.2, n).tolist())
        gamma = float(rng.choice(GAMMA_GRID))
        m = oracle.eb_prefix_margins(H, gamma)
        assert len(m) == max(0, n - 1)
        for j in range(2, n + 1):
            thr = min(sum(sorted(H[a] for a in A)[:-1])
                      for A in itertools.combinations(range(n), j))
            assert abs(m[j - 2] - abs(thr - gamma)) <= 1e-12, (H, gamma, j)


def test_prefix_margins_locate_the_decision():
    """Each margin is how far gamma may move before the accept count of
    Eq. 3 changes at that rank: for rank j one of gamma +- margin is the
    threshold c where eb_accept_count first admits j positions (admits j
    just above c, fewer just below; "just" is 1e-12, far below the gaps
    between prefix sums and above the rounding of gamma +- margin)."""
    rng = np.random.default_rng(32)
    for _ in range(80):
        n = int(rng.integers(2, 10))
        H = sorted(rng.exponential(0.15, n).tolist())
        gamma = float(rng.uniform(0.0, 0.6))
        m = oracle.eb_prefix_margins(H, gamma)
        for j in range(2, n + 1):
            hits = 0
            for c in (gamma + m[j - 2], gamma - m[j - 2]):
                if c < 0.0:
                    continue
                if (oracle.eb_accept_count(H, c + 1e-12) >= j
                        and oracle.eb_accept_count(H, c - 1e-12) < j):
                    hits += 1
            assert hits >= 1, (H, gamma, j, m)
