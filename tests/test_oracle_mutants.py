"""Planted mistakes in the oracle must be caught by its pins (CPU only).

Each mutant is the oracle with one plausible mistake (a dropped term, a wrong
index, a wrong sign or inequality); the test runs the pins of the other
oracle test files against it through monkeypatch and asserts that at least
one of them fails."""
import numpy as np
import pytest

import oracle
import oracle.sbd_oracle as so
from tests import test_oracle_attention as TA
from tests import test_oracle_eb as TE
from tests import test_oracle_head as TH


def _fails(fn, *args):
    try:
        fn(*args)
    except AssertionError:
        return True
    return False


# ---------------------------------------------------------------- attention

def _attn_drop_block(q, k_cache, v_cache, cache_len, k_blk, v_blk, scale=None):
    B, k, Hq, D = q.shape
    G = Hq // k_cache.shape[2]
    scale = 1.0 / np.sqrt(D) if scale is None else scale
    out = np.zeros_like(q)
    for b in range(B):
        L = int(cache_len[b])
        for hq in range(Hq):
            hk = hq // G
            keys = np.concatenate([k_cache[b, :L, hk], k_blk[b, :1, hk]])   # only one block key
            vals = np.concatenate([v_cache[b, :L, hk], v_blk[b, :1, hk]])
            s = q[b, :, hq] @ keys.T * scale
            p = np.exp(s - s.max(axis=1, keepdims=True))
            out[b, :, hq] = (p / p.sum(axis=1, keepdims=True)) @ vals
    return out


def _attn_mutant(scale_fn=None, head_fn=None):
    def f(q, k_cache, v_cache, cache_len, k_blk, v_blk, scale=None):
        B, k, Hq, D = q.shape
        Hkv = k_cache.shape[2]
        G = Hq // Hkv
        sc = (scale_fn(D) if scale_fn else 1.0 / np.sqrt(D)) if scale is None else scale
        out = np.zeros_like(q)
        for b in range(B):
            L = int(cache_len[b])
            for hq in range(Hq):
                hk = head_fn(hq, G, Hkv) if head_fn else hq // G
                keys = np.concatenate([k_cache[b, :L, hk], k_blk[b, :, hk]])
                vals = np.concatenate([v_cache[b, :L, hk], v_blk[b, :, hk]])
                s = q[b, :, hq] @ keys.T * sc
                p = np.exp(s - s.max(axis=1, keepdims=True))
                out[b, :, hq] = (p / p.sum(axis=1, keepdims=True)) @ vals
        return out
    return f


ATTN_PINS = [
    (TA.test_block_attention_equals_explicit_mask, (3, 4, 4, 2)),
    (TA.test_k1_is_plain_causal_decode_sdpa, (8, 2)),
    (TA.test_zero_query_is_uniform_average, ()),
]


@pytest.mark.parametrize("mutant", [
    _attn_drop_block,
    _attn_mutant(scale_fn=lambda D: 1.0 / D),
    _attn_mutant(head_fn=lambda hq, G, Hkv: hq % Hkv),
])
def test_attention_mutants_are_caught(monkeypatch, mutant):
    monkeypatch.setattr(oracle, "block_attention", mutant)
    assert any(_fails(fn, *args) for fn, args in ATTN_PINS)


# ---------------------------------------------------------------- entropy

def _entropy_no_logz(z_row):
    z = np.asarray(z_row, dtype=np.float64)
    m = z.max()
    e = np.exp(z - m)
    p = e / e.sum()
    return float((-p * (z - m)).sum())          # dropped the log Z term


def _entropy_wrong_sign(z_row):
    return -so.entropy(z_row)


HEAD_PINS = [
    (TH.test_uniform_logits_entropy_is_log_v, (512,)),
    (TH.test_two_point_binary_entropy, (1.0, -0.5)),
    (TH.test_entropy_matches_scipy_and_is_shift_invariant, ()),
]


@pytest.mark.parametrize("mutant", [_entropy_no_logz, _entropy_wrong_sign])
def test_entropy_mutants_are_caught(monkeypatch, mutant):
    monkeypatch.setattr(oracle, "entropy", mutant)
    assert any(_fails(fn, *args) for fn, args in HEAD_PINS)


def _token_ignores_tau(z_row, g_row, tau):
    z = np.asarray(z_row, dtype=np.float64)
    if g_row is None:
        return int(np.argmax(z))
    return int(np.argmax(z + np.asarray(g_row, dtype=np.float64)))


def _token_last_tie(z_row, g_row, tau):
    z = np.asarray(z_row, dtype=np.float64)
    score = z if (tau == 0.0 or g_row is None) else z + tau * np.asarray(g_row)
    return int(len(score) - 1 - np.argmax(score[::-1]))


@pytest.mark.parametrize("mutant", [_token_ignores_tau, _token_last_tie])
def test_token_mutants_are_caught(monkeypatch, mutant):
    monkeypatch.setattr(oracle, "sample_token", mutant)
    pins = [(TH.test_greedy_and_ties, ()), (TH.test_gumbel_max_is_softmax_sampling, (0.5,))]
    assert any(_fails(fn, *args) for fn, args in pins)


# ---------------------------------------------------------------- EB rule

def _eb_strict(sorted_entropies, gamma):
    n = len(sorted_entropies)
    if n == 0:
        return 0
    s, prefix = 1, 0.0
    for j in range(1, n):
        prefix += float(sorted_entropies[j - 1])
        if prefix < gamma:                     # < instead of <=
            s = j + 1
        else:
            break
    return s


def _eb_includes_own(sorted_entropies, gamma):
    n = len(sorted_entropies)
    if n == 0:
        return 0
    s, prefix = 1, float(sorted_entropies[0])
    for j in range(1, n):
        prefix += float(sorted_entropies[j])   # S_s instead of S_{s-1}
        if prefix <= gamma:
            s = j + 1
        else:
            break
    return s


@pytest.mark.parametrize("mutant", [_eb_strict, _eb_includes_own])
def test_eb_mutants_are_caught(monkeypatch, mutant):
    monkeypatch.setattr(so, "eb_accept_count", mutant)
    monkeypatch.setattr(oracle, "eb_accept_count", mutant)
    pins = [(TE.test_worked_example, ()), (TE.test_gamma_zero_literal_reading_with_zero_entropy, ()),
            (TE.test_brute_force_subsets, (0.1,))]
    assert any(_fails(fn, *args) for fn, args in pins)


def test_eb_descending_sort_is_caught(monkeypatch):
    real = so.eb_select

    def desc(entropy_bk, token_bk, masked_bk, block_tokens_bk, gamma):
        return real(-np.where(np.isfinite(entropy_bk), entropy_bk, -np.inf), token_bk,
                    masked_bk, block_tokens_bk, gamma)

    monkeypatch.setattr(oracle, "eb_select", desc)
    pins = [(TE.test_worked_example, ()), (TE.test_ties_ordered_by_position, ())]
    assert any(_fails(fn, *args) for fn, args in pins)


# ------------------------------------------------- confidence and other rules
from tests import test_oracle_select as TS   # noqa: E402


def _patch(monkeypatch, name, fn):
    monkeypatch.setattr(so, name, fn)
    monkeypatch.setattr(oracle, name, fn)


def _conf_mean_shift(z_row):
    z = np.asarray(z_row, dtype=np.float64)
    return float(1.0 / np.exp(z - z.mean()).sum())   # the mean subtracted, not the max


def _conf_without_shift(z_row):
    z = np.asarray(z_row, dtype=np.float64)
    return float(1.0 / np.exp(z).sum())            # max subtracted nowhere


@pytest.mark.parametrize("mutant", [_conf_mean_shift, _conf_without_shift])
def test_confidence_mutants_are_caught(monkeypatch, mutant):
    _patch(monkeypatch, "confidence", mutant)
    pins = [(TS.test_uniform_logits_confidence_is_one_over_v, (7,)),
            (TS.test_two_point_confidence_is_logistic, (1.0, -1.0)),
            (TS.test_confidence_matches_softmax_and_bounds_entropy, ())]
    assert any(_fails(fn, *args) for fn, args in pins)


def _general_without_max(H_in_order, gamma):
    n = len(H_in_order)
    if n == 0:
        return 0
    s, total = 1, float(H_in_order[0])
    for j in range(1, n):
        total += float(H_in_order[j])
        if total <= gamma:                         # the max term dropped
            s = j + 1
        else:
            break
    return s


def _general_exclusive_prefix(H_in_order, gamma):
    n = len(H_in_order)
    if n == 0:
        return 0
    s, prefix = 1, 0.0
    for j in range(1, n):
        prefix += float(H_in_order[j - 1])         # Eq. 3's sum, in a non-sorted order
        if prefix <= gamma:
            s = j + 1
        else:
            break
    return s


@pytest.mark.parametrize("mutant", [_general_without_max, _general_exclusive_prefix])
def test_general_bound_mutants_are_caught(monkeypatch, mutant):
    _patch(monkeypatch, "eb_general_accept_count", mutant)
    pins = [(TS.test_confidence_proxy_worked_example, ()), (TS.test_running_max_matters, ()),
            (TS.test_general_bound_invariants, ())]
    assert any(_fails(fn, *args) for fn, args in pins)


def _factor_off_by_one(confidences_desc, f, complement=False):
    n_m = len(confidences_desc)
    if n_m == 0:
        return 0
    best = 1
    for n in range(1, n_m + 1):
        c = float(confidences_desc[n - 1])
        if n * ((1.0 - c) if complement else c) < f:   # n instead of n + 1
            best = n
    return best


def _factor_first_failure(confidences_desc, f, complement=False):
    n_m = len(confidences_desc)
    if n_m == 0:
        return 0
    best = 1
    for n in range(1, n_m + 1):
        c = float(confidences_desc[n - 1])
        if (n + 1) * ((1.0 - c) if complement else c) < f:
            best = n
        else:
            break                                   # stops at the first failing count
    return best


@pytest.mark.parametrize("mutant", [_factor_off_by_one, _factor_first_failure])
def test_factor_mutants_are_caught(monkeypatch, mutant):
    _patch(monkeypatch, "factor_accept_count", mutant)
    pins = [(TS.test_factor_worked_examples, ()),
            (TS.test_factor_constant_confidence_closed_form, (0.3, 1.0))]
    assert any(_fails(fn, *args) for fn, args in pins)


def test_ascending_confidence_order_is_caught(monkeypatch):
    real = so.select_step

    def asc(entropy_bk, confidence_bk, token_bk, masked_bk, block_tokens_bk, rule, thr):
        return real(entropy_bk, -np.asarray(confidence_bk), token_bk, masked_bk,
                    block_tokens_bk, rule, thr)

    monkeypatch.setattr(oracle, "select_step", asc)
    pins = [(TS.test_confidence_proxy_worked_example, ()),
            (TS.test_factor_select_takes_a_confidence_prefix, ())]
    assert any(_fails(fn, *args) for fn, args in pins)


# ------------------------------------------------ causal prefix rows (first iteration)

def _prefix_mutant(shift):
    """block_attention whose causal rows see block keys j <= i + shift."""
    def f(q, k_cache, v_cache, cache_len, k_blk, v_blk, scale=None, n_causal=0):
        B, k, Hq, D = q.shape
        G = Hq // k_cache.shape[2]
        sc = 1.0 / np.sqrt(D) if scale is None else scale
        out = np.zeros_like(q)
        for b in range(B):
            L = int(cache_len[b])
            for hq in range(Hq):
                hk = hq // G
                keys = np.concatenate([k_cache[b, :L, hk], k_blk[b, :, hk]])
                vals = np.concatenate([v_cache[b, :L, hk], v_blk[b, :, hk]])
                s = q[b, :, hq] @ keys.T * sc
                for i in range(min(n_causal, k)):
                    s[i, max(L + i + 1 + shift, L + 1):] = -np.inf
                p = np.exp(s - s.max(axis=1, keepdims=True))
                out[b, :, hq] = (p / p.sum(axis=1, keepdims=True)) @ vals
        return out
    return f


def _prefix_ignored(q, k_cache, v_cache, cache_len, k_blk, v_blk, scale=None, n_causal=0):
    return so.block_attention(q, k_cache, v_cache, cache_len, k_blk, v_blk, scale)


@pytest.mark.parametrize("mutant", [_prefix_mutant(-1), _prefix_mutant(1), _prefix_ignored])
def test_causal_prefix_mutants_are_caught(monkeypatch, mutant):
    monkeypatch.setattr(oracle, "block_attention", mutant)
    pins = [(TA.test_causal_prefix_rows_equal_explicit_mask, (4, 2, 5)),
            (TA.test_all_causal_block_is_torch_causal_prefill, ())]
    assert all(_fails(fn, *args) for fn, args in pins)


# ------------------------------------------------------- timing model
from tests import test_oracle_roofline as TR   # noqa: E402


def _speedup_no_first_forward(k, l, time_fn):
    return k * time_fn(1) / (l * time_fn(k))                   # first forward of k rows, not 2k


def _attention_one_contraction(block, kv_len, batch, c=so.ROOFLINE_H100):
    tokens = block * batch
    width = c["n_heads"] * c["head_dim"]
    mem = (2 * tokens * width * c["bytes_per_el"]
           + 2 * batch * kv_len * c["n_kv_heads"] * c["head_dim"] * c["kv_bytes"])
    flops = so.roofline_gemm(tokens, kv_len, width, c)[1]      # PV dropped
    return max(mem / c["bandwidth"], flops / c["peak_flops_attention"])


def _linear_corrected_shapes(block, batch, c=so.ROOFLINE_H100):
    t, h, f = block * batch, c["hidden"], c["ffn"]
    shapes = [(t, f, h), (t, h, f), (t, h, h), (t, 1024, h), (t, 1024, h), (t, h, h)]
    return sum(so.roofline_gemm(m, n, k, c)[0] for (m, n, k) in shapes)


@pytest.mark.parametrize("name,mutant", [("sbd_speedup", _speedup_no_first_forward),
                                         ("roofline_attention", _attention_one_contraction),
                                         ("roofline_linear", _linear_corrected_shapes)])
def test_timing_model_mutants_are_caught(monkeypatch, name, mutant):
    _patch(monkeypatch, name, mutant)
    assert _fails(TR.test_every_printed_cell)


# ------------------------------------------------------ EB margins to gamma

def _margins_own_term(entropy_row_sorted, gamma):
    out, prefix = [], 0.0
    for j in range(1, len(entropy_row_sorted)):
        prefix += float(entropy_row_sorted[j])      # S_j instead of S_{j-1}
        out.append(abs(prefix - gamma))
    return out


def _margins_shifted(entropy_row_sorted, gamma):
    out, prefix = [], 0.0
    for j in range(len(entropy_row_sorted)):          # ranks start at 1, not 2
        if j:
            prefix += float(entropy_row_sorted[j - 1])
        out.append(abs(prefix - gamma))
    return out[:-1]


def _margins_signed(entropy_row_sorted, gamma):
    out, prefix = [], 0.0
    for j in range(1, len(entropy_row_sorted)):
        prefix += float(entropy_row_sorted[j - 1])
        out.append(prefix - gamma)                   # no absolute value
    return out


@pytest.mark.parametrize("mutant", [_margins_own_term, _margins_shifted, _margins_signed])
def test_margin_mutants_are_caught(monkeypatch, mutant):
    _patch(monkeypatch, "eb_prefix_margins", mutant)
    pins = [(TE.test_prefix_margins_worked_example, ()),
            (TE.test_prefix_margins_equal_brute_force_thresholds, ()),
            (TE.test_prefix_margins_locate_the_decision, ())]
    assert all(_fails(fn, *args) for fn, args in pins[:2])
