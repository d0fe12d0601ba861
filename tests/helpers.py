"""Shared helpers of the test suite: device transfer of generator arrays,
cached full-size inputs, and the comparison rules of the parity tests."""
from __future__ import annotations

import functools
import math

import numpy as np

import gen
import oracle

F32_ATTN_TOL = 1e-5      # max-abs, fp32 inputs
BF16_ATTN_TOL = 2e-2     # max-abs, bf16 inputs with fp32 accumulation
ENTROPY_TOL = 1e-3       # nats
GAMMA_MARGIN = 1e-4      # oracle margin |S_{j-1} - gamma| below which a decision is exempt


def to_dev(x: np.ndarray, dtype: str, device="cuda"):
    import torch
    x = np.ascontiguousarray(x)
    if dtype == "bf16":
        return torch.from_numpy(x.view(np.int16)).view(torch.bfloat16).to(device)
    return torch.from_numpy(x).to(device)


@functools.lru_cache(maxsize=2)
def cached_weight(vocab: int, hidden: int, dtype: str, seed: int = 0):
    w = gen.shrink(gen.WORKLOADS["llama8b_k16"], vocab=vocab, hidden=hidden, dtype=dtype)
    return gen.lm_head_weight(w, seed)


def step_inputs(w: gen.Workload, seed: int, step: int = 0):
    d = gen.attention_inputs(w, seed, 0, poison_tail=True)
    d["w"] = cached_weight(w.vocab, w.hidden, w.dtype, seed)
    d["hidden"] = gen.hidden_states(w, seed, step)
    d["gumbel"] = gen.gumbel_noise(w, seed, step)
    bt, m = gen.block_state(w, seed)
    d["block_tokens"] = bt
    d["masked"] = m
    return d


def token_tolerance(z_row: np.ndarray, accumulations: int) -> float:
    """Score gap below which the top-1 and top-2 tokens are a tie at the
    kernel's precision: `accumulations` fp32 additions of partial sums whose
    magnitude is bounded by max |z| (2^-23 relative each)."""
    return max(1e-6, accumulations * 2.0 ** -23 * float(np.abs(z_row).max()))


def top2_gap(z_row: np.ndarray, g_row, tau: float) -> float:
    score = z_row if (tau == 0.0 or g_row is None) else z_row + tau * np.asarray(g_row, np.float64)
    top = np.partition(score, -2)[-2:]
    return float(top[1] - top[0])


def compare_unmask(masked_before, ent_ref, gamma, masked_after_gpu, tie_tol=0.0):
    """Unmask sets: the GPU's accepted set must equal the oracle's EB set,
    except (i) at a rank j >= 2 whose oracle margin |S_{j-1} - gamma| is
    below GAMMA_MARGIN (+ the entropy tolerance accumulated over the j-1
    summands when the GPU used its own entropies), or (ii) between positions
    whose oracle entropies differ by less than tie_tol (an order tie).
    Returns the number of exempted sequences; raises AssertionError on a
    real mismatch."""
    B, k = masked_before.shape
    gamma = float(np.float32(gamma))          # the threshold the kernel receives
    exempt = 0
    for b in range(B):
        M = [i for i in range(k) if masked_before[b, i]]
        order = sorted(M, key=lambda i: (float(ent_ref[b, i]), i))
        s_ref = oracle.eb_accept_count([ent_ref[b, i] for i in order], gamma)
        ref_set = set(order[:s_ref])
        got = {i for i in M if not masked_after_gpu[b, i]}
        if got == ref_set:
            continue
        s_got = len(got)
        ok = s_got >= (1 if M else 0)
        # (ii) the GPU set must still be a prefix of an order consistent
        # with the oracle entropies up to tie_tol
        if ok and got:
            hi = max(float(ent_ref[b, i]) for i in got)
            rest = [float(ent_ref[b, i]) for i in M if i not in got]
            ok = not rest or hi <= min(rest) + tie_tol
        # (i) every rank between the two counts is a margin case
        if ok:
            sorted_h = sorted(float(ent_ref[b, i]) for i in M)
            lo, hi_s = sorted((s_got, s_ref))
            prefix = 0.0
            for j in range(1, len(sorted_h)):
                prefix += sorted_h[j - 1]
                rank = j + 1
                if lo < rank <= hi_s:
                    if abs(prefix - gamma) >= GAMMA_MARGIN + (rank - 1) * tie_tol / 2:
                        ok = False
        assert ok, (b, sorted(got), sorted(ref_set), [float(ent_ref[b, i]) for i in order], gamma)
        exempt += 1
    return exempt
