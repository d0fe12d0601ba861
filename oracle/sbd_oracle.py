"""fp64 CPU oracle for the Set Block Decoding (SBD) block step.

TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check of the graft entry
point and the CPU-baseline leg of the bench may import or call this module.
The product path (the CUDA library and its Python binding) never does, and it
shares no code with it: this file imports numpy and nothing else of the repo.

Every function is the plain definition written out in float64 over the input
values (bf16 inputs are widened exactly), with library primitives (matmul,
exp, log, sort) as the only helpers and no blocking or fusion beyond what the
definition states.  Each cites the passage of arXiv 2509.04185 it follows.

Readings of points the paper leaves open (each listed in the design notes):
  * softmax scale 1/sqrt(head_dim) unless given;
  * grouped-query heads: query head hq reads KV head hq // (Hq / Hkv);
  * entropy in nats of softmax(z) at temperature 1;
  * sampling is Gumbel-max on z + tau * g (tau = 0: greedy, the paper's
    temperature-0 setting), ties to the lowest vocabulary id;
  * EB rule with the inequality exactly as printed (<=), gamma = 0 allowed,
    equal entropies ordered by block position;
  * confidence c^i = max_v p_v of softmax(z) at temperature 1; confidence
    orders are descending, equal confidences ordered by block position;
  * the first iteration of a block after the previous one carries the
    previous block's tokens as n_causal causal rows ahead of the new block
    (their keys and values then enter the cache); the new block's rows see
    them like the rest of the cache;
  * Factor rule: c^n is the n-th largest confidence, n the largest count in
    1..|M| with (n + 1) c^n < f, and n = 1 when no count qualifies (a step
    unmasks at least one token); the complement reading (n + 1)(1 - c^n) < f
    is provided beside it.

Pins (what each function is checked against, none of it itself) live in
tests/test_oracle_*.py; no function here is "parity unpinned".
"""
from __future__ import annotations

import numpy as np

MASK_TOKEN = -1


# ----------------------------------------------------------------- inputs

def widen(x: np.ndarray, dtype: str) -> np.ndarray:
    """Storage -> float64.  bf16 is stored as its raw 16-bit pattern, which is
    the upper half of the fp32 with the same value, so widening is exact."""
    if dtype == "bf16":
        bits = np.asarray(x, dtype=np.uint16).astype(np.uint32) << 16
        return bits.view(np.float32).astype(np.float64)
    if dtype == "f32":
        return np.asarray(x, dtype=np.float32).astype(np.float64)
    return np.asarray(x, dtype=np.float64)


# ------------------------------------------------------------- attention

def inference_mask_allows(q_idx: int, kv_idx: int, causal_point: int) -> bool:
    """Inference attention mask of the SBD network (Eq. 5 and the inference
    mask of the FlexAttention appendix): a query may see a key when the key is
    not in its future, or when the query lies in the prediction block, which
    starts at causal_point; block queries therefore see every key."""
    return (kv_idx <= q_idx) or (causal_point <= q_idx)


def block_attention(q, k_cache, v_cache, cache_len, k_blk, v_blk, scale=None,
                    n_causal: int = 0):
    """Block attention of one SBD forward (Eq. 5; Fig. 3 mask).

    Block query row i of sequence b attends to the L_b cached keys (the exact
    KV cache of x_<t, causal among themselves and all in the past of the
    block) and to all k block keys (bidirectional inside the block).

    n_causal > 0 is the first iteration of a block after the previous one
    (Algorithm 3, "first iteration and t >= k"): the forward then carries
    the n_causal tokens of the previous block, whose keys and values still
    have to enter the cache, ahead of the new block.  Under the inference
    mask with its causal point at the new block, block row i < n_causal sees
    the cache and block keys j <= i; rows i >= n_causal see every key.

    q [B,k,Hq,D]; k_cache, v_cache [B,Lmax,Hkv,D]; cache_len [B];
    k_blk, v_blk [B,k,Hkv,D]; all float64.  Returns o [B,k,Hq,D] float64.
    """
    B, k, Hq, D = q.shape
    Hkv = k_cache.shape[2]
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    out = np.zeros((B, k, Hq, D), dtype=np.float64)
    for b in range(B):
        L = int(cache_len[b])
        for hq in range(Hq):
            hk = hq // G
            keys = np.concatenate([k_cache[b, :L, hk, :], k_blk[b, :, hk, :]], axis=0)
            vals = np.concatenate([v_cache[b, :L, hk, :], v_blk[b, :, hk, :]], axis=0)
            s = (q[b, :, hq, :] @ keys.T) * scale            # [k, L+k]
            for i in range(min(n_causal, k)):                 # causal rows of the block
                s[i, L + i + 1:] = -np.inf
            s = s - s.max(axis=1, keepdims=True)
            p = np.exp(s)
            p = p / p.sum(axis=1, keepdims=True)
            out[b, :, hq, :] = p @ vals
    return out


def kv_append(k_cache, v_cache, cache_len, k_rows, v_rows):
    """The keys and values of the n tokens the cache lacks (the previous
    block, processed causally in the first iteration of the next one,
    Algorithm 3) are written at positions L_b .. L_b + n - 1 of the cache.
    k_rows, v_rows [B,n,Hkv,D].  Returns new (k_cache, v_cache, cache_len);
    the inputs are not modified."""
    kc = np.array(k_cache, copy=True)
    vc = np.array(v_cache, copy=True)
    n = k_rows.shape[1]
    lens = np.array(cache_len, dtype=np.int64, copy=True)
    for b in range(kc.shape[0]):
        L = int(lens[b])
        if L + n > kc.shape[1]:
            raise ValueError("cache overflow")
        kc[b, L:L + n] = k_rows[b]
        vc[b, L:L + n] = v_rows[b]
        lens[b] = L + n
    return kc, vc, lens


def masked_sequence_attention(q_seq, k_seq, v_seq, causal_point, scale=None):
    """Brute force: full-sequence attention under the explicit inference mask
    predicate, for one head.  q_seq, k_seq, v_seq [T, D].  Used only to pin
    block_attention on tiny inputs."""
    T, D = q_seq.shape
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    out = np.zeros((T, D), dtype=np.float64)
    for qi in range(T):
        allowed = [j for j in range(T) if inference_mask_allows(qi, j, causal_point)]
        s = np.array([float(q_seq[qi] @ k_seq[j]) * scale for j in allowed])
        s = s - s.max()
        p = np.exp(s)
        p = p / p.sum()
        out[qi] = sum(p[a] * v_seq[j] for a, j in enumerate(allowed))
    return out


# ------------------------------------------------------------- LM head

def logits(hidden_rows: np.ndarray, w_store: np.ndarray, w_dtype: str,
           vocab_chunk: int = 8192) -> np.ndarray:
    """z_{r,v} = sum_c h_{r,c} W_{v,c}: the LM head that produces the block
    logits z_hat of Eq. 5 (nn.Linear layout, W [V,H]).  hidden_rows [R,H]
    float64; w_store [V,H] in storage form.  Vocabulary rows are widened one
    slice at a time only to bound memory: every logit is the same single dot
    product."""
    R = hidden_rows.shape[0]
    V = w_store.shape[0]
    z = np.empty((R, V), dtype=np.float64)
    for v0 in range(0, V, vocab_chunk):
        v1 = min(V, v0 + vocab_chunk)
        z[:, v0:v1] = hidden_rows @ widen(w_store[v0:v1], w_dtype).T
    return z


def entropy(z_row: np.ndarray) -> float:
    """H(p) = -sum_v p_v log p_v in nats, p = softmax(z) (the entropy of the
    predicted marginal used by the EB rule, Eq. 3); 0 log 0 := 0.  Computed
    with the max subtracted for range: log p_v = (z_v - max z) - log Z."""
    z = np.asarray(z_row, dtype=np.float64)
    m = z.max()
    e = np.exp(z - m)
    Z = e.sum()
    p = e / Z
    logp = (z - m) - np.log(Z)
    terms = np.where(p > 0.0, -p * logp, 0.0)
    return float(terms.sum())


def confidence(z_row: np.ndarray) -> float:
    """Confidence c^i = max_v p(x_i = v | x_<t, x_J) of a position's
    predicted marginal, p = softmax(z) (Appendix "Sampling algorithm": the
    Factor rule and the confidence error proxy of the general EB-Sampler).
    With the max subtracted: max_v p_v = 1 / sum_v exp(z_v - max z)."""
    z = np.asarray(z_row, dtype=np.float64)
    return float(1.0 / np.exp(z - z.max()).sum())


def sample_token(z_row: np.ndarray, g_row, tau: float) -> int:
    """Gumbel-max sample: argmax_v (z_v + tau * g_v); tau = 0 (or no noise)
    is greedy decoding, the paper's temperature-0 setting (Sec. 3.1).  For
    tau > 0 this samples softmax(z / tau).  Ties go to the lowest id."""
    z = np.asarray(z_row, dtype=np.float64)
    if tau == 0.0 or g_row is None:
        score = z
    else:
        score = z + float(tau) * np.asarray(g_row, dtype=np.float64)
    return int(np.argmax(score))          # first maximum = lowest id


def head_entropy_sample(hidden, w_store, w_dtype, masked, gumbel, tau,
                        rows=None, vocab_chunk: int = 8192, with_confidence=False):
    """Per block position: entropy (nats) and sampled token of the masked
    positions' predicted marginals p_theta(x_{t+i} | x_<t; x_hat) (Eqs. 6-7,
    Algorithm 3 "compute probabilities").  Position t+i predicts its own
    token (no shift).

    hidden [B,k,H] float64; w_store [V,H] storage; masked [B,k] (nonzero =
    masked); gumbel [B,k,V] or None.  Unmasked positions get entropy +inf and
    token -1.  `rows`, if given, restricts the work to those (b, i) pairs
    (the others are left as +inf / -1).  Returns (entropy [B,k] f64,
    token [B,k] int32, z dict {(b,i): z_row}) -- z is returned for test
    diagnostics (top-2 gaps).  with_confidence=True appends confidence
    [B,k] f64 (0 at unmasked positions)."""
    B, k, H = hidden.shape
    ent = np.full((B, k), np.inf, dtype=np.float64)
    tok = np.full((B, k), MASK_TOKEN, dtype=np.int32)
    conf = np.zeros((B, k), dtype=np.float64)
    if rows is None:
        rows = [(b, i) for b in range(B) for i in range(k) if masked[b, i]]
    else:
        rows = [(b, i) for (b, i) in rows if masked[b, i]]
    if not rows:
        return (ent, tok, {}, conf) if with_confidence else (ent, tok, {})
    hr = np.stack([hidden[b, i] for (b, i) in rows])
    z = logits(hr, w_store, w_dtype, vocab_chunk)
    zs = {}
    for n, (b, i) in enumerate(rows):
        ent[b, i] = entropy(z[n])
        conf[b, i] = confidence(z[n])
        g = None if gumbel is None else gumbel[b, i]
        tok[b, i] = sample_token(z[n], g, tau)
        zs[(b, i)] = z[n]
    return (ent, tok, zs, conf) if with_confidence else (ent, tok, zs)


# ------------------------------------------------------------- EB select

def eb_accept_count(sorted_entropies, gamma: float) -> int:
    """EB-Sampler, entropy proxy (Eq. 3): with the masked entropies sorted
    ascending, s >= 1 is the largest integer with
        sum_{j=1}^{s-1} H_{i_j} <= gamma,
    capped at |M|.  Prefix sums in float64.  For non-negative entropies the
    prefix sums are non-decreasing, so the largest such s is found by walking
    the sorted list until the first prefix sum above gamma."""
    n = len(sorted_entropies)
    if n == 0:
        return 0
    s = 1
    prefix = 0.0
    for j in range(1, n):                  # candidate s = j + 1 needs S_j
        prefix += float(sorted_entropies[j - 1])
        if prefix <= gamma:
            s = j + 1
        else:
            break
    return s


def eb_select(entropy_bk, token_bk, masked_bk, block_tokens_bk, gamma: float):
    """One EB unmasking step over a batch (Algorithm 3, "unmask tokens
    according to Eq. 3").  Per sequence: sort the masked positions by
    (entropy, position) ascending, accept the first s of Eq. 3, write their
    sampled tokens into the block buffer and clear their masked flags.

    Returns (new_masked [B,k] uint8, new_block_tokens [B,k] int32,
    n_unmasked [B] int32, accepted list of sets, sorted orders)."""
    B, k = masked_bk.shape
    new_masked = np.array(masked_bk, dtype=np.uint8, copy=True)
    new_bt = np.array(block_tokens_bk, dtype=np.int32, copy=True)
    n_un = np.zeros(B, dtype=np.int32)
    accepted = []
    orders = []
    for b in range(B):
        M = [i for i in range(k) if masked_bk[b, i]]
        order = sorted(M, key=lambda i: (float(entropy_bk[b, i]), i))
        s = eb_accept_count([entropy_bk[b, i] for i in order], gamma)
        acc = set(order[:s])
        for i in acc:
            new_bt[b, i] = token_bk[b, i]
            new_masked[b, i] = 0
        n_un[b] = s
        accepted.append(acc)
        orders.append(order)
    return new_masked, new_bt, n_un, accepted, orders


def eb_prefix_margins(entropy_row_sorted, gamma: float):
    """|S_{j-1} - gamma| for each rank j >= 2 (1-based) of a sorted list:
    the oracle's margin to gamma at each acceptance decision."""
    out = []
    prefix = 0.0
    for j in range(1, len(entropy_row_sorted)):
        prefix += float(entropy_row_sorted[j - 1])
        out.append(abs(prefix - gamma))
    return out


# ------------------------------------------------- other selection rules

def eb_general_accept_count(entropies_in_order, gamma: float) -> int:
    """General EB-Sampler bound (Appendix "Sampling algorithm", the general
    form of Eq. 3): with the masked positions taken in the order i_1, i_2,
    ... of the error proxy, s >= 1 is the largest count with
        sum_{j<=s} H_{i_j} - max_{j'<=s} H_{i_j'} <= gamma,
    capped at |M|.  Sums in float64.  For non-negative entropies the left
    side never decreases as s grows (a new term adds H and raises the max by
    at most H), so the largest such s is found by walking the order until
    the first count that breaks the bound."""
    n = len(entropies_in_order)
    if n == 0:
        return 0
    s = 1
    total = float(entropies_in_order[0])
    top = total
    for j in range(1, n):                  # candidate s = j + 1
        h = float(entropies_in_order[j])
        total += h
        top = max(top, h)
        if total - top <= gamma:
            s = j + 1
        else:
            break
    return s


def factor_accept_count(confidences_desc, f: float, complement: bool = False) -> int:
    """Factor parallel decoding (Appendix "Sampling algorithm"): with the
    masked confidences sorted descending c^1 >= c^2 >= ..., unmask the first
    n, n the largest count in 1..|M| with
        (n + 1) c^n < f                 (c^n read as the n-th confidence),
    or, with complement=True, (n + 1) (1 - c^n) < f.  When no count
    qualifies n = 1, so that every step unmasks a token; 0 when |M| = 0.
    The literal condition need not hold for a prefix of counts, so every
    count is tested."""
    n_m = len(confidences_desc)
    if n_m == 0:
        return 0
    best = 1
    for n in range(1, n_m + 1):
        c = float(confidences_desc[n - 1])
        lhs = (n + 1) * ((1.0 - c) if complement else c)
        if lhs < f:
            best = n
    return best


SELECT_RULES = ("eb_entropy", "eb_confidence", "factor", "factor_complement")


def select_step(entropy_bk, confidence_bk, token_bk, masked_bk, block_tokens_bk,
                rule: str, threshold: float):
    """One unmasking step under one of the selection rules of the paper
    (Algorithm 3 "unmask tokens", with the rule of Eq. 3 or of the Appendix
    "Sampling algorithm"):
      eb_entropy         Eq. 3 (same as eb_select; threshold = gamma);
      eb_confidence      positions ordered by confidence, descending, and the
                         general EB bound (threshold = gamma);
      factor             confidence order, (n + 1) c^n < f (threshold = f);
      factor_complement  confidence order, (n + 1)(1 - c^n) < f.
    Ties of the ordering key go to the lower block position.  Returns the
    same tuple as eb_select."""
    if rule not in SELECT_RULES:
        raise ValueError(rule)
    if rule == "eb_entropy":
        return eb_select(entropy_bk, token_bk, masked_bk, block_tokens_bk, threshold)
    B, k = masked_bk.shape
    new_masked = np.array(masked_bk, dtype=np.uint8, copy=True)
    new_bt = np.array(block_tokens_bk, dtype=np.int32, copy=True)
    n_un = np.zeros(B, dtype=np.int32)
    accepted = []
    orders = []
    for b in range(B):
        M = [i for i in range(k) if masked_bk[b, i]]
        order = sorted(M, key=lambda i: (-float(confidence_bk[b, i]), i))
        if rule == "eb_confidence":
            s = eb_general_accept_count([entropy_bk[b, i] for i in order], threshold)
        else:
            s = factor_accept_count([confidence_bk[b, i] for i in order], threshold,
                                    complement=(rule == "factor_complement"))
        acc = set(order[:s])
        for i in acc:
            new_bt[b, i] = token_bk[b, i]
            new_masked[b, i] = 0
        n_un[b] = s
        accepted.append(acc)
        orders.append(order)
    return new_masked, new_bt, n_un, accepted, orders


# ------------------------------------------- counter-based Gumbel noise

PHILOX_M0, PHILOX_M1 = 0xD2511F53, 0xCD9E8D57       # round multipliers
PHILOX_W0, PHILOX_W1 = 0x9E3779B9, 0xBB67AE85       # key schedule increments


def philox4x32_10(ctr, key):
    """Philox4x32 with 10 rounds (Salmon, Moraes, Dror, Shaw, "Parallel random
    numbers: as easy as 1, 2, 3", SC 2011), vectorised over the leading axis.
    ctr: uint32 [..., 4]; key: uint32 [..., 2].  Each round multiplies words
    0 and 2 by the round constants (64-bit products split into high and low
    halves) and mixes in words 1 and 3 and the key; the key grows by the Weyl
    increments between rounds.  Returns uint32 [..., 4]."""
    c = np.array(ctr, dtype=np.uint64) & 0xFFFFFFFF
    k = np.array(key, dtype=np.uint64) & 0xFFFFFFFF
    c0, c1, c2, c3 = c[..., 0], c[..., 1], c[..., 2], c[..., 3]
    k0, k1 = k[..., 0], k[..., 1]
    for r in range(10):
        if r > 0:
            k0 = (k0 + PHILOX_W0) & 0xFFFFFFFF
            k1 = (k1 + PHILOX_W1) & 0xFFFFFFFF
        p0 = c0 * np.uint64(PHILOX_M0)            # < 2^64: exact in uint64
        p1 = c2 * np.uint64(PHILOX_M1)
        hi0, lo0 = p0 >> np.uint64(32), p0 & np.uint64(0xFFFFFFFF)
        hi1, lo1 = p1 >> np.uint64(32), p1 & np.uint64(0xFFFFFFFF)
        c0, c1, c2, c3 = hi1 ^ c1 ^ k0, lo1, hi0 ^ c3 ^ k1, lo0
    return np.stack([c0, c1, c2, c3], axis=-1).astype(np.uint32)


def philox_gumbel(row_ids, vocab: int, seed: int, offset: int = 0):
    """Gumbel noise of the in-kernel generator, in float64: for block
    position n (= b * k + i) and vocabulary id v, x is word v mod 4 of
    Philox4x32-10 with counter (v div 4, n, offset low, offset high) and key
    (seed low, seed high); u = ((x >> 9) + 1/2) 2^-23 lies strictly inside
    (0, 1) and is exact in fp32 (24 significant bits); g = -log(-log u).  Returns (g [len(row_ids), V] float64,
    x [len(row_ids), V] uint32)."""
    n = np.asarray(row_ids, dtype=np.uint64)
    v = np.arange(vocab, dtype=np.uint64)
    R = n.shape[0]
    ctr = np.zeros((R, (vocab + 3) // 4, 4), dtype=np.uint64)
    ctr[..., 0] = np.arange((vocab + 3) // 4, dtype=np.uint64)[None, :]
    ctr[..., 1] = n[:, None]
    ctr[..., 2] = offset & 0xFFFFFFFF
    ctr[..., 3] = (offset >> 32) & 0xFFFFFFFF
    key = np.zeros((R, (vocab + 3) // 4, 2), dtype=np.uint64)
    key[..., 0] = seed & 0xFFFFFFFF
    key[..., 1] = (seed >> 32) & 0xFFFFFFFF
    words = philox4x32_10(ctr, key).reshape(R, -1)[:, :vocab]   # word v mod 4 of call v div 4
    assert words.shape[1] == v.shape[0]
    u = ((words >> 9).astype(np.float64) + 0.5) * 2.0 ** -23
    return -np.log(-np.log(u)), words


# ------------------------------------------------- theoretical timing model

# Constants of the paper's roofline analysis (Sec. "Timing analysis"): an
# H100 with FP8 weights and KV (1 byte per element), BF16 attention, and an
# 8B transformer with 32 query heads of 128 and 8 KV heads.
ROOFLINE_H100 = dict(bytes_per_el=1, peak_flops=1978e12, peak_flops_attention=989e12,
                     bandwidth=3.35 * 1024 ** 4, hidden=4096, ffn=4 * 4096, n_heads=32,
                     head_dim=128, n_kv_heads=8, kv_bytes=1)


def roofline_gemm(m: int, n: int, k: int, c=ROOFLINE_H100):
    """Roofline time of C = A B with A [m, k], B [k, n]: the larger of
    (m k + k n + m n) elements moved at the bandwidth and 2 m n k flops at
    the peak.  Returns (seconds, flops)."""
    io = (m * k + n * k + m * n) * c["bytes_per_el"]
    flops = 2.0 * m * n * k
    return max(io / c["bandwidth"], flops / c["peak_flops"]), flops


def roofline_attention(block: int, kv_len: int, batch: int, c=ROOFLINE_H100) -> float:
    """One fused attention kernel: Q, the K and V of the cache, and the
    output move once; QK^T and PV are the two contractions over the cache
    length at the attention peak."""
    tokens = block * batch
    width = c["n_heads"] * c["head_dim"]
    q = tokens * width * c["bytes_per_el"]
    kv = 2 * batch * kv_len * c["n_kv_heads"] * c["head_dim"] * c["kv_bytes"]
    o = tokens * width * c["bytes_per_el"]
    flops = 2 * roofline_gemm(tokens, kv_len, width, c)[1]
    return max((q + kv + o) / c["bandwidth"], flops / c["peak_flops_attention"])


def roofline_linear(block: int, batch: int, c=ROOFLINE_H100) -> float:
    """The layer's GEMMs with the shapes of the paper's analysis, as printed:
    the FFN up- and down-projections contract over hidden * ffn, and the K and
    V projections have width n_heads * n_kv_heads (the reading this build
    takes of the printed model, which reproduces its tables)."""
    t, h, f = block * batch, c["hidden"], c["ffn"]
    nh, hd, nkv = c["n_heads"], c["head_dim"], c["n_kv_heads"]
    shapes = [(t, h, h * f), (t, h * f, h), (t, h, nh * hd), (t, h, nh * nkv), (t, h, nh * nkv),
              (t, nh * hd, h)]
    return sum(roofline_gemm(m, n, k, c)[0] for (m, n, k) in shapes)


def linear(x, w):
    """y = x W^T in fp64 over the given values (x [T, K], W [N, K], the
    nn.Linear layout): the GEMM of a linear layer, which the timing section
    counts in every forward besides the attention."""
    return np.asarray(x, np.float64) @ np.asarray(w, np.float64).T


def roofline_forward(block: int, kv_len: int, batch: int, c=ROOFLINE_H100) -> float:
    """Forward time of one layer for a block of `block` tokens per sequence:
    attention plus the linear layers (the layer count cancels in ratios)."""
    return roofline_attention(block, kv_len, batch, c) + roofline_linear(block, batch, c)


def block_slowdown(block: int, kv_len: int, batch: int, c=ROOFLINE_H100) -> float:
    """time(block) / time(1): the cost of a block forward over an NTP one."""
    return roofline_forward(block, kv_len, batch, c) / roofline_forward(1, kv_len, batch, c)


def sbd_speedup(k: int, l: int, time_fn) -> float:
    """Wall-clock speedup of SBD over NTP for a block of k tokens decoded in
    l forwards: k time(1) / (time(2k) + (l - 1) time(k)) -- the first forward
    of a block also carries the previous block's k tokens (2k rows)."""
    return k * time_fn(1) / (time_fn(2 * k) + (l - 1) * time_fn(k))
