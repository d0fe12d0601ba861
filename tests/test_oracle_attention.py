"""Pins of the oracle's block attention (CPU only).

Each check is independent of the oracle's own code path: an explicit
mask-matrix brute force written from the inference mask predicate, PyTorch's
scaled_dot_product_attention for the k = 1 (plain causal decode) case, and
closed forms.  A mutation test at the end plants plausible mistakes in the
oracle and checks that one of these pins catches each."""
import numpy as np
import pytest
import torch

import gen
import oracle


def _rand_inputs(B, k, Hq, Hkv, D, L, seed, lens=None):
    rng = np.random.default_rng(seed)
    q = rng.standard_normal((B, k, Hq, D))
    kc = rng.standard_normal((B, L, Hkv, D))
    vc = rng.standard_normal((B, L, Hkv, D))
    kb = rng.standard_normal((B, k, Hkv, D))
    vb = rng.standard_normal((B, k, Hkv, D))
    if lens is None:
        lens = np.full(B, L, dtype=np.int32)
    return q, kc, vc, np.asarray(lens, dtype=np.int32), kb, vb


def _explicit_mask_attention(q, kc, vc, lens, kb, vb, scale=None, n_causal=0):
    """Full-sequence attention, one head at a time, where every position of
    the sequence x_<t ; x_hat_t..x_hat_{t+k-1} is a query and the mask is an
    explicit [T, T] boolean matrix built from the paper's inference predicate
    (causal before the block start, everything visible from inside the
    block).  Only the block rows are returned."""
    B, k, Hq, D = q.shape
    Hkv = kc.shape[2]
    G = Hq // Hkv
    if scale is None:
        scale = 1.0 / np.sqrt(D)
    out = np.zeros_like(q)
    for b in range(B):
        L = int(lens[b])
        T = L + k
        mask = np.zeros((T, T), dtype=bool)
        for qi in range(T):
            for kv in range(T):
                mask[qi, kv] = oracle.inference_mask_allows(qi, kv, L + n_causal)
        for hq in range(Hq):
            hk = hq // G
            K = np.concatenate([kc[b, :L, hk], kb[b, :, hk]])
            V = np.concatenate([vc[b, :L, hk], vb[b, :, hk]])
            # queries of the prefix are irrelevant for the block rows; use
            # the block queries in rows L..T-1 and zeros elsewhere
            Q = np.zeros((T, D))
            Q[L:] = q[b, :, hq]
            s = Q @ K.T * scale
            s = np.where(mask, s, -np.inf)
            s = s - s.max(axis=1, keepdims=True)
            p = np.exp(s)
            p /= p.sum(axis=1, keepdims=True)
            out[b, :, hq] = (p @ V)[L:]
    return out


@pytest.mark.parametrize("k,L,Hq,Hkv", [(1, 5, 2, 1), (3, 4, 4, 2), (4, 7, 4, 4), (2, 0, 2, 2)])
def test_block_attention_equals_explicit_mask(k, L, Hq, Hkv):
    q, kc, vc, lens, kb, vb = _rand_inputs(2, k, Hq, Hkv, 8, max(L, 1), seed=k * 10 + L,
                                           lens=[L, max(L - 1, 0)])
    got = oracle.block_attention(q, kc, vc, lens, kb, vb)
    ref = _explicit_mask_attention(q, kc, vc, lens, kb, vb)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_mask_predicate_matches_paper_picture():
    # Fig. 3: prefix rows lower-triangular, block rows fully visible.
    L, k = 5, 4
    T = L + k
    M = np.array([[oracle.inference_mask_allows(i, j, L) for j in range(T)] for i in range(T)])
    assert np.array_equal(M[:L, :L], np.tril(np.ones((L, L), dtype=bool)))
    assert not M[:L, L:].any()
    assert M[L:, :].all()


def test_brute_force_sequence_attention_agrees():
    # the per-query brute force over the predicate agrees with the block rows
    rng = np.random.default_rng(3)
    L, k, D = 6, 3, 8
    T = L + k
    qs, ks, vs = rng.standard_normal((3, T, D))
    full = oracle.masked_sequence_attention(qs, ks, vs, causal_point=L)
    q = qs[None, L:, None, :]
    kc = ks[None, :L, None, :]
    vc = vs[None, :L, None, :]
    kb = ks[None, L:, None, :]
    vb = vs[None, L:, None, :]
    got = oracle.block_attention(q, kc, vc, np.array([L]), kb, vb)
    np.testing.assert_allclose(got[0, :, 0, :], full[L:], atol=1e-12)


@pytest.mark.parametrize("Hq,Hkv", [(4, 2), (8, 2), (2, 2)])
def test_k1_is_plain_causal_decode_sdpa(Hq, Hkv):
    """k = 1: the single block query at position L sees keys 0..L, i.e. plain
    next-token decode with a causal mask (Eq. 1).  Checked against PyTorch's
    SDPA over the whole sequence with is_causal and KV heads repeated
    (query head hq uses KV head hq // G)."""
    B, D, L = 2, 16, 9
    q, kc, vc, lens, kb, vb = _rand_inputs(B, 1, Hq, Hkv, D, L, seed=7)
    got = oracle.block_attention(q, kc, vc, lens, kb, vb)
    G = Hq // Hkv
    rng = np.random.default_rng(11)
    qpre = rng.standard_normal((B, L, Hq, D))
    Qs = np.concatenate([qpre, q], axis=1)              # [B, L+1, Hq, D]
    Ks = np.concatenate([kc, kb], axis=1)               # [B, L+1, Hkv, D]
    Vs = np.concatenate([vc, vb], axis=1)
    Qt = torch.from_numpy(Qs).permute(0, 2, 1, 3)
    Kt = torch.from_numpy(Ks).permute(0, 2, 1, 3).repeat_interleave(G, dim=1)
    Vt = torch.from_numpy(Vs).permute(0, 2, 1, 3).repeat_interleave(G, dim=1)
    ref = torch.nn.functional.scaled_dot_product_attention(Qt, Kt, Vt, is_causal=True)
    ref = ref.permute(0, 2, 1, 3).numpy()[:, L:]
    np.testing.assert_allclose(got, ref, atol=1e-10)


def test_zero_query_is_uniform_average():
    q, kc, vc, lens, kb, vb = _rand_inputs(2, 3, 4, 2, 8, 10, seed=5, lens=[10, 4])
    q[:] = 0.0
    got = oracle.block_attention(q, kc, vc, lens, kb, vb)
    for b in range(2):
        L = lens[b]
        for hq in range(4):
            hk = hq // 2
            mean = np.concatenate([vc[b, :L, hk], vb[b, :, hk]]).mean(axis=0)
            for i in range(3):
                np.testing.assert_allclose(got[b, i, hq], mean, atol=1e-12)


def test_equal_keys_give_mean_of_values():
    q, kc, vc, lens, kb, vb = _rand_inputs(1, 4, 2, 1, 8, 6, seed=9)
    key = np.random.default_rng(1).standard_normal(8)
    kc[:] = key
    kb[:] = key
    got = oracle.block_attention(q, kc, vc, lens, kb, vb)
    mean = np.concatenate([vc[0, :, 0], vb[0, :, 0]]).mean(axis=0)
    np.testing.assert_allclose(got[0, :, 0], np.broadcast_to(mean, (4, 8)), atol=1e-12)


def test_block_is_a_set():
    """Bidirectional block: permuting the block queries permutes the outputs;
    permuting the block keys/values together leaves them unchanged."""
    q, kc, vc, lens, kb, vb = _rand_inputs(1, 5, 4, 2, 8, 7, seed=13)
    base = oracle.block_attention(q, kc, vc, lens, kb, vb)
    perm = np.array([3, 0, 4, 1, 2])
    pq = oracle.block_attention(q[:, perm], kc, vc, lens, kb, vb)
    np.testing.assert_allclose(pq, base[:, perm], atol=1e-12)
    pkv = oracle.block_attention(q, kc, vc, lens, kb[:, perm], vb[:, perm])
    np.testing.assert_allclose(pkv, base, atol=1e-12)


def test_slots_beyond_length_are_not_read():
    w = gen.shrink(gen.WORKLOADS["ragged_b32_k8"], batch=3, cache_len=(3, 9), n_q_heads=4,
                   n_kv_heads=2, head_dim=8, block_k=3)
    d = gen.attention_inputs(w, seed=1, poison_tail=True)
    f = {k: oracle.widen(v, w.dtype) for k, v in d.items() if k != "cache_len"}
    out = oracle.block_attention(f["q"], f["k_cache"], f["v_cache"], d["cache_len"],
                                 f["k_blk"], f["v_blk"])
    assert np.isfinite(out).all()
    assert (d["cache_len"] < w.max_cache_len).any()


def test_scale_override():
    q, kc, vc, lens, kb, vb = _rand_inputs(1, 2, 2, 1, 8, 5, seed=21)
    a = oracle.block_attention(q, kc, vc, lens, kb, vb, scale=0.5)
    b = oracle.block_attention(2 * q, kc, vc, lens, kb, vb, scale=0.25)
    np.testing.assert_allclose(a, b, atol=1e-12)
    ref = _explicit_mask_attention(q, kc, vc, lens, kb, vb, scale=0.5)
    np.testing.assert_allclose(a, ref, atol=1e-12)


# ------------------------------------------- first iteration: causal prefix rows

@pytest.mark.parametrize("k,n_causal,L", [(4, 2, 5), (6, 3, 0), (2, 1, 3), (8, 4, 6), (3, 3, 4)])
def test_causal_prefix_rows_equal_explicit_mask(k, n_causal, L):
    q, kc, vc, lens, kb, vb = _rand_inputs(2, k, 4, 2, 8, max(L, 1), seed=100 + k * 7 + n_causal,
                                           lens=[L, max(L - 2, 0)])
    got = oracle.block_attention(q, kc, vc, lens, kb, vb, n_causal=n_causal)
    ref = _explicit_mask_attention(q, kc, vc, lens, kb, vb, n_causal=n_causal)
    np.testing.assert_allclose(got, ref, rtol=0, atol=1e-12)


def test_all_causal_block_is_torch_causal_prefill():
    # every block row causal: plain causal attention over cache + block
    B, k, Hq, Hkv, D, L = 2, 5, 4, 2, 16, 6
    q, kc, vc, lens, kb, vb = _rand_inputs(B, k, Hq, Hkv, D, L, seed=77)
    got = oracle.block_attention(q, kc, vc, lens, kb, vb, n_causal=k)
    G = Hq // Hkv
    for b in range(B):
        K = torch.from_numpy(np.concatenate([kc[b], kb[b]]))          # [L+k, Hkv, D]
        V = torch.from_numpy(np.concatenate([vc[b], vb[b]]))
        Q = torch.from_numpy(q[b])                                      # [k, Hq, D]
        allowed = torch.ones(k, L + k, dtype=torch.bool)
        allowed[:, L:] = torch.tril(torch.ones(k, k, dtype=torch.bool))
        for hq in range(Hq):
            ref = torch.nn.functional.scaled_dot_product_attention(
                Q[:, hq][None], K[:, hq // G][None], V[:, hq // G][None], attn_mask=allowed)[0]
            np.testing.assert_allclose(got[b, :, hq], ref.numpy(), rtol=0, atol=1e-12)


def test_bidirectional_rows_equal_block_after_append():
    # The new block's rows of a first-iteration forward (2k rows, the first k
    # causal) see what a plain block forward sees once the previous block is
    # in the cache.
    B, k, Hq, Hkv, D, L = 2, 4, 4, 2, 8, 9
    rng = np.random.default_rng(5)
    q2 = rng.standard_normal((B, 2 * k, Hq, D))
    kc = rng.standard_normal((B, L + k, Hkv, D))
    vc = rng.standard_normal((B, L + k, Hkv, D))
    kb2 = rng.standard_normal((B, 2 * k, Hkv, D))
    vb2 = rng.standard_normal((B, 2 * k, Hkv, D))
    lens = np.array([L, L - 3], dtype=np.int32)
    two_k = oracle.block_attention(q2, kc, vc, lens, kb2, vb2, n_causal=k)
    kc2, vc2, lens2 = oracle.kv_append(kc, vc, lens, kb2[:, :k], vb2[:, :k])
    assert list(lens2) == [L + k, L - 3 + k]
    one = oracle.block_attention(q2[:, k:], kc2, vc2, lens2, kb2[:, k:], vb2[:, k:])
    np.testing.assert_allclose(two_k[:, k:], one, rtol=0, atol=1e-12)


def test_kv_append_writes_only_the_new_rows():
    rng = np.random.default_rng(2)
    kc = rng.standard_normal((2, 10, 2, 4))
    vc = rng.standard_normal((2, 10, 2, 4))
    kr = rng.standard_normal((2, 3, 2, 4))
    vr = rng.standard_normal((2, 3, 2, 4))
    lens = np.array([4, 7])
    kc0, lens0 = kc.copy(), lens.copy()
    k2, v2, l2 = oracle.kv_append(kc, vc, lens, kr, vr)
    assert list(l2) == [7, 10]
    np.testing.assert_array_equal(k2[0, 4:7], kr[0])
    np.testing.assert_array_equal(v2[1, 7:10], vr[1])
    np.testing.assert_array_equal(k2[0, :4], kc[0, :4])
    np.testing.assert_array_equal(k2[0, 7:], kc[0, 7:])
    np.testing.assert_array_equal(kc, kc0)         # inputs unmodified
    np.testing.assert_array_equal(lens, lens0)
    with pytest.raises(ValueError):
        oracle.kv_append(kc, vc, np.array([8, 0]), kr, vr)


def test_empty_cache_and_one_block_key_return_its_value():
    """A sequence with no cached keys and a block of one position: the only
    key has softmax weight 1, so each query head returns its KV head's
    block value exactly, whatever the query."""
    q, kc, vc, lens, kb, vb = _rand_inputs(2, 1, 8, 2, 64, 5, seed=7, lens=[0, 0])
    out = oracle.block_attention(q, kc, vc, lens, kb, vb)
    for h in range(8):
        np.testing.assert_allclose(out[:, 0, h], vb[:, 0, h // 4], rtol=0, atol=1e-15)


def test_query_scale_trades_with_softmax_scale():
    """s = scale * q.k: multiplying q by c and the scale by 1/c leaves every
    score, hence the output, unchanged."""
    q, kc, vc, lens, kb, vb = _rand_inputs(1, 4, 4, 2, 64, 40, seed=8, lens=[33])
    a = oracle.block_attention(q, kc, vc, lens, kb, vb, scale=0.125)
    b = oracle.block_attention(q * 4.0, kc, vc, lens, kb, vb, scale=0.125 / 4.0)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-12)
