"""First iteration of a block after the previous one (Algorithm 3): block
attention with n_causal causal leading rows whose keys/values enter the
cache, against the oracle (block_attention with n_causal, kv_append).
Output within the attention tolerances; the cache append bit-exact, with
every other cache slot untouched (slots past the lengths hold NaN, so a
stray read or write shows)."""
import numpy as np
import pytest

import gen
import oracle
from tests.helpers import BF16_ATTN_TOL, F32_ATTN_TOL, to_dev

pytestmark = pytest.mark.gpu

BF16 = gen.get_workload("llama8b_k16")


@pytest.fixture(scope="module")
def sbd():
    import paper_2509_04185_gb300 as m
    return m


def _inputs(w, seed, lens):
    d = dict(gen.attention_inputs(w, seed, poison_tail=False))
    d["cache_len"] = np.asarray(lens, dtype=np.int32)
    nanv = gen.BF16_NAN if w.dtype == "bf16" else np.float32("nan")
    for b in range(w.batch):
        d["k_cache"][b, lens[b]:] = nanv
        d["v_cache"][b, lens[b]:] = nanv
    return d


def _run(sbd, w, d, n_causal, num_splits=0):
    import torch
    dt = w.dtype
    t = {x: to_dev(d[x], dt) for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    lens_t = torch.from_numpy(d["cache_len"]).cuda()
    out = sbd.sbd_block_attention_causal_prefix(t["q"], t["k_cache"], t["v_cache"], lens_t,
                                                t["k_blk"], t["v_blk"], n_causal,
                                                num_splits=num_splits)
    torch.cuda.synchronize()

    def back(x):
        a = x.cpu()
        return a.view(torch.int16).numpy().view(np.uint16) if dt == "bf16" else a.numpy()
    return out.float().cpu().numpy(), back(t["k_cache"]), back(t["v_cache"])


def _check(sbd, w, d, n_causal, num_splits=0, expect_append=True):
    got, kc, vc = _run(sbd, w, d, n_causal, num_splits)
    dt = w.dtype
    f = {x: oracle.widen(d[x], dt) for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    ref = oracle.block_attention(f["q"], f["k_cache"], f["v_cache"], d["cache_len"], f["k_blk"],
                                 f["v_blk"], n_causal=n_causal)
    assert np.isfinite(got).all()
    err = float(np.abs(got - ref).max())
    assert err <= (F32_ATTN_TOL if dt == "f32" else BF16_ATTN_TOL), err
    if expect_append:
        kc_ref, vc_ref, _ = oracle.kv_append(d["k_cache"], d["v_cache"], d["cache_len"],
                                             d["k_blk"][:, :n_causal], d["v_blk"][:, :n_causal])
    else:
        kc_ref, vc_ref = d["k_cache"], d["v_cache"]
    # bit patterns (NaN poison included) must match exactly
    assert np.array_equal(kc.view(np.uint8), np.ascontiguousarray(kc_ref).view(np.uint8))
    assert np.array_equal(vc.view(np.uint8), np.ascontiguousarray(vc_ref).view(np.uint8))
    return err


@pytest.mark.parametrize("k,n_causal", [(8, 4), (4, 4), (6, 1), (32, 16)])
def test_f32(sbd, k, n_causal):
    w = gen.shrink(gen.get_workload("tiny_f32"), batch=2, block_k=k, n_q_heads=4, n_kv_heads=2,
                   cache_len=(0, 300))
    _check(sbd, w, _inputs(w, k, [0, 300 - n_causal]), n_causal)
    assert sbd.sbd_device_error() == 0


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("G,k,n_causal", [(1, 16, 8), (2, 8, 4), (4, 4, 2),     # <= 16 packed rows
                                          (4, 8, 4), (3, 10, 5),
                                          (4, 16, 8), (2, 32, 16),               # up to 64: attn_tc_kernel
                                          (4, 32, 16), (4, 32, 32), (8, 16, 1)])
def test_bf16_kernels(sbd, D, G, k, n_causal):
    Hkv = 2
    w = gen.shrink(BF16, batch=3, block_k=k, n_q_heads=G * Hkv, n_kv_heads=Hkv, head_dim=D,
                   cache_len=(1, 400))
    _check(sbd, w, _inputs(w, G + k, [0, 129, 400 - n_causal]), n_causal)
    assert sbd.sbd_device_error() == 0


@pytest.mark.parametrize("splits", [1, 2, 5, 19])
def test_first_iteration_at_llama_shapes(sbd, splits):
    # 2k = 32 rows (the previous block's 16 tokens, then the 16 masks),
    # 32/8 heads, D = 128, cache 4096 (room for the 16 appended rows)
    w = gen.shrink(BF16, block_k=32, cache_len=4096 + 16)
    _check(sbd, w, _inputs(w, 0, [4096]), 16, num_splits=splits)
    assert sbd.sbd_device_error() == 0


def test_zero_causal_rows_is_block_attention(sbd):
    import torch
    w = gen.shrink(BF16, batch=2, block_k=16, cache_len=(100, 700))
    d = _inputs(w, 3, [100, 700])
    t = {x: to_dev(d[x], "bf16") for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    lens = torch.from_numpy(d["cache_len"]).cuda()
    a = sbd.sbd_block_attention(t["q"], t["k_cache"], t["v_cache"], lens, t["k_blk"], t["v_blk"])
    b = sbd.sbd_block_attention_causal_prefix(t["q"], t["k_cache"], t["v_cache"], lens,
                                              t["k_blk"], t["v_blk"], 0)
    assert torch.equal(a, b)
    _check(sbd, w, d, 0)


def test_append_overflow_is_reported_and_skipped(sbd):
    w = gen.shrink(BF16, batch=2, block_k=8, n_q_heads=8, n_kv_heads=2, cache_len=(0, 200))
    d = _inputs(w, 1, [50, 197])            # 197 + 4 > 200: the second sequence cannot append
    got, kc, vc = _run(sbd, w, d, 4)
    assert sbd.sbd_device_error() & sbd.SBD_DEVERR_CACHE_LEN
    f = {x: oracle.widen(d[x], "bf16") for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    ref = oracle.block_attention(f["q"], f["k_cache"], f["v_cache"], d["cache_len"], f["k_blk"],
                                 f["v_blk"], n_causal=4)
    assert float(np.abs(got - ref).max()) <= BF16_ATTN_TOL
    assert np.array_equal(kc[1], d["k_cache"][1]) and np.array_equal(vc[1], d["v_cache"][1])
    assert np.array_equal(kc[0, 50:54], d["k_blk"][0, :4])


@pytest.mark.parametrize("case", range(16))
def test_bf16_random_shapes(sbd, case):
    """Seeded random first-iteration calls: both tcgen05 kernels (up to 64
    and 65-128 packed rows), both head dims, n_causal from 1 to k, ragged
    lengths with room for the append, automatic or explicit split counts."""
    rng = np.random.default_rng(2000 + case)
    D = int(rng.choice([64, 128]))
    Hkv = int(rng.integers(1, 4))
    G = int(rng.integers(1, 9))
    k = int(rng.integers(1, min(32, 128 // G) + 1))
    n_causal = int(rng.integers(1, k + 1))
    B = int(rng.integers(1, 5))
    Lmax = int(rng.integers(n_causal, 900))
    lens = [int(x) for x in rng.integers(0, Lmax - n_causal + 1, size=B)]
    splits = int(rng.choice([0, 0, 1, 2, 5, 9]))
    w = gen.shrink(BF16, batch=B, block_k=k, n_q_heads=G * Hkv, n_kv_heads=Hkv, head_dim=D,
                   cache_len=(0, Lmax))
    _check(sbd, w, _inputs(w, case, lens), n_causal, num_splits=splits)
    assert sbd.sbd_device_error() == 0
