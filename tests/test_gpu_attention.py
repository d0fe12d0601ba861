"""Block attention kernels against the fp64 oracle (Eq. 5, inference mask):
max-abs 1e-5 for fp32 inputs, 2e-2 for bf16 inputs with fp32 accumulation.
Cache slots past each sequence's length hold NaN, so any read of them that
reaches the result fails the comparison."""
import numpy as np
import pytest

import gen
import oracle
from tests.helpers import BF16_ATTN_TOL, F32_ATTN_TOL, to_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def sbd():
    import paper_2509_04185_gb300 as m
    return m


def _run_and_compare(sbd, w, seed=0, num_splits=0, lens=None, scale=0.0):
    import torch
    d = gen.attention_inputs(w, seed, poison_tail=lens is None)
    if lens is not None:
        d = dict(d)
        d["cache_len"] = np.asarray(lens, dtype=np.int32)
        nanv = gen.BF16_NAN if w.dtype == "bf16" else np.float32("nan")
        for b in range(w.batch):
            d["k_cache"][b, lens[b]:] = nanv
            d["v_cache"][b, lens[b]:] = nanv
    dt = w.dtype
    args = [to_dev(d[x], dt) for x in ("q", "k_cache", "v_cache")]
    lens_t = torch.from_numpy(d["cache_len"]).cuda()
    out = sbd.sbd_block_attention(args[0], args[1], args[2], lens_t, to_dev(d["k_blk"], dt),
                                  to_dev(d["v_blk"], dt), num_splits=num_splits, scale=scale)
    got = out.float().cpu().numpy()
    f = {x: oracle.widen(d[x], dt) for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    ref = oracle.block_attention(f["q"], f["k_cache"], f["v_cache"], d["cache_len"], f["k_blk"],
                                 f["v_blk"], scale=None if scale == 0.0 else scale)
    assert np.isfinite(got).all()
    err = float(np.abs(got - ref).max())
    tol = F32_ATTN_TOL if dt == "f32" else BF16_ATTN_TOL
    assert err <= tol, err
    assert sbd.sbd_device_error() == 0
    return err


def test_tiny_f32_config(sbd):
    for seed in range(3):
        _run_and_compare(sbd, gen.get_workload("tiny_f32"), seed)


@pytest.mark.parametrize("k,Hq,Hkv", [(1, 4, 2), (3, 8, 2), (7, 4, 4), (32, 2, 2)])
def test_f32_shapes(sbd, k, Hq, Hkv):
    w = gen.shrink(gen.get_workload("tiny_f32"), batch=2, block_k=k, n_q_heads=Hq,
                   n_kv_heads=Hkv, cache_len=(0, 300))
    _run_and_compare(sbd, w, seed=k)


BF16 = gen.get_workload("llama8b_k16")


@pytest.mark.parametrize("case", range(8))
def test_f32_random_shapes(sbd, case):
    """Seeded random fp32 shapes: both head dims, GQA groups, ragged cache
    lengths (zero included) past the kernel's 128-key blocks."""
    rng = np.random.default_rng(4000 + case)
    D = int(rng.choice([64, 128]))
    Hkv = int(rng.integers(1, 4))
    G = int(rng.integers(1, 5))
    k = int(rng.integers(1, 17))
    B = int(rng.integers(1, 4))
    Lmax = int(rng.integers(1, 400))
    lens = [int(x) for x in rng.integers(0, Lmax + 1, size=B)]
    w = gen.shrink(gen.get_workload("tiny_f32"), batch=B, block_k=k, n_q_heads=G * Hkv,
                   n_kv_heads=Hkv, head_dim=D, cache_len=(0, Lmax))
    _run_and_compare(sbd, w, seed=case, lens=lens)


@pytest.mark.parametrize("D", [64, 128])
@pytest.mark.parametrize("G,k", [(4, 1), (4, 4), (1, 16), (4, 8), (3, 7), (2, 9), (4, 12), (4, 16),
                                 (2, 40 // 2), (4, 32), (8, 16), (3, 25), (5, 20), (2, 32)])
def test_bf16_shapes(sbd, D, G, k):
    Hkv = 2
    w = gen.shrink(BF16, batch=2, block_k=k, n_q_heads=G * Hkv, n_kv_heads=Hkv, head_dim=D,
                   cache_len=(1, 333))
    _run_and_compare(sbd, w, seed=G * 100 + k)


@pytest.mark.parametrize("splits", [1, 2, 3, 7, 40])
def test_bf16_split_counts(sbd, splits):
    w = gen.shrink(BF16, batch=3, block_k=16, n_q_heads=8, n_kv_heads=2, cache_len=(0, 700))
    _run_and_compare(sbd, w, seed=splits, num_splits=splits)


def test_bf16_ragged_edges(sbd):
    # lengths 0, 1, a full tile, a tile + 1 and the maximum
    w = gen.shrink(BF16, batch=5, block_k=8, n_q_heads=8, n_kv_heads=2, cache_len=(0, 129))
    _run_and_compare(sbd, w, lens=[0, 1, 64, 65, 129], num_splits=2)
    _run_and_compare(sbd, w, lens=[0, 1, 64, 65, 129], num_splits=1)


@pytest.mark.parametrize("k,splits", [(8, 5), (8, 16), (32, 1), (32, 2), (32, 7)])
def test_bf16_ragged_edges_every_kernel(sbd, k, splits):
    """Lengths 0, 1, 64, 65 and 129 through both tcgen05 kernels (32 and 128
    packed rows), with splits merged in a cluster (2, 5, 7, 16 splits, some
    of them empty) or unsplit."""
    w = gen.shrink(BF16, batch=5, block_k=k, n_q_heads=8, n_kv_heads=2, cache_len=(0, 129))
    _run_and_compare(sbd, w, lens=[0, 1, 64, 65, 129], num_splits=splits)


@pytest.mark.parametrize("case", range(24))
def test_bf16_random_shapes(sbd, case):
    """Seeded random shapes across both tcgen05 kernels (up to 64 and 65-128
    packed rows G k), both head dims, ragged cache lengths (zero, tile
    edges, anything up to the maximum) and automatic or explicit split
    counts, so that both split merges (inside a cluster, and the combine
    kernel) and empty splits are taken."""
    rng = np.random.default_rng(1000 + case)
    D = int(rng.choice([64, 128]))
    Hkv = int(rng.integers(1, 5))
    G = int(rng.integers(1, 9))
    k = int(rng.integers(1, min(32, 128 // G) + 1))
    B = int(rng.integers(1, 7))
    Lmax = int(rng.integers(1, 1200))
    lens = [int(x) for x in rng.integers(0, Lmax + 1, size=B)]
    if case % 3 == 0:      # tile edges
        lens[0] = min(Lmax, 64 * int(rng.integers(0, 4)) + int(rng.integers(0, 2)))
    splits = int(rng.choice([0, 0, 0, 1, 2, 3, 5, 9, 17, 33]))
    w = gen.shrink(BF16, batch=B, block_k=k, n_q_heads=G * Hkv, n_kv_heads=Hkv, head_dim=D,
                   cache_len=(0, Lmax))
    _run_and_compare(sbd, w, seed=case, num_splits=splits, lens=lens)


def test_bf16_scale_override(sbd):
    w = gen.shrink(BF16, batch=1, block_k=4, n_q_heads=8, n_kv_heads=2, cache_len=100)
    _run_and_compare(sbd, w, scale=0.05)


def test_cache_len_out_of_range_is_reported(sbd):
    import torch
    w = gen.shrink(BF16, batch=1, block_k=4, n_q_heads=8, n_kv_heads=2, cache_len=64)
    d = gen.attention_inputs(w, 0, poison_tail=False)
    t = {x: to_dev(d[x], "bf16") for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    lens = torch.tensor([65], dtype=torch.int32, device="cuda")     # > Lmax: clamped
    sbd.sbd_block_attention(t["q"], t["k_cache"], t["v_cache"], lens, t["k_blk"], t["v_blk"])
    assert sbd.sbd_device_error() & sbd.SBD_DEVERR_CACHE_LEN
    assert sbd.sbd_device_error() == 0


@pytest.mark.parametrize("name", ["llama8b_k16", "ragged_b32_k8", "qwen8b_long_k16"])
def test_full_size_configs(sbd, name):
    _run_and_compare(sbd, gen.get_workload(name), seed=0)


@pytest.mark.parametrize("k", [4, 8, 16, 32])
def test_sweep_layer(sbd, k):
    """One layer of the 32-layer sweep at each of its block sizes (k = 32:
    128 packed rows per KV head; k = 4: 16, the register-accumulator
    kernel), batch 16, cache 8192."""
    _run_and_compare(sbd, gen.sweep_workload(k), seed=k)


@pytest.mark.parametrize("k,L,splits", [(8, 8192, 0), (8, 8192, 13), (16, 4096, 0), (32, 2048, 3),
                                        (4, 4096, 0), (12, 1000, 7)])
def test_repeated_calls_leave_no_device_error(sbd, k, L, splits):
    """Back-to-back launches (as in a decode loop) of the same call: every
    bounded wait inside the kernels must succeed, and the result must not
    change between repetitions."""
    import torch
    w = gen.shrink(BF16, batch=16, block_k=k, cache_len=L)
    d = gen.attention_inputs(w, seed=3, poison_tail=False)
    t = {x: to_dev(d[x], "bf16") for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    lens = torch.from_numpy(d["cache_len"]).cuda()
    out0 = sbd.sbd_block_attention(t["q"], t["k_cache"], t["v_cache"], lens, t["k_blk"], t["v_blk"],
                                   num_splits=splits)
    ref = out0.clone()
    for _ in range(30):
        sbd.sbd_block_attention(t["q"], t["k_cache"], t["v_cache"], lens, t["k_blk"], t["v_blk"],
                                out0, num_splits=splits)
    torch.cuda.synchronize()
    assert sbd.sbd_device_error() == 0
    assert torch.equal(out0, ref)


@pytest.mark.parametrize("G,k,splits", [(4, 16, 0), (4, 16, 3), (4, 32, 0), (4, 32, 2), (4, 8, 0),
                                        (1, 16, 1)])
def test_growing_scores_take_the_rescale_path(sbd, G, k, splits):
    """Scores that grow along the cache (keys scaled up to 7x toward the end,
    queries 4x): every row's running maximum jumps by more than the lazy
    rescale threshold many times, at different tiles for different rows of a
    warp, so the O rescale runs and must stay exact."""
    import torch
    Hkv = 2
    w = gen.shrink(BF16, batch=2, block_k=k, n_q_heads=G * Hkv, n_kv_heads=Hkv,
                   cache_len=(900, 1500))
    d = dict(gen.attention_inputs(w, seed=G * 13 + k, poison_tail=False))
    q = gen.bf16_bits_to_f32(d["q"]) * 4.0
    kc = gen.bf16_bits_to_f32(d["k_cache"])
    ramp = (1.0 + 6.0 * np.arange(kc.shape[1]) / kc.shape[1]).astype(np.float32)
    kc = kc * ramp[None, :, None, None]
    d["q"] = gen.f32_to_bf16_bits(q)
    d["k_cache"] = gen.f32_to_bf16_bits(kc)
    t = {x: to_dev(d[x], "bf16") for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    lens = torch.from_numpy(d["cache_len"]).cuda()
    out = sbd.sbd_block_attention(t["q"], t["k_cache"], t["v_cache"], lens, t["k_blk"],
                                  t["v_blk"], num_splits=splits)
    got = out.float().cpu().numpy()
    f = {x: oracle.widen(d[x], "bf16") for x in ("q", "k_cache", "v_cache", "k_blk", "v_blk")}
    ref = oracle.block_attention(f["q"], f["k_cache"], f["v_cache"], d["cache_len"], f["k_blk"],
                                 f["v_blk"])
    assert np.isfinite(got).all()
    assert float(np.abs(got - ref).max()) <= BF16_ATTN_TOL
    assert sbd.sbd_device_error() == 0


@pytest.mark.parametrize("k,G", [(8, 4), (4, 4), (16, 4)])
def test_multi_wave_launch_takes_sequences_longest_first(sbd, k, G):
    """40 sequences x 8 KV heads = 320 CTAs, more than one wave: the CTAs
    take the sequences in descending length, ties by index (lengths with
    repeats and zeros here); every output must still land in its own row."""
    rng = np.random.default_rng(k)
    lens = rng.choice([0, 1, 63, 64, 65, 200, 333, 500], size=40).astype(np.int32)
    lens[[3, 17, 29]] = 333                                  # ties
    w = gen.shrink(BF16, batch=40, block_k=k, n_q_heads=8 * G, n_kv_heads=8,
                   cache_len=(0, 512))
    _run_and_compare(sbd, w, seed=k, lens=lens.tolist())
