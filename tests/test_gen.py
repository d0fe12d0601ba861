"""Pins of the seeded synthetic-input generator (CPU only).

Every parity result stands on these arrays, so the generator is checked
against definitions that do not come from itself: the bf16 rounding against
exact nearest-even rounding worked out in float64 and against PyTorch's
conversion; thread-count invariance of every draw; the moments and
distributions the workload recipes state (N(0,1), N(0, 0.02^2),
log-uniform row scales, standard Gumbel); and the block state and cache
lengths against their stated ranges."""
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest

import gen
import gen.synth as synth

scipy_stats = pytest.importorskip("scipy.stats")


# ------------------------------------------------------------ bf16 rounding

def _nearest_even_bf16(x32: np.ndarray) -> np.ndarray:
    """Round-to-nearest-even to bf16 by its definition: of the two bf16
    values that bracket x (truncation and the next value away from zero),
    take the nearer one exactly in float64, and on an exact tie the one
    with an even last mantissa bit.  Finite inputs only."""
    bits = x32.view(np.uint32)
    lo = (bits >> 16).astype(np.uint32)                  # truncation toward zero
    hi = lo + 1                                          # next bf16 away from zero
    x = x32.astype(np.float64)
    v_lo = (lo << 16).view(np.float32).astype(np.float64)
    v_hi = (hi << 16).astype(np.uint32).view(np.float32).astype(np.float64)
    # hi may step into the inf encoding; its value is then the overflow limit
    top = (hi & 0x7FFF) == 0x7F80
    limit = np.where(bits >> 31, -1.0, 1.0) * 2.0 ** 128
    v_hi = np.where(top, limit, v_hi)
    d_lo = np.abs(x - v_lo)
    d_hi = np.abs(v_hi - x)
    take_hi = (d_hi < d_lo) | ((d_hi == d_lo) & ((lo & 1) == 1))
    return np.where(take_hi, hi, lo).astype(np.uint16)


def _edge_values() -> np.ndarray:
    rng = np.random.default_rng(5)
    upper = np.arange(1 << 16, dtype=np.uint32)
    lowers = np.array([0, 1, 0x7FFF, 0x8000, 0x8001, 0xFFFF], dtype=np.uint32)
    cols = [(upper << 16) | l for l in lowers]
    cols.append((upper << 16) | rng.integers(0, 1 << 16, upper.shape[0], dtype=np.uint32))
    return np.concatenate(cols).view(np.float32)


def test_bf16_rounding_is_nearest_even():
    x = _edge_values()
    finite = np.isfinite(x)
    got = gen.f32_to_bf16_bits(x)
    want = _nearest_even_bf16(x[finite])
    assert np.array_equal(got[finite], want)


def test_bf16_rounding_matches_torch_on_non_nan():
    torch = pytest.importorskip("torch")
    x = _edge_values()
    keep = ~np.isnan(x)
    t = torch.from_numpy(x[keep]).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(gen.f32_to_bf16_bits(x[keep]), t)


def test_bf16_specials():
    cases = {
        0x00000000: 0x0000, 0x80000000: 0x8000,          # +-0
        0x7F800000: 0x7F80, 0xFF800000: 0xFF80,          # +-inf
        0x7F7FFFFF: 0x7F80, 0xFF7FFFFF: 0xFF80,          # largest finite rounds to inf
        0x7F7F7FFF: 0x7F7F,                              # largest finite bf16 stays
        0x00000001: 0x0000, 0x00008000: 0x0000,          # subnormal tie -> even (0)
        0x00018000: 0x0002, 0x00008001: 0x0001,          # subnormal tie up / above half
        0x3F808000: 0x3F80, 0x3F818000: 0x3F82,          # normal ties to even
    }
    x = np.array(list(cases), dtype=np.uint32).view(np.float32)
    got = gen.f32_to_bf16_bits(x)
    assert [int(v) for v in got] == list(cases.values())


def test_bf16_nan_stays_nan_with_its_sign():
    x = np.array([0x7FC00000, 0xFFC00000, 0x7F800001, 0xFF812345, 0x7FA00000],
                 dtype=np.uint32).view(np.float32)
    got = gen.f32_to_bf16_bits(x).astype(np.uint32)
    assert np.all((got & 0x7F80) == 0x7F80) and np.all((got & 0x007F) != 0)
    assert list(got >> 15) == [0, 1, 0, 1, 0]
    assert np.isnan(gen.bf16_bits_to_f32(got.astype(np.uint16))).all()


def test_bf16_widening_is_exact():
    b = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    f = gen.bf16_bits_to_f32(b)
    fin = np.isfinite(f)
    assert np.array_equal(gen.f32_to_bf16_bits(f[fin]), b[fin])


# ------------------------------------------------ thread-count invariance

def _with_workers(monkeypatch, n, fn):
    pool = ThreadPoolExecutor(max_workers=n)
    monkeypatch.setattr(synth, "_POOL", pool)
    try:
        return fn()
    finally:
        pool.shutdown()
        monkeypatch.setattr(synth, "_POOL", None)


@pytest.mark.parametrize("draw", [
    lambda: gen.normal_f32((3, synth.CHUNK + 12345), 4, "t", "normal"),
    lambda: gen.gumbel_f32((2 * synth.CHUNK + 7,), 4, "t", "gumbel"),
    lambda: gen.uniform_open01_f64((synth.CHUNK + 3,), 4, "t", "u"),
    lambda: gen.f32_to_bf16_bits(gen.normal_f32((synth.CHUNK * 2 + 5,), 9, "t", "b")),
])
def test_draws_do_not_depend_on_thread_count(monkeypatch, draw):
    one = _with_workers(monkeypatch, 1, draw)
    many = _with_workers(monkeypatch, 8, draw)
    assert one.tobytes() == many.tobytes()
    again = _with_workers(monkeypatch, 3, draw)
    assert one.tobytes() == again.tobytes()


def test_workload_tensors_do_not_depend_on_thread_count(monkeypatch):
    w = gen.shrink(gen.get_workload("ragged_b32_k8"), batch=4, cache_len=(512, 6000), vocab=70000,
                   hidden=128)

    def draw():
        d = gen.step_inputs(w, seed=3, step=2)
        return b"".join(np.ascontiguousarray(d[x]).tobytes() for x in sorted(d))

    assert _with_workers(monkeypatch, 1, draw) == _with_workers(monkeypatch, 8, draw)


def test_seeds_keys_and_steps_give_different_streams():
    a = gen.normal_f32((1000,), 0, "x", "y")
    assert np.array_equal(a, gen.normal_f32((1000,), 0, "x", "y"))
    assert not np.array_equal(a, gen.normal_f32((1000,), 1, "x", "y"))
    assert not np.array_equal(a, gen.normal_f32((1000,), 0, "x", "z"))
    w = gen.get_workload("tiny_f32")
    assert not np.array_equal(gen.hidden_states(w, 0, 0), gen.hidden_states(w, 0, 1))
    assert not np.array_equal(gen.gumbel_noise(w, 0, 0), gen.gumbel_noise(w, 0, 1))
    # chunks of one tensor are separate streams, not one stream repeated
    big = gen.normal_f32((2 * synth.CHUNK,), 0, "x")
    assert not np.array_equal(big[:1000], big[synth.CHUNK:synth.CHUNK + 1000])


# ------------------------------------------------------- distributions

def _ks(x, cdf):
    return scipy_stats.kstest(np.asarray(x, np.float64), cdf).pvalue


def test_normal_draws_are_standard_normal():
    x = gen.normal_f32((400_000,), 11, "t", "n")
    assert abs(x.mean()) < 5 / np.sqrt(x.size)
    assert abs(x.var() - 1.0) < 5 * np.sqrt(2.0 / x.size)
    assert _ks(x[:50_000], "norm") > 1e-4


def test_lm_head_weight_is_normal_with_stated_std():
    w = gen.shrink(gen.get_workload("llama8b_k16"), vocab=1000, hidden=256)
    W = gen.bf16_bits_to_f32(gen.lm_head_weight(w, 0)).astype(np.float64)
    assert W.shape == (1000, 256)
    n = W.size
    assert abs(W.mean()) < 5 * 0.02 / np.sqrt(n)
    # bf16 rounding changes the variance by a relative 2^-18 at most
    assert abs(W.std() / 0.02 - 1.0) < 5 * np.sqrt(0.5 / n) + 1e-4
    assert _ks(W.reshape(-1)[:50_000] / 0.02, "norm") > 1e-4


def test_hidden_scales_are_log_uniform():
    w = gen.shrink(gen.get_workload("llama8b_k16"), batch=400, block_k=32)
    s = gen.hidden_scales(w, 0, 0).astype(np.float64)
    assert s.shape == (400, 32)
    assert s.min() >= 0.1 * (1 - 1e-6) and s.max() <= 10.0 * (1 + 1e-6)
    lo, hi = np.log(0.1), np.log(10.0)
    assert _ks(np.log(s).ravel(), scipy_stats.uniform(lo, hi - lo).cdf) > 1e-4


def test_hidden_rows_are_normal_times_their_scale():
    w = gen.shrink(gen.get_workload("tiny_f32"), batch=3, block_k=5, hidden=4096)
    h = gen.hidden_states(w, 2, 1).astype(np.float64)
    s = gen.hidden_scales(w, 2, 1).astype(np.float64)
    z = h / s[:, :, None]
    # each row divided by its own scale is N(0,1): its rms is 1 within 4 sigma
    rms = np.sqrt((z ** 2).mean(axis=2))
    assert np.all(np.abs(rms - 1.0) < 4 * np.sqrt(0.5 / 4096))
    assert _ks(z.ravel()[:40_000], "norm") > 1e-4


def test_gumbel_draws_are_standard_gumbel():
    g = gen.gumbel_f32((300_000,), 7, "t", "g").astype(np.float64)
    euler_gamma = 0.5772156649015329
    assert abs(g.mean() - euler_gamma) < 5 * (np.pi / np.sqrt(6)) / np.sqrt(g.size)
    assert abs(g.var() - np.pi ** 2 / 6) < 0.03
    assert _ks(g[:50_000], "gumbel_r") > 1e-4
    assert np.isfinite(g).all()


def test_uniforms_are_inside_the_open_interval():
    u = gen.uniform_open01_f64((200_000,), 3, "t", "u")
    assert (u > 0).all() and (u < 1).all()
    assert abs(u.mean() - 0.5) < 5 * np.sqrt(1 / 12 / u.size)
    assert _ks(u[:50_000], "uniform") > 1e-4


# ------------------------------------------------ block state and lengths

@pytest.mark.parametrize("name", ["tiny_f32", "llama8b_k16", "ragged_b32_k8", "sweep32_k32"])
def test_block_state_masks_exactly_the_undecoded_positions(name):
    w = gen.get_workload(name)
    for seed in range(5):
        bt, m = gen.block_state(w, seed)
        assert bt.shape == m.shape == (w.batch, w.block_k)
        assert bt.dtype == np.int32 and m.dtype == np.uint8
        assert np.array_equal(bt == gen.MASK_TOKEN, m.astype(bool))
        assert ((bt[~m.astype(bool)] >= 0) & (bt[~m.astype(bool)] < w.vocab)).all()
        n_dec = (m == 0).sum(axis=1)
        # the decoded positions are the leading ones
        for b in range(w.batch):
            assert not m[b, :n_dec[b]].any() and m[b, n_dec[b]:].all()
        kind = w.decoded[0]
        if kind == "fixed":
            assert (n_dec == w.decoded[1]).all()
        else:
            assert (n_dec >= w.decoded[1]).all() and (n_dec <= w.decoded[2]).all()


def test_ragged_decoded_counts_cover_their_range():
    w = gen.get_workload("ragged_b32_k8")
    seen = set()
    for seed in range(8):
        _, m = gen.block_state(w, seed)
        seen |= set(((m == 0).sum(axis=1)).tolist())
    assert seen == set(range(1, 8))


def test_cache_lengths_and_poisoned_tails():
    w = gen.shrink(gen.get_workload("ragged_b32_k8"), hidden=64, vocab=100)
    lens = gen.cache_lengths(w, 0)
    assert lens.dtype == np.int32 and lens.shape == (32,)
    assert (lens >= 512).all() and (lens <= 2048).all()
    assert len(set(lens.tolist())) > 20
    d = gen.attention_inputs(gen.shrink(w, batch=4), 0, 0, poison_tail=True)
    kc = gen.bf16_bits_to_f32(d["k_cache"])
    for b in range(4):
        L = int(d["cache_len"][b])
        assert np.isfinite(kc[b, :L]).all() and np.isnan(kc[b, L:]).all()
    d2 = gen.attention_inputs(gen.shrink(w, batch=4), 0, 0, poison_tail=False)
    assert np.isfinite(gen.bf16_bits_to_f32(d2["v_cache"])).all()
    assert np.array_equal(d["q"], d2["q"])


def test_fixed_lengths_fill_the_cache():
    w = gen.get_workload("qwen8b_long_k16")
    assert (gen.cache_lengths(w, 0) == 32768).all()
