"""Counter-based Gumbel noise on the GPU against the oracle's Philox4x32-10
(philox_gumbel): the noise tensor within fp32 rounding of the fp64 transform;
the LM-head call with in-kernel noise bit-identical to the buffer call fed
the same noise tensor, and its tokens equal to the oracle's except at
near-ties of the score."""
import numpy as np
import pytest

import gen
import oracle
from tests.helpers import ENTROPY_TOL, cached_weight, to_dev, token_tolerance, top2_gap

pytestmark = pytest.mark.gpu

NOISE_TOL = 1e-5       # absolute, g = -ln(-ln u) in fp32 with |g| < 17


@pytest.fixture(scope="module")
def sbd():
    import paper_2509_04185_gb300 as m
    return m


@pytest.mark.parametrize("rows,V", [([0, 1, 2, 3], 4096), ([5, 77, 511], 1003), ([12], 151936)])
@pytest.mark.parametrize("seed,offset", [(0, 0), (0xDEADBEEF12345678, (3 << 32) + 17)])
def test_noise_tensor_matches_oracle(sbd, rows, V, seed, offset):
    import torch
    ids = torch.tensor(rows, dtype=torch.int32, device="cuda")
    g = sbd.sbd_gumbel_philox(ids, V, seed, offset).cpu().numpy()
    ref, _ = oracle.philox_gumbel(rows, V, seed, offset)
    assert np.isfinite(g).all()
    assert np.abs(g - ref).max() < NOISE_TOL


def _case(B, k, V, H, dtype, seed, n_masked=None):
    w = gen.shrink(gen.get_workload("llama8b_k16"), batch=B, block_k=k, vocab=V, hidden=H,
                   dtype=dtype)
    rng = np.random.default_rng(seed)
    if n_masked is None:
        masked = (rng.uniform(size=(B, k)) < 0.7).astype(np.uint8)
        masked[0, -1] = 1
    else:
        masked = np.zeros(B * k, dtype=np.uint8)
        masked[rng.choice(B * k, size=n_masked, replace=False)] = 1
        masked = masked.reshape(B, k)
    return {"w": cached_weight(V, H, dtype, seed), "hidden": gen.hidden_states(w, seed, 0),
            "masked": masked}


@pytest.mark.parametrize("B,k,V,H,dtype", [(1, 16, 4096 + 5, 512, "bf16"), (2, 16, 40000, 1024, "bf16"),
                                           (16, 32, 1500, 128, "bf16"), (3, 7, 777, 64, "bf16"),
                                           (2, 8, 2000, 128, "f32"),
                                           (1, 16, 128256, 4096, "bf16")])
@pytest.mark.parametrize("tau", [1.0, 0.3])
def test_head_with_philox_noise(sbd, B, k, V, H, dtype, tau):
    _check_philox_head(sbd, _case(B, k, V, H, dtype, seed=B * 7 + k), B, k, V, H, dtype, tau)


@pytest.mark.parametrize("R", [100, 150, 200, 300])
def test_head_with_philox_noise_row_counts(sbd, R):
    """Exactly R of 512 rows masked: the CTA-pair kernel's vocabulary-lane
    layout (R <= 160), its row-lane layout with one row group (161..256)
    and with two (above 256)."""
    B, k, V, H = 16, 32, 3001, 256
    _check_philox_head(sbd, _case(B, k, V, H, "bf16", seed=R, n_masked=R), B, k, V, H, "bf16", 1.0)


def _check_philox_head(sbd, d, B, k, V, H, dtype, tau):
    import torch
    seed, offset = 1234567 + B, 99 + k
    hid = to_dev(d["hidden"], dtype)
    W = to_dev(d["w"], dtype)
    m = torch.from_numpy(d["masked"]).cuda()
    ent, tok = sbd.sbd_head_entropy_sample_philox(hid, W, m, seed, offset, tau)
    # the same noise as a tensor, through the buffer call: bit-identical results
    ids = torch.arange(B * k, dtype=torch.int32, device="cuda")
    g_dev = sbd.sbd_gumbel_philox(ids, V, seed, offset).view(B, k, V)
    ent_b, tok_b = sbd.sbd_head_entropy_sample(hid, W, m, g_dev, tau)
    assert torch.equal(ent, ent_b) and torch.equal(tok, tok_b)
    # against the oracle with its own fp64 noise
    g_ref, _ = oracle.philox_gumbel(np.arange(B * k), V, seed, offset)
    g_ref = g_ref.reshape(B, k, V)
    rent, rtok, zs = oracle.head_entropy_sample(oracle.widen(d["hidden"], dtype), d["w"], dtype,
                                                d["masked"], g_ref, tau)
    e, t = ent.cpu().numpy(), tok.cpu().numpy()
    mk = d["masked"].astype(bool)
    assert np.abs(e[mk] - rent[mk]).max() <= ENTROPY_TOL
    assert (t[~mk] == -1).all()
    acc = H // (16 if dtype == "bf16" else 1)
    exempt = 0
    for (b, i), z in zs.items():
        if t[b, i] == rtok[b, i]:
            continue
        gap = top2_gap(z, g_ref[b, i], tau)
        assert gap < token_tolerance(z, acc) + tau * 2 * NOISE_TOL, (b, i, gap)
        exempt += 1
    assert exempt <= max(1, len(zs) // 20)


def test_fresh_offsets_give_fresh_samples(sbd):
    import torch
    d = _case(1, 16, 4096, 256, "bf16", seed=3)
    hid, W = to_dev(d["hidden"], "bf16"), to_dev(d["w"], "bf16")
    m = torch.ones(1, 16, dtype=torch.uint8, device="cuda")
    toks = [sbd.sbd_head_entropy_sample_philox(hid, W, m, 7, off, 1.0)[1].cpu().numpy()
            for off in range(4)]
    assert any(not np.array_equal(toks[0], x) for x in toks[1:])
    again = sbd.sbd_head_entropy_sample_philox(hid, W, m, 7, 0, 1.0)[1].cpu().numpy()
    assert np.array_equal(toks[0], again)                       # same counter, same sample
