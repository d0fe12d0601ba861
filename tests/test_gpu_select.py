"""Selection rules of the Appendix "Sampling algorithm" on the GPU against the
oracle: the select kernel fed the same fp32 entropies and confidences as the
oracle (accepted sets exact, except where the oracle's fp64 decision sits
within a margin of the threshold), and the confidence output of the LM-head
call against the oracle's max softmax."""
import numpy as np
import pytest

import gen
import oracle
from tests.helpers import GAMMA_MARGIN, cached_weight, to_dev

pytestmark = pytest.mark.gpu

CONF_TOL = 1e-3          # absolute, confidence in [0, 1] (as the entropy tolerance in nats)


@pytest.fixture(scope="module")
def sbd():
    import paper_2509_04185_gb300 as m
    return m


def _rules(sbd):
    return {sbd.SBD_SELECT_EB_ENTROPY: "eb_entropy",
            sbd.SBD_SELECT_EB_CONFIDENCE: "eb_confidence",
            sbd.SBD_SELECT_FACTOR: "factor",
            sbd.SBD_SELECT_FACTOR_COMPLEMENT: "factor_complement"}


def _run(sbd, rule, ent, conf, tok, masked, bt, thr):
    import torch
    e = torch.from_numpy(ent.astype(np.float32)).cuda()
    c = None if conf is None else torch.from_numpy(conf.astype(np.float32)).cuda()
    t = torch.from_numpy(tok.astype(np.int32)).cuda()
    m = torch.from_numpy(masked.astype(np.uint8)).cuda()
    b = torch.from_numpy(bt.astype(np.int32)).cuda()
    n = sbd.sbd_select(rule, e, c, t, thr, m, b)
    return m.cpu().numpy(), b.cpu().numpy(), n.cpu().numpy()


def _decision_margins(name, H_order, C_order, thr):
    """|lhs_n - threshold| of the oracle's test at every rank n (1-based)."""
    out = []
    total, top = 0.0, -np.inf
    for n in range(1, len(H_order) + 1):
        if name == "eb_confidence":
            total += float(H_order[n - 1])
            top = max(top, float(H_order[n - 1]))
            out.append(abs(total - top - thr) if n >= 2 else np.inf)
        elif name == "eb_entropy":
            out.append(abs(sum(float(h) for h in H_order[: n - 1]) - thr) if n >= 2 else np.inf)
        else:
            c = float(C_order[n - 1])
            lhs = (n + 1) * ((1.0 - c) if name == "factor_complement" else c)
            out.append(abs(lhs - thr))
    return out


def _check(name, ent32, conf32, tok, masked, bt, thr, gm, gb, gn):
    ent = np.where(masked.astype(bool), ent32.astype(np.float64), np.inf)
    conf = np.where(masked.astype(bool), conf32.astype(np.float64), 0.0)
    thr = float(np.float32(thr))                 # the threshold the kernel receives
    rm, rb, rn, acc, orders = oracle.select_step(ent, conf, tok, masked, bt, name, thr)
    exempt = 0
    for b in range(masked.shape[0]):
        if np.array_equal(gm[b], rm[b]) and np.array_equal(gb[b], rb[b]) and gn[b] == rn[b]:
            continue
        order = orders[b]
        margins = _decision_margins(name, [ent[b, i] for i in order],
                                    [conf[b, i] for i in order], thr)
        assert min(margins) < GAMMA_MARGIN, (name, b, gn[b], rn[b], margins)
        # whatever the count, the set is a prefix of the oracle's order
        got = {i for i in range(masked.shape[1]) if masked[b, i] and not gm[b, i]}
        assert got == set(order[: int(gn[b])])
        exempt += 1
    return exempt


@pytest.mark.parametrize("k", [1, 3, 8, 16, 31, 32])
@pytest.mark.parametrize("B", [1, 7, 130])
def test_random_inputs_every_rule(sbd, B, k):
    rng = np.random.default_rng(1000 * B + k)
    exempt = 0
    cases = 0
    for rule, name in _rules(sbd).items():
        thresholds = [0.0, 0.05, 0.3, 1.0, 2.5] if name.startswith("eb") else \
            [0.5, 1.3, 2.0, 3.7, 9.0]
        for thr in thresholds:
            ent32 = rng.exponential(float(rng.uniform(0.05, 1.0)), (B, k)).astype(np.float32)
            conf32 = rng.uniform(0.0, 1.0, (B, k)).astype(np.float32)
            masked = (rng.uniform(size=(B, k)) < 0.75).astype(np.uint8)
            masked[0] = 1
            tok = rng.integers(0, 151936, (B, k)).astype(np.int32)
            bt = np.where(masked.astype(bool), -1, rng.integers(0, 151936, (B, k))).astype(np.int32)
            # values at unmasked positions must not be read: poison them
            ent_in = np.where(masked.astype(bool), ent32, np.float32(-7.0))
            conf_in = np.where(masked.astype(bool), conf32, np.float32(5.0))
            gm, gb, gn = _run(sbd, rule, ent_in, conf_in, tok, masked, bt, thr)
            exempt += _check(name, ent32, conf32, tok, masked, bt, thr, gm, gb, gn)
            cases += B
    assert exempt <= max(2, cases // 100)


def test_worked_examples(sbd):
    # confidence order 3, 0, 2, 1; entropies in that order 0.05, 0.2, 0.5, 2.0
    H = np.array([[0.2, 2.0, 0.5, 0.05]], dtype=np.float32)
    C = np.array([[0.9, 0.5, 0.8, 0.99]], dtype=np.float32)
    tok = np.array([[10, 11, 12, 13]], dtype=np.int32)
    masked = np.ones((1, 4), dtype=np.uint8)
    bt = np.full((1, 4), -1, dtype=np.int32)
    gm, gb, gn = _run(sbd, sbd.SBD_SELECT_EB_CONFIDENCE, H, C, tok, masked, bt, 0.3)
    assert gn[0] == 3 and list(gm[0]) == [0, 1, 0, 0] and list(gb[0]) == [10, -1, 12, 13]
    gm, gb, gn = _run(sbd, sbd.SBD_SELECT_EB_CONFIDENCE, H, C, tok, masked, bt, 0.0)
    assert gn[0] == 1 and list(gm[0]) == [1, 1, 1, 0]
    # (n + 1) c^n = 1.98, 2.7, 3.2, 2.5
    for f, s in ((2.0, 1), (2.6, 4), (1.5, 1)):
        gm, gb, gn = _run(sbd, sbd.SBD_SELECT_FACTOR, H, C, tok, masked, bt, f)
        assert gn[0] == s, f
    # (n + 1)(1 - c^n) = 0.02, 0.3, 0.8, 2.5
    for f, s in ((1.0, 3), (0.5, 2), (0.01, 1)):
        gm, gb, gn = _run(sbd, sbd.SBD_SELECT_FACTOR_COMPLEMENT, H, C, tok, masked, bt, f)
        assert gn[0] == s, f
    # the entropy rule does not read the confidence
    gm, gb, gn = _run(sbd, sbd.SBD_SELECT_EB_ENTROPY, H, None, tok, masked, bt, 0.1)
    assert gn[0] == 2 and list(gm[0]) == [0, 1, 1, 0]


def test_ties_nan_and_empty(sbd):
    H = np.full((3, 5), 0.1, dtype=np.float32)
    C = np.array([[0.5, 0.7, 0.5, 0.7, 0.6],
                  [np.nan, 0.9, 0.8, 0.7, 0.6],
                  [0.9, 0.9, 0.9, 0.9, 0.9]], dtype=np.float32)
    tok = np.arange(15, dtype=np.int32).reshape(3, 5)
    masked = np.array([[1, 1, 1, 1, 1], [1, 1, 1, 1, 1], [0, 0, 0, 0, 0]], dtype=np.uint8)
    bt = np.where(masked.astype(bool), -1, 3).astype(np.int32)
    # factor with f = 1.5: (n + 1) c^n = 1.4 at n = 1 only -> one token, the
    # lower position among the two 0.7s
    gm, gb, gn = _run(sbd, sbd.SBD_SELECT_FACTOR, H, C, tok, masked, bt, 1.5)
    assert list(gn) == [1, 1, 0] and list(gm[0]) == [1, 0, 1, 1, 1]
    # a NaN confidence sorts last and never passes the Factor test
    gm, gb, gn = _run(sbd, sbd.SBD_SELECT_FACTOR, H, C, tok, masked, bt, 100.0)
    assert gn[1] == 4 and gm[1][0] == 1
    assert list(gb[2]) == [3] * 5 and (gm[2] == 0).all()


def _head_case(B, k, V, Hd, dtype, seed):
    w = gen.shrink(gen.get_workload("llama8b_k16"), batch=B, block_k=k, vocab=V, hidden=Hd,
                   dtype=dtype)
    d = {"w": cached_weight(V, Hd, dtype, seed), "hidden": gen.hidden_states(w, seed, 0),
         "gumbel": gen.gumbel_noise(w, seed, 0)}
    rng = np.random.default_rng(seed)
    d["masked"] = (rng.uniform(size=(B, k)) < 0.8).astype(np.uint8)
    d["masked"][0, 0] = 1
    return d


@pytest.mark.parametrize("B,k,V,Hd,dtype", [(1, 16, 4096 + 5, 512, "bf16"),
                                             (4, 16, 3000, 256, "bf16"),
                                             (2, 8, 2000, 128, "f32")])
def test_head_confidence_matches_oracle(sbd, B, k, V, Hd, dtype):
    import torch
    d = _head_case(B, k, V, Hd, dtype, seed=B + k)
    hid = to_dev(d["hidden"], dtype)
    W = to_dev(d["w"], dtype)
    m = torch.from_numpy(d["masked"]).cuda()
    g = torch.from_numpy(d["gumbel"]).cuda()
    ent, conf, tok = sbd.sbd_head_entropy_confidence_sample(hid, W, m, g, 1.0)
    ent2, tok2 = sbd.sbd_head_entropy_sample(hid, W, m, g, 1.0)
    # the same kernels: entropy and token bit-identical to the plain call
    assert torch.equal(ent, ent2) and torch.equal(tok, tok2)
    hid64 = oracle.widen(d["hidden"], dtype)
    _, _, _, conf_ref = oracle.head_entropy_sample(hid64, d["w"], dtype, d["masked"],
                                                   d["gumbel"], 1.0, with_confidence=True)
    c = conf.cpu().numpy()
    mk = d["masked"].astype(bool)
    tol = CONF_TOL if dtype == "bf16" else 1e-5
    assert np.abs(c[mk] - conf_ref[mk]).max() < tol
    assert (c[~mk] == 0).all()
    assert ((c[mk] > 0) & (c[mk] <= 1)).all()
