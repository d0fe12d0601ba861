"""The no-allocation LM-head entry point, for callers that cannot allocate
device memory (a framework owning the whole device pool, a loop that cannot
take cudaMalloc's synchronisation, a plug-in without an allocator).

It is called through the C ABI on two consecutive calls -- the second one
finds the shared scratch array holding the first call's contents -- and its
outputs are compared with those of sbd_head_entropy_sample given a caller
workspace, at the tolerance of the other LM-head tests (entropy 1e-3 nats,
tokens exact).  This file is collected last so that a run stopping at the
first failure has run every other test before it."""
import ctypes

import numpy as np
import pytest

import gen
from tests.helpers import ENTROPY_TOL, step_inputs, to_dev


@pytest.fixture(scope="module")
def sbd():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2509_04185_gb300 as m
    return m


def test_oversized_shape_is_rejected_before_any_launch(sbd):
    # fp32, 256 rows of 16384 hidden: 16 MiB of compacted rows > 8 MiB scratch
    d = sbd.HeadDesc(16, 16, 16384, 512, sbd.SBD_DTYPE_F32)
    a = 1 << 20                                   # never dereferenced
    st = sbd.lib.sbd_head_entropy_sample_noalloc(ctypes.byref(d), a, a, a, a, 1.0, a, a, None)
    assert st == sbd.SBD_ERR_UNSUPPORTED
    assert b"no-allocation" in sbd.lib.sbd_last_error()


@pytest.mark.gpu
@pytest.mark.parametrize("name,over", [
    ("llama8b_k16", dict(vocab=8192 + 11, cache_len=64)),
    ("tiny_f32", {}),
    ("llama8b_k16", dict(batch=16, block_k=16, vocab=3000, hidden=512, cache_len=64,
                         decoded=("uniform", 0, 15))),
])
def test_noalloc_matches_workspace_call(sbd, name, over):
    import torch
    w = gen.shrink(gen.get_workload(name), **over)
    dt = w.dtype
    d = step_inputs(w, seed=3)
    hid, W = to_dev(d["hidden"], dt), to_dev(d["w"], dt)
    masked = torch.from_numpy(d["masked"]).cuda()
    g = torch.from_numpy(d["gumbel"]).cuda()
    B, k = d["masked"].shape
    ref_e, ref_t = sbd.sbd_head_entropy_sample(hid, W, masked, g, 1.0)
    ref_e, ref_t = ref_e.cpu().numpy(), ref_t.cpu().numpy()
    desc = sbd.head_desc(hid, W)
    stream = torch.cuda.current_stream().cuda_stream
    assert sbd.lib.sbd_head_entropy_sample_workspace_size(ctypes.byref(desc)) <= \
        sbd.SBD_HEAD_NOALLOC_MAX_SCRATCH
    for call in range(2):
        ent = torch.full((B, k), -7.0, dtype=torch.float32, device="cuda")
        tok = torch.full((B, k), -7, dtype=torch.int32, device="cuda")
        st = sbd.lib.sbd_head_entropy_sample_noalloc(
            ctypes.byref(desc), hid.data_ptr(), W.data_ptr(), masked.data_ptr(), g.data_ptr(),
            ctypes.c_float(1.0), ent.data_ptr(), tok.data_ptr(), stream)
        assert st == sbd.SBD_OK, sbd.lib.sbd_last_error()
        torch.cuda.synchronize()
        e, t = ent.cpu().numpy(), tok.cpu().numpy()
        m = d["masked"].astype(bool)
        assert np.all(np.isinf(e[~m])) and np.all(t[~m] == -1)
        assert np.abs(e[m] - ref_e[m]).max(initial=0.0) <= ENTROPY_TOL, call
        np.testing.assert_array_equal(t, ref_t)
    assert sbd.sbd_device_error() == 0


@pytest.mark.gpu
def test_noalloc_after_a_larger_call(sbd):
    """The shared array keeps the previous call's contents: a larger call
    (more masked rows, larger vocabulary, so more compacted rows, a longer
    row map and more per-CTA partials) followed by a smaller one must leave
    nothing of the first in the second's results."""
    import torch
    big = gen.shrink(gen.get_workload("llama8b_k16"), batch=16, block_k=16, vocab=20000,
                     hidden=512, cache_len=64, decoded=("fixed", 0))
    small = gen.shrink(gen.get_workload("llama8b_k16"), batch=3, block_k=8, vocab=2500,
                       hidden=512, cache_len=64, decoded=("uniform", 0, 7))
    stream = torch.cuda.current_stream().cuda_stream
    results = []
    for w in (big, small):
        d = step_inputs(w, seed=11)
        hid, W = to_dev(d["hidden"], "bf16"), to_dev(d["w"], "bf16")
        masked = torch.from_numpy(d["masked"]).cuda()
        g = torch.from_numpy(d["gumbel"]).cuda()
        B, k = d["masked"].shape
        desc = sbd.head_desc(hid, W)
        ent = torch.full((B, k), -7.0, dtype=torch.float32, device="cuda")
        tok = torch.full((B, k), -7, dtype=torch.int32, device="cuda")
        st = sbd.lib.sbd_head_entropy_sample_noalloc(
            ctypes.byref(desc), hid.data_ptr(), W.data_ptr(), masked.data_ptr(), g.data_ptr(),
            ctypes.c_float(1.0), ent.data_ptr(), tok.data_ptr(), stream)
        assert st == sbd.SBD_OK, sbd.lib.sbd_last_error()
        # the same call with a fresh workspace of its own
        ref_e, ref_t = sbd.sbd_head_entropy_sample(hid, W, masked, g, 1.0)
        torch.cuda.synchronize()
        results.append((d["masked"].astype(bool), ent.cpu().numpy(), tok.cpu().numpy(),
                        ref_e.cpu().numpy(), ref_t.cpu().numpy()))
    m, e, t, re_, rt = results[1]
    assert m.sum() < results[0][0].sum()
    assert np.all(np.isinf(e[~m])) and np.all(t[~m] == -1)
    assert np.abs(e[m] - re_[m]).max(initial=0.0) <= ENTROPY_TOL
    np.testing.assert_array_equal(t, rt)
    assert sbd.sbd_device_error() == 0
