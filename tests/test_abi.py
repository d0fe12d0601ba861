"""The C-ABI library: it builds, loads, exports every symbol include/sbd.h
declares, and rejects bad arguments on the host before touching the GPU
(CPU only: no compute call is made here)."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "sbd.h")


@pytest.fixture(scope="module")
def sbd():
    import __graft_entry__
    __graft_entry__.build()
    import paper_2509_04185_gb300
    return paper_2509_04185_gb300


def _declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    names = re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*(sbd_[a-z_0-9]+)\s*\(", text, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_three_calls():
    names = _declared_functions()
    for n in ("sbd_block_attention", "sbd_head_entropy_sample", "sbd_eb_select"):
        assert n in names


def test_library_exports_every_declared_symbol(sbd):
    names = _declared_functions()
    assert set(names) == set(sbd.EXPORTS)
    for n in names:
        assert hasattr(sbd.lib, n), n
    out = subprocess.run(["nm", "-D", "--defined-only", sbd.LIB_PATH], capture_output=True,
                         text=True).stdout
    exported = set(re.findall(r"\b(sbd_[a-z_0-9]+)\b", out))
    assert set(names) <= exported


def test_no_torch_types_in_the_header():
    text = open(HEADER).read()
    assert "torch" not in text.lower().replace("pytorch", "")
    assert "at::" not in text and "c10" not in text


def test_status_strings(sbd):
    assert sbd.lib.sbd_status_string(0) == b"SBD_OK"
    assert sbd.lib.sbd_status_string(3) == b"SBD_ERR_WORKSPACE"
    assert sbd.lib.sbd_status_string(99) == b"SBD_ERR_UNKNOWN"
    assert sbd.sbd_version() >= 100


def _attn_desc(sbd, **over):
    d = dict(batch=1, block_k=16, n_q_heads=32, n_kv_heads=8, head_dim=128, max_cache_len=4096,
             dtype=sbd.SBD_DTYPE_BF16, scale=0.0, num_splits=0)
    d.update(over)
    return sbd.AttnDesc(**d)


@pytest.mark.parametrize("over,status", [
    (dict(block_k=33), 2), (dict(head_dim=96), 2), (dict(n_q_heads=30), 1),
    (dict(dtype=7), 1), (dict(scale=-1.0), 1), (dict(batch=-1), 1),
    (dict(block_k=0), 1), (dict(n_q_heads=64, n_kv_heads=1), 2), (dict(num_splits=-2), 1),
])
def test_attention_rejects_bad_descriptors(sbd, over, status):
    d = _attn_desc(sbd, **over)
    fake = 1 << 20                       # never dereferenced: rejected first
    st = sbd.lib.sbd_block_attention(ctypes.byref(d), fake, fake, fake, fake, fake, fake, fake,
                                     None, 0, None)
    assert st == status, sbd.lib.sbd_last_error()
    assert sbd.lib.sbd_last_error() != b""


def test_attention_rejects_null_and_misaligned(sbd):
    d = _attn_desc(sbd, dtype=sbd.SBD_DTYPE_F32)
    a = 1 << 20
    st = sbd.lib.sbd_block_attention(ctypes.byref(d), None, a, a, a, a, a, a, None, 0, None)
    assert st == sbd.SBD_ERR_INVALID_ARG and b"q is NULL" in sbd.lib.sbd_last_error()
    st = sbd.lib.sbd_block_attention(ctypes.byref(d), a + 4, a, a, a, a, a, a, None, 0, None)
    assert st == sbd.SBD_ERR_INVALID_ARG and b"aligned" in sbd.lib.sbd_last_error()
    assert sbd.lib.sbd_block_attention(None, a, a, a, a, a, a, a, None, 0, None) == 1


def test_causal_prefix_rejects_bad_arguments(sbd):
    a = 1 << 20
    d = _attn_desc(sbd, block_k=32)
    f = sbd.lib.sbd_block_attention_causal_prefix
    for nc in (-1, 33):
        assert f(ctypes.byref(d), nc, a, a, a, a, a, a, a, None, 0, None) == sbd.SBD_ERR_INVALID_ARG
        assert b"n_causal" in sbd.lib.sbd_last_error()
    d = _attn_desc(sbd, block_k=33)
    assert f(ctypes.byref(d), 4, a, a, a, a, a, a, a, None, 0, None) == sbd.SBD_ERR_UNSUPPORTED
    d = _attn_desc(sbd, head_dim=96)
    assert f(ctypes.byref(d), 4, a, a, a, a, a, a, a, None, 0, None) == sbd.SBD_ERR_UNSUPPORTED
    d = _attn_desc(sbd, dtype=sbd.SBD_DTYPE_F32)
    assert f(ctypes.byref(d), 4, a, None, a, a, a, a, a, None, 0, None) == sbd.SBD_ERR_INVALID_ARG


def test_head_rejects_bad_arguments(sbd):
    a = 1 << 20
    d = sbd.HeadDesc(32, 17, 4096, 128256, sbd.SBD_DTYPE_BF16)      # 544 rows > 512
    assert sbd.lib.sbd_head_entropy_sample(ctypes.byref(d), a, a, a, a, 1.0, a, a, a, 1 << 30,
                                           None) == sbd.SBD_ERR_UNSUPPORTED
    d = sbd.HeadDesc(1, 16, 4000, 128256, sbd.SBD_DTYPE_BF16)       # H % 64 != 0
    assert sbd.lib.sbd_head_entropy_sample(ctypes.byref(d), a, a, a, a, 1.0, a, a, a, 1 << 30,
                                           None) == sbd.SBD_ERR_UNSUPPORTED
    d = sbd.HeadDesc(1, 16, 4096, 128256, sbd.SBD_DTYPE_BF16)
    for tau in (-1.0, float("nan"), float("inf")):
        assert sbd.lib.sbd_head_entropy_sample(ctypes.byref(d), a, a, a, a, tau, a, a, a,
                                               1 << 30, None) == sbd.SBD_ERR_INVALID_ARG
    # gumbel required when tau != 0
    assert sbd.lib.sbd_head_entropy_sample(ctypes.byref(d), a, a, a, None, 1.0, a, a, a,
                                           1 << 30, None) == sbd.SBD_ERR_INVALID_ARG


def test_eb_rejects_bad_arguments(sbd):
    a = 1 << 20
    assert sbd.lib.sbd_eb_select(1, 33, a, a, 0.1, a, a, a, None) == sbd.SBD_ERR_UNSUPPORTED
    assert sbd.lib.sbd_eb_select(1, 0, a, a, 0.1, a, a, a, None) == sbd.SBD_ERR_INVALID_ARG
    assert sbd.lib.sbd_eb_select(-1, 4, a, a, 0.1, a, a, a, None) == sbd.SBD_ERR_INVALID_ARG
    for g in (-0.5, float("nan"), float("inf")):
        assert sbd.lib.sbd_eb_select(1, 4, a, a, g, a, a, a, None) == sbd.SBD_ERR_INVALID_ARG
    assert sbd.lib.sbd_eb_select(1, 4, None, a, 0.1, a, a, a, None) == sbd.SBD_ERR_INVALID_ARG
    assert sbd.lib.sbd_eb_select(0, 4, None, None, 0.1, None, None, None, None) == sbd.SBD_OK


def test_select_rejects_bad_arguments(sbd):
    a = 1 << 20
    for rule in (-1, 4, 99):
        assert sbd.lib.sbd_select(rule, 1, 4, a, a, a, 0.1, a, a, a, None) == sbd.SBD_ERR_INVALID_ARG
        assert b"rule" in sbd.lib.sbd_last_error()
    for rule in (sbd.SBD_SELECT_EB_CONFIDENCE, sbd.SBD_SELECT_FACTOR,
                 sbd.SBD_SELECT_FACTOR_COMPLEMENT):
        # confidence-ordered rules need the confidence
        assert sbd.lib.sbd_select(rule, 1, 4, a, None, a, 0.1, a, a, a, None) == \
            sbd.SBD_ERR_INVALID_ARG
        assert sbd.lib.sbd_select(rule, 1, 33, a, a, a, 0.1, a, a, a, None) == \
            sbd.SBD_ERR_UNSUPPORTED
        for thr in (-0.5, float("nan"), float("inf")):
            assert sbd.lib.sbd_select(rule, 1, 4, a, a, a, thr, a, a, a, None) == \
                sbd.SBD_ERR_INVALID_ARG
    assert sbd.lib.sbd_select(sbd.SBD_SELECT_FACTOR, 0, 4, None, None, None, 1.0, None, None,
                              None, None) == sbd.SBD_OK


def test_confidence_head_rejects_bad_arguments(sbd):
    a = 1 << 20
    d = sbd.HeadDesc(1, 16, 4096, 128256, sbd.SBD_DTYPE_BF16)
    f = sbd.lib.sbd_head_entropy_confidence_sample
    assert f(ctypes.byref(d), a, a, a, a, 1.0, a, None, a, a, 1 << 30, None) == \
        sbd.SBD_ERR_INVALID_ARG
    assert f(ctypes.byref(d), a, a, a, a, 1.0, a, a + 4, a, a, 1 << 30, None) == \
        sbd.SBD_ERR_INVALID_ARG
    assert b"confidence" in sbd.lib.sbd_last_error()
    d = sbd.HeadDesc(32, 17, 4096, 128256, sbd.SBD_DTYPE_BF16)      # 544 rows > 512
    assert f(ctypes.byref(d), a, a, a, a, 1.0, a, a, a, a, 1 << 30, None) == \
        sbd.SBD_ERR_UNSUPPORTED


def test_philox_calls_reject_bad_arguments(sbd):
    a = 1 << 20
    d = sbd.HeadDesc(32, 17, 4096, 128256, sbd.SBD_DTYPE_BF16)      # 544 rows > 512
    f = sbd.lib.sbd_head_entropy_sample_philox
    assert f(ctypes.byref(d), a, a, a, 1, 2, 1.0, a, a, a, 1 << 30, None) == sbd.SBD_ERR_UNSUPPORTED
    d = sbd.HeadDesc(1, 16, 4096, 128256, sbd.SBD_DTYPE_BF16)
    for tau in (-1.0, float("nan")):
        assert f(ctypes.byref(d), a, a, a, 1, 2, tau, a, a, a, 1 << 30, None) == \
            sbd.SBD_ERR_INVALID_ARG
    g = sbd.lib.sbd_gumbel_philox
    assert g(-1, a, 10, 0, 0, a, None) == sbd.SBD_ERR_INVALID_ARG
    assert g(70000, a, 10, 0, 0, a, None) == sbd.SBD_ERR_UNSUPPORTED
    assert g(4, None, 10, 0, 0, a, None) == sbd.SBD_ERR_INVALID_ARG
    assert g(0, None, 10, 0, 0, None, None) == sbd.SBD_OK


def test_linear_rejects_bad_arguments(sbd):
    a = 1 << 20
    f = sbd.lib.sbd_linear
    L = sbd.LinearDesc
    bf = sbd.SBD_DTYPE_BF16
    big = 1 << 30
    assert f(None, a, a, a, a, big, None) == sbd.SBD_ERR_INVALID_ARG
    assert f(ctypes.byref(L(-1, 64, 8, bf)), a, a, a, a, big, None) == sbd.SBD_ERR_INVALID_ARG
    assert f(ctypes.byref(L(4, 0, 8, bf)), a, a, a, a, big, None) == sbd.SBD_ERR_INVALID_ARG
    assert f(ctypes.byref(L(4, 64, 8, 7)), a, a, a, a, big, None) == sbd.SBD_ERR_INVALID_ARG
    assert f(ctypes.byref(L(4, 64, 8, sbd.SBD_DTYPE_F32)), a, a, a, a, big, None) == \
        sbd.SBD_ERR_UNSUPPORTED
    assert f(ctypes.byref(L(513, 64, 8, bf)), a, a, a, a, big, None) == sbd.SBD_ERR_UNSUPPORTED
    assert f(ctypes.byref(L(4, 96, 8, bf)), a, a, a, a, big, None) == sbd.SBD_ERR_UNSUPPORTED
    assert f(ctypes.byref(L(4, 64, 8, bf)), None, a, a, a, big, None) == sbd.SBD_ERR_INVALID_ARG
    assert f(ctypes.byref(L(4, 64, 8, bf)), a + 2, a, a, a, big, None) == sbd.SBD_ERR_INVALID_ARG
    assert f(ctypes.byref(L(0, 64, 8, bf)), None, None, None, None, 0, None) == sbd.SBD_OK
    size = sbd.lib.sbd_linear_workspace_size
    assert size(None) == 0 and size(ctypes.byref(L(513, 64, 8, bf))) == 0
    # a narrow layer at few rows splits K: fp32 partials need a workspace
    d = L(16, 4096, 4096, bf)
    need = size(ctypes.byref(d))
    assert need == 16 * 16 * 4096 * 4        # sized for the largest split (16 ranges)
    assert f(ctypes.byref(d), a, a, a, None, 0, None) == sbd.SBD_ERR_WORKSPACE
    assert f(ctypes.byref(d), a, a, a, a, need - 1, None) == sbd.SBD_ERR_WORKSPACE
    assert size(ctypes.byref(L(512, 4096, 65536, bf))) == 0     # 512 tiles: never split


def test_binding_refuses_cpu_tensors(sbd):
    import torch
    x = torch.zeros(1, 4, 4, 64)
    with pytest.raises(ValueError, match="CUDA"):
        sbd.sbd_block_attention(x, x, x, torch.zeros(1, dtype=torch.int32), x, x)
    with pytest.raises(ValueError, match="CUDA"):
        sbd.sbd_eb_select(torch.zeros(1, 4), torch.zeros(1, 4, dtype=torch.int32), 0.1,
                          torch.zeros(1, 4, dtype=torch.uint8), torch.zeros(1, 4, dtype=torch.int32))


def test_product_path_does_not_import_the_oracle():
    pkg = os.path.join(ROOT, "paper_2509_04185_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                text = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in text and "from oracle" not in text, f
                assert "sbd_oracle" not in text, f
