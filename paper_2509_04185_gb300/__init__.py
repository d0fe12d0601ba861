"""Python binding of libsbd, the GB300 (sm_103a) Set Block Decoding block step.

Argument marshalling only: every computation runs in the CUDA kernels of
libsbd.so (csrc/), reached through its C ABI (include/sbd.h) with ctypes.
PyTorch supplies device memory and streams.  There is no CPU path: the
functions require CUDA tensors, and importing this package raises if the
library has not been built (``python -c "import __graft_entry__ as g;
g.build()"``).

The three calls of one SBD forward (arXiv 2509.04185, Eq. 5, Eqs. 6-7,
Eq. 3 / Algorithm 3) keep the names of the C ABI:

    sbd_block_attention(q, k_cache, v_cache, cache_len, k_blk, v_blk)
    sbd_head_entropy_sample(hidden, w, masked, gumbel, tau)
    sbd_eb_select(entropy, token, gamma, masked, block_tokens)
"""
from __future__ import annotations

import ctypes
import os

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libsbd.so")

SBD_OK = 0
SBD_ERR_INVALID_ARG = 1
SBD_ERR_UNSUPPORTED = 2
SBD_ERR_WORKSPACE = 3
SBD_ERR_CUDA = 4
SBD_DTYPE_F32 = 0
SBD_DTYPE_BF16 = 1
SBD_DEVERR_CACHE_LEN = 1
SBD_DEVERR_TIMEOUT = 2
SBD_DEVERR_ROWS = 4
SBD_HEAD_NOALLOC_MAX_SCRATCH = 8 << 20
SBD_SELECT_EB_ENTROPY = 0
SBD_SELECT_EB_CONFIDENCE = 1
SBD_SELECT_FACTOR = 2
SBD_SELECT_FACTOR_COMPLEMENT = 3

# Every symbol include/sbd.h declares.
EXPORTS = (
    "sbd_block_attention_workspace_size",
    "sbd_block_attention",
    "sbd_block_attention_causal_prefix",
    "sbd_head_entropy_sample_workspace_size",
    "sbd_head_entropy_sample",
    "sbd_head_entropy_sample_noalloc",
    "sbd_head_entropy_confidence_sample",
    "sbd_head_entropy_sample_philox",
    "sbd_gumbel_philox",
    "sbd_linear_workspace_size",
    "sbd_linear",
    "sbd_eb_select",
    "sbd_select",
    "sbd_status_string",
    "sbd_last_error",
    "sbd_device_error",
    "sbd_version",
)


class AttnDesc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("block_k", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("max_cache_len", ctypes.c_int32),
                ("dtype", ctypes.c_int32), ("scale", ctypes.c_float),
                ("num_splits", ctypes.c_int32)]


class HeadDesc(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("block_k", ctypes.c_int32),
                ("hidden", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("dtype", ctypes.c_int32)]


class LinearDesc(ctypes.Structure):
    _fields_ = [("rows", ctypes.c_int32), ("in_features", ctypes.c_int32),
                ("out_features", ctypes.c_int32), ("dtype", ctypes.c_int32)]


class SbdError(RuntimeError):
    def __init__(self, status: int, detail: str):
        self.status = status
        super().__init__(f"{_status_name(status)}: {detail}")


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(f"{path} is missing: build it first (__graft_entry__.build())")
    lib = ctypes.CDLL(path)
    vp, sz, i32, f32 = ctypes.c_void_p, ctypes.c_size_t, ctypes.c_int32, ctypes.c_float
    lib.sbd_block_attention_workspace_size.argtypes = [ctypes.POINTER(AttnDesc)]
    lib.sbd_block_attention_workspace_size.restype = sz
    lib.sbd_block_attention.argtypes = [ctypes.POINTER(AttnDesc), vp, vp, vp, vp, vp, vp, vp,
                                        vp, sz, vp]
    lib.sbd_block_attention.restype = ctypes.c_int
    lib.sbd_block_attention_causal_prefix.argtypes = [ctypes.POINTER(AttnDesc), i32, vp, vp, vp,
                                                      vp, vp, vp, vp, vp, sz, vp]
    lib.sbd_block_attention_causal_prefix.restype = ctypes.c_int
    lib.sbd_head_entropy_sample_workspace_size.argtypes = [ctypes.POINTER(HeadDesc)]
    lib.sbd_head_entropy_sample_workspace_size.restype = sz
    lib.sbd_head_entropy_sample.argtypes = [ctypes.POINTER(HeadDesc), vp, vp, vp, vp, f32, vp,
                                            vp, vp, sz, vp]
    lib.sbd_head_entropy_sample.restype = ctypes.c_int
    lib.sbd_head_entropy_sample_noalloc.argtypes = [ctypes.POINTER(HeadDesc), vp, vp, vp, vp,
                                                    f32, vp, vp, vp]
    lib.sbd_head_entropy_sample_noalloc.restype = ctypes.c_int
    lib.sbd_head_entropy_confidence_sample.argtypes = [ctypes.POINTER(HeadDesc), vp, vp, vp, vp,
                                                       f32, vp, vp, vp, vp, sz, vp]
    lib.sbd_head_entropy_confidence_sample.restype = ctypes.c_int
    u64 = ctypes.c_uint64
    lib.sbd_head_entropy_sample_philox.argtypes = [ctypes.POINTER(HeadDesc), vp, vp, vp, u64, u64,
                                                   f32, vp, vp, vp, sz, vp]
    lib.sbd_head_entropy_sample_philox.restype = ctypes.c_int
    lib.sbd_gumbel_philox.argtypes = [i32, vp, i32, u64, u64, vp, vp]
    lib.sbd_gumbel_philox.restype = ctypes.c_int
    lib.sbd_linear_workspace_size.argtypes = [ctypes.POINTER(LinearDesc)]
    lib.sbd_linear_workspace_size.restype = sz
    lib.sbd_linear.argtypes = [ctypes.POINTER(LinearDesc), vp, vp, vp, vp, sz, vp]
    lib.sbd_linear.restype = ctypes.c_int
    lib.sbd_eb_select.argtypes = [i32, i32, vp, vp, f32, vp, vp, vp, vp]
    lib.sbd_eb_select.restype = ctypes.c_int
    lib.sbd_select.argtypes = [i32, i32, i32, vp, vp, vp, f32, vp, vp, vp, vp]
    lib.sbd_select.restype = ctypes.c_int
    lib.sbd_status_string.argtypes = [ctypes.c_int]
    lib.sbd_status_string.restype = ctypes.c_char_p
    lib.sbd_last_error.argtypes = []
    lib.sbd_last_error.restype = ctypes.c_char_p
    lib.sbd_device_error.argtypes = [ctypes.POINTER(ctypes.c_int32)]
    lib.sbd_device_error.restype = ctypes.c_int
    lib.sbd_version.argtypes = []
    lib.sbd_version.restype = i32
    return lib


lib = load_library()


def _status_name(st: int) -> str:
    return lib.sbd_status_string(st).decode()


def _check(st: int) -> None:
    if st != SBD_OK:
        raise SbdError(st, lib.sbd_last_error().decode())


# ------------------------------------------------------------------ helpers

def _torch():
    import torch
    return torch


def _dtype_code(t) -> int:
    torch = _torch()
    if t.dtype == torch.bfloat16:
        return SBD_DTYPE_BF16
    if t.dtype == torch.float32:
        return SBD_DTYPE_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _need_cuda(**tensors):
    for name, t in tensors.items():
        if t is None:
            continue
        if not t.is_cuda:
            raise ValueError(f"{name} must be a CUDA tensor (libsbd has no CPU path)")
        if not t.is_contiguous():
            raise ValueError(f"{name} must be contiguous")


def _ptr(t) -> int | None:
    return None if t is None else t.data_ptr()


def _stream(stream) -> int | None:
    torch = _torch()
    if stream is None:
        stream = torch.cuda.current_stream()
    return stream.cuda_stream


def attn_desc(q, k_cache, scale: float = 0.0, num_splits: int = 0) -> AttnDesc:
    B, k, Hq, D = q.shape
    return AttnDesc(B, k, Hq, k_cache.shape[2], D, k_cache.shape[1], _dtype_code(q),
                    float(scale), int(num_splits))


def head_desc(hidden, w) -> HeadDesc:
    B, k, H = hidden.shape
    return HeadDesc(B, k, H, w.shape[0], _dtype_code(hidden))


def _nbytes(t) -> int:
    return 0 if t is None else t.numel() * t.element_size()


def _workspace(nbytes: int, device, workspace=None):
    torch = _torch()
    if nbytes == 0:
        return None
    if workspace is not None and _nbytes(workspace) >= nbytes:
        return workspace
    return torch.empty(nbytes, dtype=torch.uint8, device=device)


# ------------------------------------------------------------------ API

def sbd_block_attention(q, k_cache, v_cache, cache_len, k_blk, v_blk, out=None, *,
                        scale: float = 0.0, num_splits: int = 0, workspace=None, stream=None):
    """Block attention (Eq. 5, inference mask of Fig. 3).  Shapes:
    q [B,k,Hq,D], k_cache/v_cache [B,Lmax,Hkv,D], cache_len [B] int32,
    k_blk/v_blk [B,k,Hkv,D]; returns out [B,k,Hq,D] (dtype of q)."""
    torch = _torch()
    _need_cuda(q=q, k_cache=k_cache, v_cache=v_cache, cache_len=cache_len, k_blk=k_blk,
               v_blk=v_blk, out=out)
    if cache_len.dtype != torch.int32:
        raise TypeError("cache_len must be int32")
    if out is None:
        out = torch.empty_like(q)
    d = attn_desc(q, k_cache, scale, num_splits)
    ws = _workspace(lib.sbd_block_attention_workspace_size(ctypes.byref(d)), q.device, workspace)
    _check(lib.sbd_block_attention(ctypes.byref(d), _ptr(q), _ptr(k_cache), _ptr(v_cache),
                                   _ptr(cache_len), _ptr(k_blk), _ptr(v_blk), _ptr(out),
                                   _ptr(ws), _nbytes(ws), _stream(stream)))
    return out


def sbd_block_attention_causal_prefix(q, k_cache, v_cache, cache_len, k_blk, v_blk,
                                      n_causal: int, out=None, *, scale: float = 0.0,
                                      num_splits: int = 0, workspace=None, stream=None):
    """First iteration of a block after the previous one (Algorithm 3): block
    rows i < n_causal (the previous block's tokens) are causal among the
    block keys and their keys/values are written into k_cache / v_cache at
    cache_len[b] + i (cache_len is not changed); the other rows see every
    key.  Shapes as sbd_block_attention; returns out."""
    torch = _torch()
    _need_cuda(q=q, k_cache=k_cache, v_cache=v_cache, cache_len=cache_len, k_blk=k_blk,
               v_blk=v_blk, out=out)
    if cache_len.dtype != torch.int32:
        raise TypeError("cache_len must be int32")
    if out is None:
        out = torch.empty_like(q)
    d = attn_desc(q, k_cache, scale, num_splits)
    ws = _workspace(lib.sbd_block_attention_workspace_size(ctypes.byref(d)), q.device, workspace)
    _check(lib.sbd_block_attention_causal_prefix(
        ctypes.byref(d), int(n_causal), _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(cache_len),
        _ptr(k_blk), _ptr(v_blk), _ptr(out), _ptr(ws), _nbytes(ws), _stream(stream)))
    return out


def sbd_head_entropy_sample(hidden, w, masked, gumbel, tau: float, entropy=None, token=None,
                            *, workspace=None, stream=None):
    """LM head + entropy + Gumbel-max token over masked positions (Eqs. 6-7).
    hidden [B,k,H], w [V,H], masked [B,k] uint8, gumbel [B,k,V] fp32 or None
    (tau == 0).  Returns (entropy [B,k] fp32, token [B,k] int32)."""
    torch = _torch()
    _need_cuda(hidden=hidden, w=w, masked=masked, gumbel=gumbel, entropy=entropy, token=token)
    if masked.dtype != torch.uint8:
        raise TypeError("masked must be uint8")
    B, k, _ = hidden.shape
    if entropy is None:
        entropy = torch.empty((B, k), dtype=torch.float32, device=hidden.device)
    if token is None:
        token = torch.empty((B, k), dtype=torch.int32, device=hidden.device)
    d = head_desc(hidden, w)
    ws = _workspace(lib.sbd_head_entropy_sample_workspace_size(ctypes.byref(d)), hidden.device,
                    workspace)
    _check(lib.sbd_head_entropy_sample(ctypes.byref(d), _ptr(hidden), _ptr(w), _ptr(masked),
                                       _ptr(gumbel), float(tau), _ptr(entropy), _ptr(token),
                                       _ptr(ws), _nbytes(ws), _stream(stream)))
    return entropy, token


def sbd_head_entropy_confidence_sample(hidden, w, masked, gumbel, tau: float, entropy=None,
                                       confidence=None, token=None, *, workspace=None,
                                       stream=None):
    """sbd_head_entropy_sample plus confidence = max_v p_v of every masked
    position (0 at unmasked ones), for the confidence-ordered selection
    rules.  Returns (entropy [B,k] fp32, confidence [B,k] fp32, token [B,k]
    int32)."""
    torch = _torch()
    _need_cuda(hidden=hidden, w=w, masked=masked, gumbel=gumbel, entropy=entropy,
               confidence=confidence, token=token)
    if masked.dtype != torch.uint8:
        raise TypeError("masked must be uint8")
    B, k, _ = hidden.shape
    if entropy is None:
        entropy = torch.empty((B, k), dtype=torch.float32, device=hidden.device)
    if confidence is None:
        confidence = torch.empty((B, k), dtype=torch.float32, device=hidden.device)
    if token is None:
        token = torch.empty((B, k), dtype=torch.int32, device=hidden.device)
    d = head_desc(hidden, w)
    ws = _workspace(lib.sbd_head_entropy_sample_workspace_size(ctypes.byref(d)), hidden.device,
                    workspace)
    _check(lib.sbd_head_entropy_confidence_sample(
        ctypes.byref(d), _ptr(hidden), _ptr(w), _ptr(masked), _ptr(gumbel), float(tau),
        _ptr(entropy), _ptr(confidence), _ptr(token), _ptr(ws), _nbytes(ws), _stream(stream)))
    return entropy, confidence, token


def sbd_head_entropy_sample_philox(hidden, w, masked, seed: int, offset: int, tau: float,
                                   entropy=None, token=None, *, workspace=None, stream=None):
    """sbd_head_entropy_sample with the Gumbel noise generated in the kernel
    from Philox4x32-10 (seed, offset) instead of read from a tensor.
    Returns (entropy [B,k] fp32, token [B,k] int32)."""
    torch = _torch()
    _need_cuda(hidden=hidden, w=w, masked=masked, entropy=entropy, token=token)
    if masked.dtype != torch.uint8:
        raise TypeError("masked must be uint8")
    B, k, _ = hidden.shape
    if entropy is None:
        entropy = torch.empty((B, k), dtype=torch.float32, device=hidden.device)
    if token is None:
        token = torch.empty((B, k), dtype=torch.int32, device=hidden.device)
    d = head_desc(hidden, w)
    ws = _workspace(lib.sbd_head_entropy_sample_workspace_size(ctypes.byref(d)), hidden.device,
                    workspace)
    _check(lib.sbd_head_entropy_sample_philox(ctypes.byref(d), _ptr(hidden), _ptr(w), _ptr(masked),
                                              int(seed), int(offset), float(tau), _ptr(entropy),
                                              _ptr(token), _ptr(ws), _nbytes(ws), _stream(stream)))
    return entropy, token


def sbd_gumbel_philox(row_ids, vocab: int, seed: int, offset: int, out=None, *, stream=None):
    """The counter-based noise written out: out[r, v] = g(row_ids[r], v),
    row_ids int32 block positions (b * k + i).  Returns out [n, vocab] fp32."""
    torch = _torch()
    _need_cuda(row_ids=row_ids, out=out)
    if row_ids.dtype != torch.int32:
        raise TypeError("row_ids must be int32")
    n = row_ids.numel()
    if out is None:
        out = torch.empty((n, vocab), dtype=torch.float32, device=row_ids.device)
    _check(lib.sbd_gumbel_philox(n, _ptr(row_ids), int(vocab), int(seed), int(offset), _ptr(out),
                                 _stream(stream)))
    return out


def _linear_desc(x, w):
    if x.dim() != 2 or w.dim() != 2 or x.shape[1] != w.shape[1]:
        raise ValueError(f"shapes x {tuple(x.shape)} and w {tuple(w.shape)} do not match")
    return LinearDesc(x.shape[0], x.shape[1], w.shape[0], _dtype_code(x))


def sbd_linear(x, w, out=None, workspace=None, *, stream=None):
    """y = x W^T on the LM-head kernel: x [T, K] bf16, w [N, K] bf16
    (nn.Linear layout), T <= 512, K a multiple of 64.  Returns out [T, N]
    bf16.  The workspace (fp32 partials when K is split at few rows) is
    allocated here when not given."""
    torch = _torch()
    _need_cuda(x=x, w=w, out=out, workspace=workspace)
    d = _linear_desc(x, w)
    if out is None:
        out = torch.empty((x.shape[0], w.shape[0]), dtype=x.dtype, device=x.device)
    need = lib.sbd_linear_workspace_size(ctypes.byref(d))
    if workspace is None and need > 0:
        workspace = torch.empty(need, dtype=torch.uint8, device=x.device)
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(lib.sbd_linear(ctypes.byref(d), _ptr(x), _ptr(w), _ptr(out), _ptr(workspace), nbytes,
                          _stream(stream)))
    return out


def prepare_linear(x, w, out, workspace=None, *, stream=None) -> "Prepared":
    """sbd_linear bound to fixed tensors (see Prepared)."""
    torch = _torch()
    _need_cuda(x=x, w=w, out=out, workspace=workspace)
    d = _linear_desc(x, w)
    need = lib.sbd_linear_workspace_size(ctypes.byref(d))
    if workspace is None and need > 0:
        workspace = torch.empty(need, dtype=torch.uint8, device=x.device)
    nbytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    args = (ctypes.byref(d), _ptr(x), _ptr(w), _ptr(out), _ptr(workspace), nbytes,
            _stream(stream))
    return Prepared(lib.sbd_linear, args, keep=(d, x, w, out, workspace))


def sbd_head_entropy_sample_noalloc(hidden, w, masked, gumbel, tau: float, entropy, token, *,
                                    stream=None):
    """sbd_head_entropy_sample for callers that cannot allocate device
    memory: the scratch is the library's fixed device array (shared by every
    call on a device; calls must not overlap on the GPU).  The outputs
    entropy [B,k] fp32 and token [B,k] int32 are caller-provided; nothing is
    allocated here or in the library."""
    torch = _torch()
    _need_cuda(hidden=hidden, w=w, masked=masked, gumbel=gumbel, entropy=entropy, token=token)
    if masked.dtype != torch.uint8:
        raise TypeError("masked must be uint8")
    d = head_desc(hidden, w)
    _check(lib.sbd_head_entropy_sample_noalloc(ctypes.byref(d), _ptr(hidden), _ptr(w),
                                               _ptr(masked), _ptr(gumbel), float(tau),
                                               _ptr(entropy), _ptr(token), _stream(stream)))
    return entropy, token


def sbd_eb_select(entropy, token, gamma: float, masked, block_tokens, n_unmasked=None, *,
                  stream=None):
    """EB select (Eq. 3): updates masked [B,k] uint8 and block_tokens [B,k]
    int32 in place; returns n_unmasked [B] int32."""
    torch = _torch()
    _need_cuda(entropy=entropy, token=token, masked=masked, block_tokens=block_tokens,
               n_unmasked=n_unmasked)
    B, k = masked.shape
    if n_unmasked is None:
        n_unmasked = torch.empty(B, dtype=torch.int32, device=masked.device)
    _check(lib.sbd_eb_select(B, k, _ptr(entropy), _ptr(token), float(gamma), _ptr(masked),
                             _ptr(block_tokens), _ptr(n_unmasked), _stream(stream)))
    return n_unmasked


def sbd_select(rule: int, entropy, confidence, token, threshold: float, masked, block_tokens,
               n_unmasked=None, *, stream=None):
    """One unmasking step under `rule` (SBD_SELECT_*: Eq. 3, the general EB
    bound in confidence order, or the Factor rule); threshold is gamma or f.
    Updates masked and block_tokens in place; returns n_unmasked [B] int32.
    confidence may be None for SBD_SELECT_EB_ENTROPY."""
    torch = _torch()
    _need_cuda(entropy=entropy, confidence=confidence, token=token, masked=masked,
               block_tokens=block_tokens, n_unmasked=n_unmasked)
    B, k = masked.shape
    if n_unmasked is None:
        n_unmasked = torch.empty(B, dtype=torch.int32, device=masked.device)
    _check(lib.sbd_select(int(rule), B, k, _ptr(entropy), _ptr(confidence), _ptr(token),
                          float(threshold), _ptr(masked), _ptr(block_tokens), _ptr(n_unmasked),
                          _stream(stream)))
    return n_unmasked


class Prepared:
    """A library call with every argument already marshalled: calling it
    re-issues the same C call (same tensors, stream and workspace) with no
    Python-side checks.  For step loops that repeat one call shape."""

    __slots__ = ("_fn", "_args", "_keep")

    def __init__(self, fn, args, keep):
        self._fn = fn
        self._args = args
        self._keep = keep          # tensors whose memory the pointers refer to

    def __call__(self) -> None:
        st = self._fn(*self._args)
        if st != SBD_OK:
            raise SbdError(st, lib.sbd_last_error().decode())


def prepare_block_attention(q, k_cache, v_cache, cache_len, k_blk, v_blk, out, workspace=None,
                            *, scale: float = 0.0, num_splits: int = 0, stream=None) -> Prepared:
    """sbd_block_attention bound to fixed tensors (see Prepared)."""
    torch = _torch()
    _need_cuda(q=q, k_cache=k_cache, v_cache=v_cache, cache_len=cache_len, k_blk=k_blk,
               v_blk=v_blk, out=out)
    if cache_len.dtype != torch.int32:
        raise TypeError("cache_len must be int32")
    d = attn_desc(q, k_cache, scale, num_splits)
    ws = _workspace(lib.sbd_block_attention_workspace_size(ctypes.byref(d)), q.device, workspace)
    args = (ctypes.byref(d), _ptr(q), _ptr(k_cache), _ptr(v_cache), _ptr(cache_len), _ptr(k_blk),
            _ptr(v_blk), _ptr(out), _ptr(ws), _nbytes(ws), _stream(stream))
    return Prepared(lib.sbd_block_attention, args,
                    (d, q, k_cache, v_cache, cache_len, k_blk, v_blk, out, ws))


def prepare_head_entropy_sample(hidden, w, masked, gumbel, tau: float, entropy, token,
                                workspace=None, *, stream=None) -> Prepared:
    """sbd_head_entropy_sample bound to fixed tensors (see Prepared)."""
    torch = _torch()
    _need_cuda(hidden=hidden, w=w, masked=masked, gumbel=gumbel, entropy=entropy, token=token)
    if masked.dtype != torch.uint8:
        raise TypeError("masked must be uint8")
    d = head_desc(hidden, w)
    ws = _workspace(lib.sbd_head_entropy_sample_workspace_size(ctypes.byref(d)), hidden.device,
                    workspace)
    args = (ctypes.byref(d), _ptr(hidden), _ptr(w), _ptr(masked), _ptr(gumbel), float(tau),
            _ptr(entropy), _ptr(token), _ptr(ws), _nbytes(ws), _stream(stream))
    return Prepared(lib.sbd_head_entropy_sample, args,
                    (d, hidden, w, masked, gumbel, entropy, token, ws))


def prepare_head_entropy_sample_philox(hidden, w, masked, seed: int, offset: int, tau: float,
                                       entropy, token, workspace=None, *,
                                       stream=None) -> Prepared:
    """sbd_head_entropy_sample_philox bound to fixed tensors (see Prepared)."""
    torch = _torch()
    _need_cuda(hidden=hidden, w=w, masked=masked, entropy=entropy, token=token)
    if masked.dtype != torch.uint8:
        raise TypeError("masked must be uint8")
    d = head_desc(hidden, w)
    ws = _workspace(lib.sbd_head_entropy_sample_workspace_size(ctypes.byref(d)), hidden.device,
                    workspace)
    args = (ctypes.byref(d), _ptr(hidden), _ptr(w), _ptr(masked), int(seed), int(offset),
            float(tau), _ptr(entropy), _ptr(token), _ptr(ws), _nbytes(ws), _stream(stream))
    return Prepared(lib.sbd_head_entropy_sample_philox, args,
                    (d, hidden, w, masked, entropy, token, ws))


def prepare_eb_select(entropy, token, gamma: float, masked, block_tokens, n_unmasked, *,
                      stream=None) -> Prepared:
    """sbd_eb_select bound to fixed tensors (see Prepared)."""
    _need_cuda(entropy=entropy, token=token, masked=masked, block_tokens=block_tokens,
               n_unmasked=n_unmasked)
    B, k = masked.shape
    args = (B, k, _ptr(entropy), _ptr(token), float(gamma), _ptr(masked), _ptr(block_tokens),
            _ptr(n_unmasked), _stream(stream))
    return Prepared(lib.sbd_eb_select, args, (entropy, token, masked, block_tokens, n_unmasked))


def sbd_device_error() -> int:
    """Reads and clears the device error word (synchronises the device)."""
    code = ctypes.c_int32(0)
    _check(lib.sbd_device_error(ctypes.byref(code)))
    return code.value


def sbd_version() -> int:
    return int(lib.sbd_version())
