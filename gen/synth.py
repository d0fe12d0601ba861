"""Seeded synthetic inputs for the SBD block step.

This module is the one source of inputs shared by the CUDA path and the fp64
oracle.  It holds no arithmetic of the method itself (no attention, softmax,
entropy or selection): it only draws random tensors of the shapes, dtypes and
distributions of the five workloads the block step is measured on, rounds them
to the storage precision, and builds the block state (which block positions
are still masked).

Determinism: every tensor is cut into fixed chunks of CHUNK elements and each
chunk is drawn from its own Philox stream keyed by (seed, workload, tensor,
chunk).  The result therefore does not depend on the number of threads used.

bf16 tensors are returned as ``np.uint16`` arrays holding the raw bf16 bit
patterns (round-to-nearest-even from the fp32 draw); fp32 tensors as
``np.float32``.  Both sides consume exactly these arrays.

Shapes of the workloads follow the paper's Llama-3.1-8B / Qwen-3-8B settings
(Sec. 4.1 constants: hidden 4096, 32 query heads, 8 KV heads, head dim 128;
Sec. 3.1: block sizes up to 16, contexts up to 32k; gamma values of Sec. 3.1
and the Fig. 5 ablation grid).
"""
from __future__ import annotations

import dataclasses
import os
import zlib
from concurrent.futures import ThreadPoolExecutor

import numpy as np

CHUNK = 1 << 22
MASK_TOKEN = -1

_POOL: ThreadPoolExecutor | None = None


def _pool() -> ThreadPoolExecutor:
    global _POOL
    if _POOL is None:
        _POOL = ThreadPoolExecutor(max_workers=max(1, min(32, os.cpu_count() or 1)))
    return _POOL


@dataclasses.dataclass(frozen=True)
class Workload:
    """One synthetic block-step workload.

    cache_len: either an int (every sequence has that many cached tokens) or a
    (lo, hi) pair: per-sequence lengths drawn uniformly from [lo, hi].
    decoded: how many leading block positions are already unmasked:
      ("fixed", n)        -> n for every sequence
      ("uniform", lo, hi) -> drawn per sequence from [lo, hi]
    """

    name: str
    batch: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    cache_len: object
    block_k: int
    hidden: int
    vocab: int
    dtype: str  # "f32" or "bf16"
    gammas: tuple
    decoded: tuple
    n_layers: int = 1
    w_std: float = 0.02
    hidden_scale: tuple = (0.1, 10.0)

    @property
    def max_cache_len(self) -> int:
        if isinstance(self.cache_len, tuple):
            return int(self.cache_len[1])
        return int(self.cache_len)


WORKLOADS = {
    "tiny_f32": Workload(
        name="tiny_f32", batch=1, n_q_heads=4, n_kv_heads=2, head_dim=64,
        cache_len=128, block_k=4, hidden=256, vocab=512, dtype="f32",
        gammas=(0.0, 0.1, 1.0), decoded=("fixed", 1)),
    "llama8b_k16": Workload(
        name="llama8b_k16", batch=1, n_q_heads=32, n_kv_heads=8, head_dim=128,
        cache_len=4096, block_k=16, hidden=4096, vocab=128256, dtype="bf16",
        gammas=(0.01, 0.1, 1.0), decoded=("fixed", 1)),
    "ragged_b32_k8": Workload(
        name="ragged_b32_k8", batch=32, n_q_heads=32, n_kv_heads=8, head_dim=128,
        cache_len=(512, 2048), block_k=8, hidden=4096, vocab=128256, dtype="bf16",
        gammas=(0.1,), decoded=("uniform", 1, 7)),
    "qwen8b_long_k16": Workload(
        name="qwen8b_long_k16", batch=4, n_q_heads=32, n_kv_heads=8, head_dim=128,
        cache_len=32768, block_k=16, hidden=4096, vocab=151936, dtype="bf16",
        gammas=(0.1, 1.0), decoded=("fixed", 1)),
}


def sweep_workload(block_k: int) -> Workload:
    """32-layer block-step sweep at Llama-3.1-8B attention shapes, batch 16,
    cache length 8192; the block starts fully masked (Algorithm 3 init)."""
    return Workload(
        name=f"sweep32_k{block_k}", batch=16, n_q_heads=32, n_kv_heads=8,
        head_dim=128, cache_len=8192, block_k=block_k, hidden=4096,
        vocab=128256, dtype="bf16", gammas=(0.1,), decoded=("fixed", 0),
        n_layers=32)


def get_workload(name: str) -> Workload:
    if name in WORKLOADS:
        return WORKLOADS[name]
    if name.startswith("sweep32_k"):
        return sweep_workload(int(name[len("sweep32_k"):]))
    raise KeyError(name)


def shrink(w: Workload, **over) -> Workload:
    """Same workload recipe at other sizes (used for small parity cases)."""
    return dataclasses.replace(w, **over)


# ---------------------------------------------------------------- streams

def _key(*parts) -> tuple:
    out = []
    for p in parts:
        if isinstance(p, str):
            out.append(zlib.crc32(p.encode()) & 0xFFFFFFFF)
        else:
            out.append(int(p) & 0xFFFFFFFF)
    return tuple(out)


def _gen(seed: int, key: tuple) -> np.random.Generator:
    ss = np.random.SeedSequence(int(seed), spawn_key=key)
    return np.random.Generator(np.random.Philox(ss))


def _chunked(n: int, fill, seed: int, key: tuple, dtype) -> np.ndarray:
    out = np.empty(n, dtype=dtype)
    nchunks = (n + CHUNK - 1) // CHUNK

    def work(c):
        lo = c * CHUNK
        hi = min(n, lo + CHUNK)
        fill(_gen(seed, key + (c,)), out[lo:hi])

    if nchunks <= 1:
        for c in range(nchunks):
            work(c)
    else:
        list(_pool().map(work, range(nchunks)))
    return out


def normal_f32(shape, seed: int, *key, std: float = 1.0) -> np.ndarray:
    n = int(np.prod(shape))

    def fill(g, dst):
        g.standard_normal(out=dst, dtype=np.float32)
        if std != 1.0:
            dst *= np.float32(std)

    return _chunked(n, fill, seed, _key(*key), np.float32).reshape(shape)


def uniform_open01_f64(shape, seed: int, *key) -> np.ndarray:
    """Uniform in the open interval (0, 1): (u53 + 0.5) / 2^53."""
    n = int(np.prod(shape))

    def fill(g, dst):
        bits = g.integers(0, 1 << 53, size=dst.shape[0], dtype=np.int64)
        dst[:] = (bits.astype(np.float64) + 0.5) * (1.0 / (1 << 53))

    return _chunked(n, fill, seed, _key(*key), np.float64).reshape(shape)


def gumbel_f32(shape, seed: int, *key) -> np.ndarray:
    """Standard Gumbel noise g = -log(-log u), u ~ U(0,1), stored as fp32."""
    n = int(np.prod(shape))

    def fill(g, dst):
        bits = g.integers(0, 1 << 53, size=dst.shape[0], dtype=np.int64)
        u = (bits.astype(np.float64) + 0.5) * (1.0 / (1 << 53))
        dst[:] = (-np.log(-np.log(u))).astype(np.float32)

    return _chunked(n, fill, seed, _key(*key), np.float32).reshape(shape)


# ---------------------------------------------------------------- storage

def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round fp32 to bf16 (nearest, ties to even); returns raw uint16 bits."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    flat_in = x.reshape(-1)
    flat_out = out.reshape(-1)
    n = flat_in.shape[0]

    def work(c):
        lo = c * CHUNK
        hi = min(n, lo + CHUNK)
        b = flat_in[lo:hi].view(np.uint32)
        nan = (b & 0x7FFFFFFF) > 0x7F800000
        r = (b + (0x7FFF + ((b >> 16) & 1))) >> 16
        r = np.where(nan, (b >> 16) | 0x40, r)
        flat_out[lo:hi] = r.astype(np.uint16)

    nchunks = (n + CHUNK - 1) // CHUNK
    if nchunks <= 1:
        for c in range(nchunks):
            work(c)
    else:
        list(_pool().map(work, range(nchunks)))
    return out


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def store(x: np.ndarray, dtype: str) -> np.ndarray:
    if dtype == "f32":
        return np.ascontiguousarray(x, dtype=np.float32)
    if dtype == "bf16":
        return f32_to_bf16_bits(x)
    raise ValueError(dtype)


BF16_NAN = np.uint16(0x7FC0)


# ---------------------------------------------------------------- workloads

def cache_lengths(w: Workload, seed: int) -> np.ndarray:
    if isinstance(w.cache_len, tuple):
        lo, hi = w.cache_len
        g = _gen(seed, _key(w.name, "cache_len"))
        return g.integers(lo, hi + 1, size=w.batch).astype(np.int32)
    return np.full(w.batch, int(w.cache_len), dtype=np.int32)


def block_state(w: Workload, seed: int):
    """Block token buffer (int32, -1 = mask token) and masked flags (uint8).

    The first n_b block positions of sequence b hold decoded tokens; the rest
    are the mask token (the input rule x_hat_j = x_j for j in J, else m)."""
    g = _gen(seed, _key(w.name, "block_state"))
    kind = w.decoded[0]
    if kind == "fixed":
        n_dec = np.full(w.batch, int(w.decoded[1]), dtype=np.int64)
    elif kind == "uniform":
        n_dec = g.integers(int(w.decoded[1]), int(w.decoded[2]) + 1, size=w.batch)
    else:
        raise ValueError(kind)
    n_dec = np.minimum(n_dec, w.block_k)
    tokens = g.integers(0, w.vocab, size=(w.batch, w.block_k)).astype(np.int32)
    pos = np.arange(w.block_k)[None, :]
    masked = (pos >= n_dec[:, None])
    block_tokens = np.where(masked, MASK_TOKEN, tokens).astype(np.int32)
    return block_tokens, masked.astype(np.uint8)


def attention_inputs(w: Workload, seed: int, layer: int = 0, poison_tail: bool = True):
    """q [B,k,Hq,D]; k_cache/v_cache [B,Lmax,Hkv,D]; cache_len [B];
    k_blk/v_blk [B,k,Hkv,D].  Entries are N(0,1).  Cache slots at or beyond a
    sequence's length hold NaN when poison_tail is set, so that any read of
    them that reaches the result shows up as NaN."""
    B, k, Hq, Hkv, D = w.batch, w.block_k, w.n_q_heads, w.n_kv_heads, w.head_dim
    Lmax = w.max_cache_len
    lens = cache_lengths(w, seed)
    q = store(normal_f32((B, k, Hq, D), seed, w.name, "q", layer), w.dtype)
    kc = store(normal_f32((B, Lmax, Hkv, D), seed, w.name, "k_cache", layer), w.dtype)
    vc = store(normal_f32((B, Lmax, Hkv, D), seed, w.name, "v_cache", layer), w.dtype)
    kb = store(normal_f32((B, k, Hkv, D), seed, w.name, "k_blk", layer), w.dtype)
    vb = store(normal_f32((B, k, Hkv, D), seed, w.name, "v_blk", layer), w.dtype)
    if poison_tail:
        nanv = BF16_NAN if w.dtype == "bf16" else np.float32("nan")
        for b in range(B):
            kc[b, lens[b]:] = nanv
            vc[b, lens[b]:] = nanv
    return dict(q=q, k_cache=kc, v_cache=vc, cache_len=lens, k_blk=kb, v_blk=vb)


def lm_head_weight(w: Workload, seed: int) -> np.ndarray:
    """W [V, H] (nn.Linear layout), N(0, w_std^2).  Keyed by shape, so the
    workloads that share a model shape share the weight."""
    return store(normal_f32((w.vocab, w.hidden), seed, "lm_head", w.vocab, w.hidden, "w",
                            std=w.w_std), w.dtype)


def hidden_scales(w: Workload, seed: int, step: int = 0) -> np.ndarray:
    """Per-row scale s [B,k] fp32, log-uniform in [hidden_scale[0],
    hidden_scale[1]]: log s ~ U[log lo, log hi]."""
    g = _gen(seed, _key(w.name, "hidden_scale", step))
    lo, hi = np.log(w.hidden_scale[0]), np.log(w.hidden_scale[1])
    return np.exp(g.uniform(lo, hi, size=(w.batch, w.block_k))).astype(np.float32)


def hidden_states(w: Workload, seed: int, step: int = 0) -> np.ndarray:
    """hidden [B,k,H]: rows N(0,1) times the per-row scale of hidden_scales
    (spreads the row entropies), rounded to the storage type."""
    B, k, H = w.batch, w.block_k, w.hidden
    h = normal_f32((B, k, H), seed, w.name, "hidden", step)
    h *= hidden_scales(w, seed, step)[:, :, None]
    return store(h, w.dtype)


def gumbel_noise(w: Workload, seed: int, step: int = 0) -> np.ndarray:
    """Gumbel noise [B,k,V] fp32, indexed by block position."""
    return gumbel_f32((w.batch, w.block_k, w.vocab), seed, w.name, "gumbel", step)


def step_inputs(w: Workload, seed: int, step: int = 0, poison_tail: bool = True) -> dict:
    d = attention_inputs(w, seed, 0, poison_tail)
    d["w"] = lm_head_weight(w, seed)
    d["hidden"] = hidden_states(w, seed, step)
    d["gumbel"] = gumbel_noise(w, seed, step)
    bt, m = block_state(w, seed)
    d["block_tokens"] = bt
    d["masked"] = m
    return d
