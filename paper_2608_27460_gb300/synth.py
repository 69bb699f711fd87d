"""Seeded synthetic inputs shaped like the output heads the paper evaluates.

This module only draws inputs.  It holds none of the head's arithmetic (no
projection, no selection, no scatter) and imports neither the CUDA binding
nor the oracle, so both sides can consume the same arrays.

The paper measures on real Gemma 3 / Llama 3.2 / Qwen3 output embeddings and
on hidden states from a Wikipedia article (Section 4.1); neither is
available here, so seeded stand-ins with the models' shapes replace them:

  * rows   w_i = s_i * g_i,  g_i ~ N(0, 0.02^2 I_d),  s_i = exp(N(0, 0.3^2)),
           rounded to bf16 (round to nearest even) and kept as raw bit patterns;
  * query  h = sum_{m<3} c_m * w_{r_m} + n,  r_m three distinct rows drawn
           uniformly, c_m ~ N(20, 2^2), n ~ N(0, I_d); stored as fp32;
  * tie stress: floor(frac * V) destination rows (distinct, uniform) each copy
           a uniformly drawn non-destination source row bit for bit, and a
           share of the queries is planted on a duplicated source row.

Randomness: numpy ``Generator(PCG64(seed))``.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np


@dataclass(frozen=True)
class HeadShape:
    """Output-head workload: vocabulary V, hidden size d and the decode
    batches / top-k values / step counts it is exercised with."""
    name: str
    V: int
    d: int
    batches: tuple
    ks: tuple
    steps: int
    dup_frac: float = 0.0
    extra: dict = field(default_factory=dict)

    @property
    def weight_bytes(self) -> int:
        return self.V * self.d * 2


# Shapes of the models in the paper's evaluation (Section 4).
HEADS = {
    "gemma3-270m": HeadShape("gemma3-270m", 262144, 640, (1,), (50,), 16),
    "qwen3-0.6b": HeadShape("qwen3-0.6b", 151936, 1024, (1,), (50,), 1000),
    "llama3.2-1b": HeadShape("llama3.2-1b", 128256, 2048, (1, 4), (50, 1), 1000),
    "gemma3-1b": HeadShape("gemma3-1b", 262144, 1152, (1, 2, 4, 8), (50,), 1000),
    "gemma3-1b-ties": HeadShape("gemma3-1b-ties", 262144, 1152, (1, 2, 4, 8), (50,), 1000,
                                dup_frac=0.05),
    "llama3.2-3b": HeadShape("llama3.2-3b", 128256, 3072, (16, 64), (50,), 500),
}
HEAD_ORDER = ("gemma3-270m", "qwen3-0.6b", "llama3.2-1b", "gemma3-1b", "llama3.2-3b")


def rng_for(seed: int) -> np.random.Generator:
    return np.random.Generator(np.random.PCG64(seed))


def f32_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round finite fp32 values to bf16, nearest even; returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    bias = np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return ((u + bias) >> np.uint32(16)).astype(np.uint16)


def bf16_bits_to_f32(bits: np.ndarray) -> np.ndarray:
    """Widen bf16 bit patterns to fp32 (exact)."""
    return (np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def make_weights(V: int, d: int, seed: int, dup_frac: float = 0.0,
                 row_chunk: int = 16384):
    """Draw W_out [V, d] as bf16 bit patterns; returns (W_bits, meta).

    meta["dup_dst"], meta["dup_src"] list the copied rows for the tie-stress
    variant (empty arrays otherwise)."""
    rng = rng_for(seed)
    W = np.empty((V, d), dtype=np.uint16)
    # chunk buffers are reused (fresh arrays per chunk cost more in page
    # faults than the drawing itself); the values are those of
    # f32_to_bf16_bits on each chunk, bit for bit
    g_buf = np.empty((min(row_chunk, V), d), dtype=np.float32)
    t_buf = np.empty((min(row_chunk, V), d), dtype=np.uint32)
    for r0 in range(0, V, row_chunk):
        n = min(row_chunk, V - r0)
        g = g_buf[:n]
        rng.standard_normal(out=g, dtype=np.float32)
        g *= np.float32(0.02)
        s = np.exp(rng.normal(0.0, 0.3, size=(n, 1))).astype(np.float32)
        g *= s
        u, t = g.view(np.uint32), t_buf[:n]
        np.right_shift(u, np.uint32(16), out=t)  # round to nearest even: + 0x7FFF + lsb
        t &= np.uint32(1)
        t += np.uint32(0x7FFF)
        t += u
        t >>= np.uint32(16)
        W[r0:r0 + n] = t
    dst = np.zeros(0, dtype=np.int64)
    src = np.zeros(0, dtype=np.int64)
    n_dup = int(np.floor(dup_frac * V))
    if n_dup > 0:
        dst = np.sort(rng.choice(V, size=n_dup, replace=False))
        pool = np.setdiff1d(np.arange(V, dtype=np.int64), dst, assume_unique=True)
        src = rng.choice(pool, size=n_dup, replace=True)
        W[dst] = W[src]
    return W, {"dup_dst": dst, "dup_src": src}


def make_queries(W_bits: np.ndarray, n: int, seed: int, planted_frac: float = 0.0,
                 dup_src=None):
    """Draw n hidden states h [n, d] (fp32) from W's rows; returns (h, rows).

    With ``planted_frac`` > 0 and ``dup_src`` given, the first
    ceil(planted_frac * n) queries take a duplicated source row as their
    first component, so exact ties appear near the top of their ranking."""
    V, d = W_bits.shape
    rng = rng_for(seed)
    rows = np.empty((n, 3), dtype=np.int64)
    for q in range(n):
        rows[q] = rng.choice(V, size=3, replace=False)
    if planted_frac > 0 and dup_src is not None and len(dup_src) > 0:
        sources = np.unique(np.asarray(dup_src, dtype=np.int64))
        n_plant = int(np.ceil(planted_frac * n))
        for q in range(n_plant):
            r = int(rng.choice(sources))
            if r not in rows[q, 1:]:
                rows[q, 0] = r
    c = rng.normal(20.0, 2.0, size=(n, 3))
    noise = rng.standard_normal((n, d))
    h = np.empty((n, d), dtype=np.float32)
    for q in range(n):
        w = bf16_bits_to_f32(W_bits[rows[q]]).astype(np.float64)
        h[q] = (c[q] @ w + noise[q]).astype(np.float32)
    return h, rows


def make_head(shape: HeadShape, seed: int = 0, n_queries: int = 16, planted_frac: float = 0.25):
    """Weights and queries for one workload; seed offset per workload name."""
    offset = HEAD_ORDER.index(shape.name) if shape.name in HEAD_ORDER else len(HEAD_ORDER)
    W, meta = make_weights(shape.V, shape.d, seed + offset, dup_frac=shape.dup_frac)
    plant = planted_frac if shape.dup_frac > 0 else 0.0
    h, rows = make_queries(W, n_queries, seed + 1000 + offset, planted_frac=plant,
                           dup_src=meta["dup_src"])
    return W, h, meta, rows


def make_candidates(batch: int, k: int, V: int, seed: int, spread: float = 3.0,
                    ties: float = 0.0):
    """Candidate rows for top-k sampling, shaped like a head's output:
    distinct vocabulary indices per row (int32 [batch, k]) and fp32 logits
    [batch, k] sorted best first, drawn N(0, spread^2); with ties > 0 about
    that share of the logits repeats its neighbour's value exactly."""
    rng = np.random.default_rng(seed)
    idx = np.stack([rng.choice(V, size=k, replace=False) for _ in range(batch)]).astype(np.int32)
    z = rng.normal(0.0, spread, size=(batch, k)).astype(np.float32)
    if ties > 0 and k > 1:
        rep = rng.random((batch, k)) < ties
        rep[:, 0] = False
        z = np.sort(z, axis=1)[:, ::-1].copy()
        for b in range(batch):
            for j in range(1, k):
                if rep[b, j]:
                    z[b, j] = z[b, j - 1]
    z = np.sort(z, axis=1)[:, ::-1].astype(np.float32, order="C", copy=True)
    return idx, z
