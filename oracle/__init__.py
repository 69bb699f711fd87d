"""Plain CPU oracle for the exact LLM output head -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` and
``--impl reference`` legs of ``bench.py`` may import this package.  The CUDA
path (``paper_2608_27460_gb300``) never imports it, and this package imports
nothing from that path: the two share no code.

The arithmetic lives in ``oracle.c`` (plain C, fp64, no blocking); this module
only builds it with gcc and marshals numpy arrays through ctypes.

  * :func:`logits`  -- z = W_out h, z_i = <w_i, h> in fp64      (Section 3)
  * :func:`topk`    -- exhaustive MIPS: full sort by (z desc, index asc),
                       first k rows                               (Sections 2, 3)
  * :func:`scatter` -- sparse full-vocabulary tensor, -inf except the k
                       retrieved logits at their indices          (Section 3)
  * :func:`sample_sorted`, :func:`sample` -- top-k sampling with temperature,
                       top-p and min-p on the k candidates, one uniform per
                       draw                                       (Sections 2-4)
  * :func:`philox4x32_10`, :func:`uniform` -- the counter-based generator that
                       gives each (seed, step, query) its uniform
  * :func:`quantize_e4m3`, :func:`logits_e4m3`, :func:`topk_e4m3` -- the head
                       on rows stored as e4m3 codes with one fp32 scale each
  * :func:`recall_hits`, :func:`recall_at_k` -- Recall@k bookkeeping: how
                       many exact top-k indices an approximate search
                       returned                                   (Section 4.3)

Parity of :func:`topk` against the paper cannot be pinned to printed values
(the paper prints no worked example); it is pinned instead to hand-worked
cases, exact rational brute force, Cauchy-Schwarz planted cases, library
argmax/sort special cases and the sparse-softmax identity (tests/test_oracle_*).
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False, src: str = _SRC, out: str = _LIB) -> str:
    """Compile oracle.c (or another C file with the same exports) with gcc."""
    if force or not os.path.exists(out) or os.path.getmtime(out) < os.path.getmtime(src):
        tmp = out + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-fPIC", "-shared",
               src, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, out)
    return out


def _ptr(a: np.ndarray) -> int:
    return a.ctypes.data


def _check_inputs(W_bits: np.ndarray, h: np.ndarray):
    if W_bits.dtype != np.uint16 or W_bits.ndim != 2:
        raise TypeError("W_bits must be a 2-D uint16 array of bf16 bit patterns")
    if h.dtype != np.float32:
        raise TypeError("h must be float32")
    W_bits = np.ascontiguousarray(W_bits)
    h = np.ascontiguousarray(h.reshape(-1, W_bits.shape[1]))
    return W_bits, h


class OracleLib:
    """ctypes marshalling around one compiled copy of the oracle."""

    def __init__(self, path: str):
        lib = ctypes.CDLL(path)
        P = ctypes.c_void_p
        lib.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
        lib.oracle_bf16_to_double.restype = ctypes.c_double
        lib.oracle_logits.argtypes = [P, ctypes.c_int64, ctypes.c_int32, P, ctypes.c_int32, P,
                                      ctypes.c_int32]
        lib.oracle_logits.restype = ctypes.c_int
        lib.oracle_topk.argtypes = [P, ctypes.c_int64, ctypes.c_int32, P, ctypes.c_int32,
                                    ctypes.c_int32, P, P, ctypes.c_int32]
        lib.oracle_topk.restype = ctypes.c_int
        lib.oracle_scatter.argtypes = [P, P, ctypes.c_int32, ctypes.c_int32, ctypes.c_int64, P]
        lib.oracle_scatter.restype = ctypes.c_int
        lib.oracle_max_threads.argtypes = []
        lib.oracle_max_threads.restype = ctypes.c_int
        lib.oracle_philox4x32_10.argtypes = [P, P, P]
        lib.oracle_philox4x32_10.restype = None
        lib.oracle_uniform.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint32]
        lib.oracle_uniform.restype = ctypes.c_double
        D = ctypes.c_double
        lib.oracle_sample_sorted.argtypes = [P, ctypes.c_int32, D, D, D, D, P, P, P]
        lib.oracle_sample_sorted.restype = ctypes.c_int
        lib.oracle_e4m3_to_double.argtypes = [ctypes.c_uint8]
        lib.oracle_e4m3_to_double.restype = ctypes.c_double
        lib.oracle_f32_to_e4m3.argtypes = [ctypes.c_float]
        lib.oracle_f32_to_e4m3.restype = ctypes.c_uint8
        lib.oracle_quantize_e4m3.argtypes = [P, ctypes.c_int64, ctypes.c_int32, P, P]
        lib.oracle_quantize_e4m3.restype = ctypes.c_int
        lib.oracle_logits_e4m3.argtypes = [P, P, ctypes.c_int64, ctypes.c_int32, P, ctypes.c_int32,
                                           P, ctypes.c_int32]
        lib.oracle_logits_e4m3.restype = ctypes.c_int
        lib.oracle_topk_e4m3.argtypes = [P, P, ctypes.c_int64, ctypes.c_int32, P, ctypes.c_int32,
                                         ctypes.c_int32, P, P, ctypes.c_int32]
        lib.oracle_topk_e4m3.restype = ctypes.c_int
        lib.oracle_recall_hits.argtypes = [P, ctypes.c_int32, P, ctypes.c_int32, ctypes.c_int64, P]
        lib.oracle_recall_hits.restype = ctypes.c_int
        self.lib = lib
        self.path = path

    def max_threads(self) -> int:
        return int(self.lib.oracle_max_threads())

    def bf16_to_double(self, bits: int) -> float:
        """Exact widening of one bf16 bit pattern."""
        return float(self.lib.oracle_bf16_to_double(int(bits) & 0xFFFF))

    def logits(self, W_bits: np.ndarray, h: np.ndarray, threads: int = 0) -> np.ndarray:
        """fp64 logits [batch, V] of z = W_out h (Section 3)."""
        W_bits, h = _check_inputs(W_bits, h)
        V, d = W_bits.shape
        out = np.empty((h.shape[0], V), dtype=np.float64)
        rc = self.lib.oracle_logits(_ptr(W_bits), V, d, _ptr(h), h.shape[0], _ptr(out),
                                    threads or self.max_threads())
        if rc != 0:
            raise ValueError(f"oracle_logits failed with code {rc}")
        return out

    def topk(self, W_bits: np.ndarray, h: np.ndarray, k: int, threads: int = 0):
        """Exact top-k by full sort: (idx int32 [batch,k], logits fp64 [batch,k])."""
        W_bits, h = _check_inputs(W_bits, h)
        V, d = W_bits.shape
        b = h.shape[0]
        idx = np.empty((b, max(k, 0)), dtype=np.int32)
        val = np.empty((b, max(k, 0)), dtype=np.float64)
        rc = self.lib.oracle_topk(_ptr(W_bits), V, d, _ptr(h), b, k, _ptr(idx), _ptr(val),
                                  threads or self.max_threads())
        if rc != 0:
            raise ValueError(f"oracle_topk failed with code {rc}")
        return idx, val

    def scatter(self, idx: np.ndarray, logits_f32: np.ndarray, V: int):
        """Sparse [batch, V] fp32 tensor; returns (out, ok) where ok is False if
        an index was out of range (that entry is skipped)."""
        idx = np.ascontiguousarray(idx, dtype=np.int32)
        logits_f32 = np.ascontiguousarray(logits_f32, dtype=np.float32)
        if idx.ndim == 1:
            idx = idx[None, :]
            logits_f32 = logits_f32[None, :]
        b, k = idx.shape
        out = np.empty((b, V), dtype=np.float32)
        rc = self.lib.oracle_scatter(_ptr(idx), _ptr(logits_f32), b, k, V, _ptr(out))
        if rc not in (0, 1):
            raise ValueError(f"oracle_scatter failed with code {rc}")
        return out, rc == 0


    def philox4x32_10(self, ctr, key):
        """Philox4x32-10 of a 4-word counter and a 2-word key: 4 uint32 words."""
        c = np.ascontiguousarray(ctr, dtype=np.uint32)
        kk = np.ascontiguousarray(key, dtype=np.uint32)
        out = np.empty(4, dtype=np.uint32)
        self.lib.oracle_philox4x32_10(_ptr(c), _ptr(kk), _ptr(out))
        return out

    def uniform(self, seed: int, step: int, q: int) -> float:
        """The uniform in [0, 1) of query q at decode step `step` under `seed`."""
        return float(self.lib.oracle_uniform(seed & (2**64 - 1), step & (2**64 - 1), q))

    def sample_sorted(self, z, T: float, top_p: float, min_p: float, u: float):
        """One draw from sorted candidate logits z: (position j, its
        probability among the kept candidates, number kept)."""
        z = np.ascontiguousarray(z, dtype=np.float64)
        j = ctypes.c_int32()
        prob = ctypes.c_double()
        kept = ctypes.c_int32()
        rc = self.lib.oracle_sample_sorted(_ptr(z), z.shape[0], T, top_p, min_p, u,
                                           ctypes.byref(j), ctypes.byref(prob), ctypes.byref(kept))
        if rc != 0:
            raise ValueError(f"oracle_sample_sorted failed with code {rc}")
        return j.value, prob.value, kept.value

    def sample(self, z, T: float, top_p: float, min_p: float, seed: int, step: int):
        """Draws for a batch of sorted candidate rows z [batch, k], query q
        using uniform(seed, step, q): (positions, probabilities, kept, u)."""
        z = np.atleast_2d(np.asarray(z, dtype=np.float64))
        res = [self.sample_sorted(z[q], T, top_p, min_p, self.uniform(seed, step, q))
               for q in range(z.shape[0])]
        u = np.array([self.uniform(seed, step, q) for q in range(z.shape[0])])
        return (np.array([r[0] for r in res], np.int32), np.array([r[1] for r in res]),
                np.array([r[2] for r in res], np.int32), u)


    def e4m3_to_double(self, code: int) -> float:
        """Exact value of one e4m3 code (NaN for 0x7f / 0xff)."""
        return float(self.lib.oracle_e4m3_to_double(int(code) & 0xFF))

    def f32_to_e4m3(self, x: float) -> int:
        """Nearest e4m3 code of an fp32 value (ties to even, saturated at 448)."""
        return int(self.lib.oracle_f32_to_e4m3(float(np.float32(x))))

    def quantize_e4m3(self, W_bits: np.ndarray):
        """Per-row e4m3 quantisation of bf16 rows: (codes uint8 [V, d], scales fp32 [V])."""
        W_bits = np.ascontiguousarray(W_bits, dtype=np.uint16)
        V, d = W_bits.shape
        q = np.empty((V, d), dtype=np.uint8)
        sc = np.empty(V, dtype=np.float32)
        rc = self.lib.oracle_quantize_e4m3(_ptr(W_bits), V, d, _ptr(q), _ptr(sc))
        if rc != 0:
            raise ValueError(f"oracle_quantize_e4m3 failed with code {rc}")
        return q, sc

    def logits_e4m3(self, q: np.ndarray, scale: np.ndarray, h: np.ndarray, threads: int = 0):
        """fp64 logits [batch, V] of the quantised head."""
        q = np.ascontiguousarray(q, dtype=np.uint8)
        scale = np.ascontiguousarray(scale, dtype=np.float32)
        V, d = q.shape
        h = np.ascontiguousarray(np.asarray(h, dtype=np.float32).reshape(-1, d))
        out = np.empty((h.shape[0], V), dtype=np.float64)
        rc = self.lib.oracle_logits_e4m3(_ptr(q), _ptr(scale), V, d, _ptr(h), h.shape[0], _ptr(out),
                                         threads or self.max_threads())
        if rc != 0:
            raise ValueError(f"oracle_logits_e4m3 failed with code {rc}")
        return out

    def topk_e4m3(self, q: np.ndarray, scale: np.ndarray, h: np.ndarray, k: int, threads: int = 0):
        """Exact top-k of the quantised head: (idx int32 [batch,k], logits fp64 [batch,k])."""
        q = np.ascontiguousarray(q, dtype=np.uint8)
        scale = np.ascontiguousarray(scale, dtype=np.float32)
        V, d = q.shape
        h = np.ascontiguousarray(np.asarray(h, dtype=np.float32).reshape(-1, d))
        b = h.shape[0]
        idx = np.empty((b, k), dtype=np.int32)
        val = np.empty((b, k), dtype=np.float64)
        rc = self.lib.oracle_topk_e4m3(_ptr(q), _ptr(scale), V, d, _ptr(h), b, k, _ptr(idx), _ptr(val),
                                       threads or self.max_threads())
        if rc != 0:
            raise ValueError(f"oracle_topk_e4m3 failed with code {rc}")
        return idx, val

    def recall_hits(self, exact: np.ndarray, approx: np.ndarray) -> np.ndarray:
        """Per query, how many of the exact top-k indices [n, k] are among the
        approximate candidates [n, m] (a set; negative entries are empty)."""
        exact = np.ascontiguousarray(np.atleast_2d(exact), dtype=np.int32)
        approx = np.ascontiguousarray(np.atleast_2d(approx), dtype=np.int32)
        if exact.shape[0] != approx.shape[0]:
            raise ValueError("exact and approx must have one row per query each")
        n, k = exact.shape
        m = approx.shape[1]
        hits = np.empty(n, dtype=np.int32)
        rc = self.lib.oracle_recall_hits(_ptr(exact), k, _ptr(approx), m, n, _ptr(hits))
        if rc != 0:
            raise ValueError(f"oracle_recall_hits failed with code {rc}")
        return hits

    def recall_at_k(self, exact: np.ndarray, approx: np.ndarray) -> float:
        """Recall@k over the queries: total hits / (n k)."""
        hits = self.recall_hits(exact, approx)
        exact = np.atleast_2d(exact)
        return float(hits.sum()) / (exact.shape[0] * exact.shape[1])


def _default() -> OracleLib:
    global _lib
    with _lock:
        if _lib is None:
            _lib = OracleLib(build())
    return _lib


def max_threads() -> int:
    return _default().max_threads()


def bf16_to_double(bits: int) -> float:
    return _default().bf16_to_double(bits)


def logits(W_bits, h, threads: int = 0):
    return _default().logits(W_bits, h, threads)


def topk(W_bits, h, k: int, threads: int = 0):
    return _default().topk(W_bits, h, k, threads)


def scatter(idx, logits_f32, V: int):
    return _default().scatter(idx, logits_f32, V)


def philox4x32_10(ctr, key):
    return _default().philox4x32_10(ctr, key)


def uniform(seed: int, step: int, q: int) -> float:
    return _default().uniform(seed, step, q)


def sample_sorted(z, T: float, top_p: float, min_p: float, u: float):
    return _default().sample_sorted(z, T, top_p, min_p, u)


def sample(z, T: float, top_p: float, min_p: float, seed: int, step: int):
    return _default().sample(z, T, top_p, min_p, seed, step)


def quantize_e4m3(W_bits):
    return _default().quantize_e4m3(W_bits)


def logits_e4m3(q, scale, h, threads: int = 0):
    return _default().logits_e4m3(q, scale, h, threads)


def topk_e4m3(q, scale, h, k: int, threads: int = 0):
    return _default().topk_e4m3(q, scale, h, k, threads)


def recall_hits(exact, approx):
    return _default().recall_hits(exact, approx)


def recall_at_k(exact, approx) -> float:
    return _default().recall_at_k(exact, approx)
