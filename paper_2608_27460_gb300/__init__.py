"""Exact LLM output head for GB300: Python binding of ``libviehead.so``.

The computation (paper, Section 3): z = W_out h over the whole vocabulary,
the k largest logits (exhaustive maximum inner product search), and the
sparse full-vocabulary tensor holding those k logits with -inf elsewhere.
Every step runs in the CUDA kernels of ``libviehead.so``; this module only
marshals arguments through ctypes.  There is no CPU fallback: if the library
cannot be built or loaded, :func:`load` raises.

Functions named like the C ABI (``vie_head_create`` ...) take raw pointers
(ints) and return the ``vie_status`` code; :class:`Head` wraps them for
torch tensors and raises :class:`VieError` on failure.
"""
from __future__ import annotations

import ctypes
import os
import threading

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libviehead.so")

VIE_OK = 0
VIE_ERR_INVALID_ARG = 1
VIE_ERR_UNSUPPORTED = 2
VIE_ERR_CUDA = 3
VIE_ERR_OOM = 4
VIE_ERR_DEVICE = 5
VIE_DTYPE_BF16 = 0
VIE_K_MAX = 1024
VIE_BATCH_MAX = 1024
VIE_D_MAX = 16384
VIE_MANY_MAX = 1 << 24
VIE_RECALL_N_MAX = 1 << 28
VIE_RECALL_M_MAX = 1 << 20

# Launch options (vie_launch_option): tuning and test hooks, never results.
VIE_OPT_STAGE_MIN_KB = 0
VIE_OPT_STATIC_PCT = 1
VIE_OPT_POOL_DIV = 2
VIE_OPT_TC_MIN_BATCH = 3
VIE_OPT_TC_KPS = 4
VIE_OPT_TC_MIN_BATCH_E4M3 = 5
VIE_OPT_HALF_ROWS = 6
VIE_OPT_HOST_H_DIRECT = 7
VIE_OPT_EARLY_MERGE = 8
VIE_OPT_COUNT = 9
VIE_OPT_DEFAULT = -(2 ** 31)

STATUS_NAMES = {0: "VIE_OK", 1: "VIE_ERR_INVALID_ARG", 2: "VIE_ERR_UNSUPPORTED",
                3: "VIE_ERR_CUDA", 4: "VIE_ERR_OOM", 5: "VIE_ERR_DEVICE"}

# Every entry point of include/vie_head.h.
EXPORTS = ("vie_head_create", "vie_head_destroy", "vie_head_get_props", "vie_head_plan", "vie_head_topk",
           "vie_head_topk_sparse", "vie_head_topk_host", "vie_sample_topk", "vie_head_topk_sample",
           "vie_head_create_e4m3", "vie_head_export_e4m3", "vie_head_topk_many", "vie_recall_hits",
           "vie_head_topk_noalloc", "vie_scatter_sparse_logits", "vie_device_status",
           "vie_head_device_status", "vie_last_error", "vie_set_launch_option", "vie_get_launch_option")


class VieError(RuntimeError):
    def __init__(self, status: int, message: str):
        super().__init__(f"{STATUS_NAMES.get(status, status)}: {message}")
        self.status = status
        self.message = message


class vie_head_props(ctypes.Structure):
    _fields_ = [("V", ctypes.c_int64), ("d", ctypes.c_int32), ("d_pad", ctypes.c_int32),
                ("ctas", ctypes.c_int32), ("device", ctypes.c_int32),
                ("weight_bytes", ctypes.c_int64), ("scratch_bytes", ctypes.c_int64)]


class vie_topk_plan(ctypes.Structure):
    _fields_ = [("path", ctypes.c_int32), ("groups", ctypes.c_int32), ("launches", ctypes.c_int32)]


_lib = None
_lock = threading.Lock()


def load(path: str | None = None, build_if_missing: bool = True):
    """Load libviehead.so (building it in-tree first if it is missing or
    older than its sources).  Raises if that is impossible."""
    global _lib
    with _lock:
        if _lib is not None and path is None:
            return _lib
        p = path or LIB_PATH
        if path is None and build_if_missing:
            from . import build as _build
            if not _build.up_to_date():
                _build.build()
        if not os.path.exists(p):
            raise RuntimeError(f"CUDA extension not built: {p} is missing "
                               "(run python -m paper_2608_27460_gb300.build)")
        lib = ctypes.CDLL(p)
        P, I32, I64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64
        F32, U64 = ctypes.c_float, ctypes.c_uint64
        sig = {
            "vie_head_create": ([P, I64, I32, ctypes.c_int, ctypes.POINTER(P)], ctypes.c_int),
            "vie_head_destroy": ([P], ctypes.c_int),
            "vie_head_create_e4m3": ([P, I64, I32, ctypes.POINTER(P)], ctypes.c_int),
            "vie_head_export_e4m3": ([P, P, P, P], ctypes.c_int),
            "vie_head_get_props": ([P, ctypes.POINTER(vie_head_props)], ctypes.c_int),
            "vie_head_plan": ([P, I32, I32, ctypes.POINTER(vie_topk_plan)], ctypes.c_int),
            "vie_head_topk": ([P, P, I32, I32, P, P, P], ctypes.c_int),
            "vie_head_topk_sparse": ([P, P, I32, I32, P, P, P, P], ctypes.c_int),
            "vie_head_topk_host": ([P, P, I32, I32, P, P, P, P], ctypes.c_int),
            "vie_sample_topk": ([P, P, I32, I32, F32, F32, F32, U64, U64, P, P, P], ctypes.c_int),
            "vie_head_topk_sample": ([P, P, I32, I32, F32, F32, F32, U64, U64, P, P, P, P, P, P],
                                     ctypes.c_int),
            "vie_head_topk_noalloc": ([P, I64, I32, P, I32, I32, P, P, P], ctypes.c_int),
            "vie_head_topk_many": ([P, P, I64, I32, P, P, P], ctypes.c_int),
            "vie_recall_hits": ([P, I32, P, I32, I64, P, P], ctypes.c_int),
            "vie_scatter_sparse_logits": ([P, P, I32, I32, I64, P, P], ctypes.c_int),
            "vie_device_status": ([P], ctypes.c_int),
            "vie_head_device_status": ([P, P], ctypes.c_int),
            "vie_last_error": ([], ctypes.c_char_p),
            "vie_set_launch_option": ([ctypes.c_int, I32], ctypes.c_int),
            "vie_get_launch_option": ([ctypes.c_int, ctypes.POINTER(I32)], ctypes.c_int),
        }
        for name, (args, res) in sig.items():
            fn = getattr(lib, name)
            fn.argtypes = args
            fn.restype = res
        if path is None:
            _lib = lib
        return lib


# ---- same names as the C ABI: raw pointers in, status out -----------------

def vie_last_error() -> str:
    return load().vie_last_error().decode(errors="replace")


def vie_head_create(W_out: int, V: int, d: int, dtype: int = VIE_DTYPE_BF16):
    """Returns (status, handle)."""
    out = ctypes.c_void_p(0)
    st = load().vie_head_create(W_out, V, d, dtype, ctypes.byref(out))
    return st, out.value


def vie_head_create_e4m3(W_out: int, V: int, d: int):
    """Returns (status, handle) of a head stored as e4m3 rows with fp32 scales."""
    out = ctypes.c_void_p(0)
    st = load().vie_head_create_e4m3(W_out, V, d, ctypes.byref(out))
    return st, out.value


def vie_head_export_e4m3(head: int, codes: int, scales: int, stream: int = 0) -> int:
    return load().vie_head_export_e4m3(head, codes, scales, stream)


def vie_head_destroy(head: int) -> int:
    return load().vie_head_destroy(head)


def vie_head_get_props(head: int):
    """Returns (status, vie_head_props)."""
    props = vie_head_props()
    st = load().vie_head_get_props(head, ctypes.byref(props))
    return st, props


def vie_head_plan(head: int, batch: int, k: int):
    """Returns (status, vie_topk_plan): path (0 streaming, 1 tensor core),
    query groups and kernel launches of a top-k call of this size."""
    plan = vie_topk_plan()
    st = load().vie_head_plan(head, batch, k, ctypes.byref(plan))
    return st, plan


def vie_head_topk(head: int, h: int, batch: int, k: int, out_idx: int, out_logits: int,
                  stream: int = 0) -> int:
    return load().vie_head_topk(head, h, batch, k, out_idx, out_logits, stream)


def vie_head_topk_sparse(head: int, h: int, batch: int, k: int, out_idx: int, out_logits: int,
                         out_sparse: int, stream: int = 0) -> int:
    return load().vie_head_topk_sparse(head, h, batch, k, out_idx, out_logits, out_sparse, stream)


def vie_head_topk_host(head: int, h_host: int, batch: int, k: int, idx_host: int, logits_host: int,
                       out_sparse: int = 0, stream: int = 0) -> int:
    return load().vie_head_topk_host(head, h_host, batch, k, idx_host, logits_host, out_sparse, stream)


def vie_sample_topk(idx: int, logits: int, batch: int, k: int, temperature: float, top_p: float,
                    min_p: float, seed: int, step: int, out_token: int, out_prob: int,
                    stream: int = 0) -> int:
    return load().vie_sample_topk(idx, logits, batch, k, temperature, top_p, min_p,
                                  seed & (2**64 - 1), step & (2**64 - 1), out_token, out_prob, stream)


def vie_head_topk_sample(head: int, h: int, batch: int, k: int, temperature: float, top_p: float,
                         min_p: float, seed: int, step: int, out_idx: int, out_logits: int,
                         out_sparse: int, out_token: int, out_prob: int, stream: int = 0) -> int:
    return load().vie_head_topk_sample(head, h, batch, k, temperature, top_p, min_p,
                                       seed & (2**64 - 1), step & (2**64 - 1), out_idx, out_logits,
                                       out_sparse, out_token, out_prob, stream)


def sample_topk(idx, logits, temperature: float = 1.0, top_p: float = 1.0, min_p: float = 0.0,
                seed: int = 0, step: int = 0, out_token=None, out_prob=None, stream=None):
    """Top-k sampling on CUDA candidates (int32 / float32 [batch, k], sorted
    best first): returns (token int32 [batch], probability float32 [batch])."""
    import torch
    b, k = int(idx.shape[0]), int(idx.shape[1])
    if out_token is None:
        out_token = torch.empty((b,), dtype=torch.int32, device=idx.device)
    if out_prob is None:
        out_prob = torch.empty((b,), dtype=torch.float32, device=idx.device)
    check(vie_sample_topk(idx.data_ptr(), logits.data_ptr(), b, k, temperature, top_p, min_p, seed,
                          step, out_token.data_ptr(), out_prob.data_ptr(), _stream_ptr(stream)))
    return out_token, out_prob


def vie_head_topk_many(head: int, h: int, n: int, k: int, out_idx: int, out_logits: int,
                       stream: int = 0) -> int:
    return load().vie_head_topk_many(head, h, n, k, out_idx, out_logits, stream)


def vie_recall_hits(exact: int, k: int, approx: int, m: int, n: int, out_hits: int,
                    stream: int = 0) -> int:
    return load().vie_recall_hits(exact, k, approx, m, n, out_hits, stream)


def recall_hits(exact, approx, out_hits=None, stream=None):
    """Recall@k bookkeeping on CUDA index lists: exact int32 [n, k] and
    approx int32 [n, m] -> hits int32 [n] (how many exact indices each
    query's candidates contain; Recall@k = hits.sum() / (n k))."""
    import torch
    if exact.dim() != 2 or approx.dim() != 2 or exact.shape[0] != approx.shape[0]:
        raise ValueError("exact [n, k] and approx [n, m] must have one row per query")
    if exact.dtype != torch.int32 or approx.dtype != torch.int32 or not (exact.is_cuda and approx.is_cuda):
        raise ValueError("exact and approx must be CUDA int32 tensors")
    exact, approx = exact.contiguous(), approx.contiguous()
    n, k, m = int(exact.shape[0]), int(exact.shape[1]), int(approx.shape[1])
    if out_hits is None:
        out_hits = torch.empty((n,), dtype=torch.int32, device=exact.device)
    check(vie_recall_hits(exact.data_ptr(), k, approx.data_ptr(), m, n, out_hits.data_ptr(),
                          _stream_ptr(stream)))
    return out_hits


def vie_head_topk_noalloc(W_out: int, V: int, d: int, h: int, batch: int, k: int, out_idx: int,
                          out_logits: int, stream: int = 0) -> int:
    """Top-k straight from caller-owned weights, scratch in a fixed library
    array: for callers that must not allocate device memory."""
    return load().vie_head_topk_noalloc(W_out, V, d, h, batch, k, out_idx, out_logits, stream)


def vie_scatter_sparse_logits(idx: int, logits: int, batch: int, k: int, V: int, out: int,
                              stream: int = 0) -> int:
    return load().vie_scatter_sparse_logits(idx, logits, batch, k, V, out, stream)


def vie_device_status(stream: int = 0) -> int:
    return load().vie_device_status(stream)


def vie_head_device_status(head: int, stream: int = 0) -> int:
    return load().vie_head_device_status(head, stream)


def vie_set_launch_option(option: int, value: int) -> int:
    return load().vie_set_launch_option(option, value)


def vie_get_launch_option(option: int):
    """Returns (status, value)."""
    v = ctypes.c_int32(0)
    st = load().vie_get_launch_option(option, ctypes.byref(v))
    return st, v.value


class launch_options:
    """Context manager that sets launch options for its body and restores
    the previous values afterwards, e.g.
    ``with launch_options({VIE_OPT_TC_MIN_BATCH: 10**6}): ...`` keeps every
    batch on the streaming kernel.  Options are process-wide."""

    def __init__(self, values: dict):
        self.values = dict(values)
        self.saved = {}

    def __enter__(self):
        for o, v in self.values.items():
            st, old = vie_get_launch_option(o)
            check(st)
            self.saved[o] = old
            check(vie_set_launch_option(o, v))
        return self

    def __exit__(self, *exc):
        for o, v in self.saved.items():
            vie_set_launch_option(o, v)


def check(status: int) -> None:
    if status != VIE_OK:
        raise VieError(status, vie_last_error())


# ---- torch convenience layer ----------------------------------------------

def _stream_ptr(stream) -> int:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


class Head:
    """An output head on the current CUDA device.

    ``W`` is a CUDA tensor [V, d] of dtype bfloat16 (or int16/uint16 holding
    bf16 bit patterns).  The head keeps its own padded copy, so ``W`` may be
    freed afterwards."""

    def __init__(self, W, storage: str = "bf16"):
        """W: bf16 weights [V, d] on a CUDA device.  storage "bf16" keeps them
        as they are; "e4m3" quantises each row to e4m3 with an fp32 scale."""
        import torch
        if not W.is_cuda or W.dim() != 2:
            raise ValueError("W must be a 2-D CUDA tensor")
        if W.dtype not in (torch.bfloat16, torch.int16, torch.uint16):
            raise ValueError("W must hold bf16 values (bfloat16, or int16/uint16 bit patterns)")
        W = W.contiguous()
        self.V, self.d = int(W.shape[0]), int(W.shape[1])
        self.device = W.device
        if storage not in ("bf16", "e4m3"):
            raise ValueError(f"storage must be 'bf16' or 'e4m3', not {storage!r}")
        self.storage = storage
        with torch.cuda.device(W.device):
            if storage == "e4m3":
                st, hd = vie_head_create_e4m3(W.data_ptr(), self.V, self.d)
            else:
                st, hd = vie_head_create(W.data_ptr(), self.V, self.d, VIE_DTYPE_BF16)
        check(st)
        self._h = hd
        st, self.props = vie_head_get_props(hd)
        check(st)

    @property
    def handle(self) -> int:
        if not self._h:
            raise ValueError("head is closed")
        return self._h

    def topk(self, h, k: int, out_idx=None, out_logits=None, stream=None):
        """Top-k (indices int32 [batch, k], logits fp32 [batch, k]) of W h."""
        import torch
        if h.dim() == 1:
            h = h[None]
        if h.dtype != torch.float32 or not h.is_cuda or h.shape[1] != self.d:
            raise ValueError(f"h must be a CUDA float32 tensor [batch, {self.d}]")
        h = h.contiguous()
        b = int(h.shape[0])
        if out_idx is None:
            out_idx = torch.empty((b, k), dtype=torch.int32, device=h.device)
        if out_logits is None:
            out_logits = torch.empty((b, k), dtype=torch.float32, device=h.device)
        check(vie_head_topk(self.handle, h.data_ptr(), b, k, out_idx.data_ptr(),
                            out_logits.data_ptr(), _stream_ptr(stream)))
        return out_idx, out_logits

    def topk_many(self, h, k: int, out_idx=None, out_logits=None, stream=None):
        """Exact top-k of many hidden states h [n, d] (any n up to
        VIE_MANY_MAX), e.g. the ground truth of a Recall@k evaluation."""
        import torch
        if h.dim() != 2 or h.dtype != torch.float32 or not h.is_cuda or h.shape[1] != self.d:
            raise ValueError(f"h must be a CUDA float32 tensor [n, {self.d}]")
        h = h.contiguous()
        n = int(h.shape[0])
        if out_idx is None:
            out_idx = torch.empty((n, k), dtype=torch.int32, device=h.device)
        if out_logits is None:
            out_logits = torch.empty((n, k), dtype=torch.float32, device=h.device)
        check(vie_head_topk_many(self.handle, h.data_ptr(), n, k, out_idx.data_ptr(),
                                 out_logits.data_ptr(), _stream_ptr(stream)))
        return out_idx, out_logits

    def plan(self, batch: int, k: int):
        st, pl = vie_head_plan(self.handle, batch, k)
        check(st)
        return pl

    def topk_sparse(self, h, k: int, out_idx=None, out_logits=None, out_sparse=None, stream=None):
        """Top-k and the sparse [batch, V] logit tensor in one launch."""
        import torch
        if h.dim() == 1:
            h = h[None]
        if h.dtype != torch.float32 or not h.is_cuda or h.shape[1] != self.d:
            raise ValueError(f"h must be a CUDA float32 tensor [batch, {self.d}]")
        h = h.contiguous()
        b = int(h.shape[0])
        if out_idx is None:
            out_idx = torch.empty((b, k), dtype=torch.int32, device=h.device)
        if out_logits is None:
            out_logits = torch.empty((b, k), dtype=torch.float32, device=h.device)
        if out_sparse is None:
            out_sparse = torch.empty((b, self.V), dtype=torch.float32, device=h.device)
        check(vie_head_topk_sparse(self.handle, h.data_ptr(), b, k, out_idx.data_ptr(),
                                   out_logits.data_ptr(), out_sparse.data_ptr(), _stream_ptr(stream)))
        return out_idx, out_logits, out_sparse

    def topk_host(self, h, k: int, out_idx=None, out_logits=None, out_sparse=None, stream=None):
        """One decode step from host memory: h (CPU float32 [batch, d], best
        pinned) in, top-k (CPU int32 / float32 [batch, k]) out, ready on
        return; out_sparse, if given, is a CUDA [batch, V] tensor."""
        import torch
        if h.dim() == 1:
            h = h[None]
        if h.dtype != torch.float32 or h.is_cuda or h.shape[1] != self.d:
            raise ValueError(f"h must be a CPU float32 tensor [batch, {self.d}]")
        h = h.contiguous()
        b = int(h.shape[0])
        if out_idx is None:
            out_idx = torch.empty((b, k), dtype=torch.int32)
        if out_logits is None:
            out_logits = torch.empty((b, k), dtype=torch.float32)
        sp = 0 if out_sparse is None else out_sparse.data_ptr()
        check(vie_head_topk_host(self.handle, h.data_ptr(), b, k, out_idx.data_ptr(),
                                 out_logits.data_ptr(), sp, _stream_ptr(stream)))
        return out_idx, out_logits

    def topk_sample(self, h, k: int, temperature: float = 1.0, top_p: float = 1.0,
                    min_p: float = 0.0, seed: int = 0, step: int = 0, out_sparse=None, stream=None):
        """Top-k of W h, then one draw per query: (idx, logits, token, prob)."""
        import torch
        if h.dim() == 1:
            h = h[None]
        if h.dtype != torch.float32 or not h.is_cuda or h.shape[1] != self.d:
            raise ValueError(f"h must be a CUDA float32 tensor [batch, {self.d}]")
        h = h.contiguous()
        b = int(h.shape[0])
        idx = torch.empty((b, k), dtype=torch.int32, device=h.device)
        val = torch.empty((b, k), dtype=torch.float32, device=h.device)
        tok = torch.empty((b,), dtype=torch.int32, device=h.device)
        prob = torch.empty((b,), dtype=torch.float32, device=h.device)
        sp = 0 if out_sparse is None else out_sparse.data_ptr()
        check(vie_head_topk_sample(self.handle, h.data_ptr(), b, k, temperature, top_p, min_p, seed,
                                   step, idx.data_ptr(), val.data_ptr(), sp, tok.data_ptr(),
                                   prob.data_ptr(), _stream_ptr(stream)))
        return idx, val, tok, prob

    def export_e4m3(self, stream=None):
        """The e4m3 codes (uint8 [V, d]) and row scales (float32 [V]) of an e4m3 head."""
        import torch
        codes = torch.empty((self.V, self.d), dtype=torch.uint8, device=self.device)
        scales = torch.empty((self.V,), dtype=torch.float32, device=self.device)
        check(vie_head_export_e4m3(self.handle, codes.data_ptr(), scales.data_ptr(), _stream_ptr(stream)))
        return codes, scales

    def sparse_logits(self, idx, logits, out=None, stream=None):
        """Sparse [batch, V] fp32 tensor: -inf except logits at idx."""
        import torch
        b, k = int(idx.shape[0]), int(idx.shape[1])
        if out is None:
            out = torch.empty((b, self.V), dtype=torch.float32, device=idx.device)
        check(vie_scatter_sparse_logits(idx.data_ptr(), logits.data_ptr(), b, k, self.V,
                                        out.data_ptr(), _stream_ptr(stream)))
        return out

    def device_status(self, stream=None) -> int:
        return vie_head_device_status(self.handle, _stream_ptr(stream))

    def close(self):
        if getattr(self, "_h", None):
            vie_head_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()
