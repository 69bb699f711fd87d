"""Acceptance of a top-k result against the oracle's fp64 logits.

Tolerance on a logit x: tol(x) = 2e-3 + 1e-3 * |x| (fp32 accumulation of a
bf16 x fp32 product).  For one query with oracle scores sorted
s_1 >= s_2 >= ... >= s_V (ties by ascending index):

  * every returned (i, v): |v - z[i]| <= tol(z[i]), i in [0, V), no repeats;
  * returned values are non-increasing, equal values in ascending index;
  * if s_k - s_{k+1} >= tol(s_k) the returned index set equals the oracle's;
    otherwise every oracle index with z > s_k + tol(s_k) is returned and every
    returned index has z >= s_k - tol(s_k)  (near-ties at rank k).
"""
import numpy as np

ABS_TOL = 2e-3
REL_TOL = 1e-3


def tol(x):
    return ABS_TOL + REL_TOL * np.abs(x)


def oracle_order(z_row: np.ndarray) -> np.ndarray:
    """All rows ordered by (z desc, index asc) from the oracle's fp64 logits."""
    return np.lexsort((np.arange(len(z_row)), -z_row))


def check_topk(idx, val, z_row, k, order=None):
    """Returns a list of failure messages (empty when the result is accepted)."""
    idx = np.asarray(idx).astype(np.int64).reshape(-1)
    val = np.asarray(val).astype(np.float64).reshape(-1)
    z_row = np.asarray(z_row, dtype=np.float64)
    V = len(z_row)
    errs = []
    if idx.shape != (k,) or val.shape != (k,):
        return [f"shape {idx.shape}/{val.shape} != ({k},)"]
    if np.any(idx < 0) or np.any(idx >= V):
        return [f"index out of range: {idx[(idx < 0) | (idx >= V)][:5]}"]
    if len(np.unique(idx)) != k:
        errs.append("repeated index")
    zi = z_row[idx]
    bad = np.abs(val - zi) > tol(zi)
    if np.any(bad):
        j = int(np.argmax(bad))
        errs.append(f"logit mismatch at rank {j}: idx {idx[j]} got {val[j]!r} want {zi[j]!r}")
    dv = np.diff(val)
    if np.any(dv > 0):
        errs.append(f"values not descending at rank {int(np.argmax(dv > 0))}")
    same = dv == 0
    if np.any(same & (np.diff(idx) < 0)):
        errs.append("equal values not in ascending index order")
    if order is None:
        order = oracle_order(z_row)
    s_k = z_row[order[k - 1]]
    if k == V:
        if set(idx.tolist()) != set(range(V)):
            errs.append("k == V but not every index returned")
        return errs
    s_k1 = z_row[order[k]]
    t = tol(s_k)
    want = set(order[:k].tolist())
    got = set(idx.tolist())
    if s_k - s_k1 >= t:
        if got != want:
            errs.append(f"index set differs: missing {sorted(want - got)[:5]}, extra {sorted(got - want)[:5]}")
    else:
        clear = set(np.flatnonzero(z_row > s_k + t).tolist())
        if not clear <= got:
            errs.append(f"near-tie case: clear winners missing {sorted(clear - got)[:5]}")
        if np.any(zi < s_k - t):
            errs.append("near-tie case: returned an index below s_k - tol")
    return errs


def check_batch(idx, val, z, k):
    """check_topk for every query of a batch; returns {query: messages}."""
    out = {}
    for q in range(z.shape[0]):
        e = check_topk(idx[q], val[q], z[q], k)
        if e:
            out[q] = e
    return out
