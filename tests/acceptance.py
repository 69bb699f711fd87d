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


def oracle_order_top(z_row: np.ndarray, k: int) -> np.ndarray:
    """The first min(k + 1, V) entries of oracle_order(z_row), without sorting
    all V rows: t = the (k+1)-th largest value; every row above t, then the
    rows equal to t by ascending index, ordered by (z desc, index asc).
    Exact, ties included (the partition is by value only)."""
    V = len(z_row)
    m = min(k + 1, V)
    if m >= V:
        return oracle_order(z_row)
    t = np.partition(z_row, V - m)[V - m]  # the m-th largest value
    above = np.flatnonzero(z_row > t)
    at = np.flatnonzero(z_row == t)[: m - len(above)]  # ascending index
    cand = np.concatenate([above, at])
    return cand[np.lexsort((cand, -z_row[cand]))]


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


def check_draw(z, T, top_p, min_p, u, j, prob, tol=None):
    """Acceptance of one top-k draw made in fp32: z the query's candidate
    logits (sorted, best first), u its uniform, j the position drawn and
    prob its reported probability.  The reference is the oracle's fp64
    definition; where a decision lies within `tol` of a boundary (the
    top-p or min-p cut, or the CDF crossing u * M) every outcome reachable
    by moving that boundary by tol is accepted.  Returns a list of problems
    (empty when the draw is acceptable)."""
    import oracle
    z = np.asarray(z, dtype=np.float64)
    k = z.shape[0]
    if tol is None:
        tol = 1e-6 + 2e-7 * k
    s = z / T
    e = np.exp(s - s[0])
    p = e / e.sum()
    C = np.cumsum(p)
    ok_n = set()
    for tp_try in (top_p - tol, top_p, top_p + tol):
        n_p = next((n for n in range(1, k + 1) if C[n - 1] >= min(tp_try, 1.0)), k)
        for mp_try in (min_p - tol, min_p, min_p + tol):
            n_m = int(np.sum(p >= max(mp_try, 0.0) * p[0]))
            ok_n.add(max(1, min(n_p, n_m)))
    ok_j = {}
    for n in ok_n:
        M = C[n - 1]
        for ut in (u - tol, u, u + tol):
            ut = min(max(ut, 0.0), 1.0 - 1e-12)
            jj = next((i for i in range(n) if C[i] > ut * M), n - 1)
            ok_j.setdefault(jj, []).append(p[jj] / M)
    problems = []
    if j not in ok_j:
        problems.append(f"position {j} not drawable (acceptable {sorted(ok_j)})")
    elif min(abs(prob - q) for q in ok_j[j]) > 1e-5 + 1e-4 * max(ok_j[j]):
        problems.append(f"probability {prob} vs {ok_j[j]}")
    # the oracle itself must be among the accepted outcomes
    jo, po, _ = oracle.sample_sorted(z, T, top_p, min_p, u)
    if jo not in ok_j:
        problems.append(f"oracle draw {jo} outside the accepted set {sorted(ok_j)}")
    return problems
