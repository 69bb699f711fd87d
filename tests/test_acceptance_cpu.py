"""The acceptance rule accepts the oracle's own answer and rejects the
mistakes a GPU path could make (CPU only)."""
import numpy as np

import oracle
from acceptance import check_topk, tol
from paper_2608_27460_gb300 import synth


def _case(seed=3, V=5000, d=48, k=50):
    W, _ = synth.make_weights(V, d, seed=seed)
    h, _ = synth.make_queries(W, 1, seed=seed + 1)
    z = oracle.logits(W, h)[0]
    idx, val = oracle.topk(W, h, k)
    return z, idx[0], val[0].astype(np.float32)


def test_accepts_oracle_answer():
    z, idx, val = _case()
    assert check_topk(idx, val, z, 50) == []


def test_accepts_values_within_tolerance():
    z, idx, val = _case()
    v = val.astype(np.float64) - 0.5 * tol(val)
    # keep descending order after the perturbation
    v = np.minimum.accumulate(v)
    assert check_topk(idx, v, z, 50) == []


def test_rejects_wrong_value():
    z, idx, val = _case()
    v = val.copy()
    v[10] += 0.05
    v[:11] = np.maximum.accumulate(v[:11][::-1])[::-1]
    assert check_topk(idx, v, z, 50)


def test_rejects_missing_clear_winner():
    z, idx, val = _case()
    order = np.lexsort((np.arange(len(z)), -z))
    i2 = idx.copy()
    i2[0] = order[400]
    assert check_topk(i2, val, z, 50)


def test_rejects_unsorted_and_repeats():
    z, idx, val = _case()
    assert check_topk(idx[::-1], val[::-1], z, 50)
    i2 = idx.copy()
    i2[1] = i2[0]
    assert check_topk(i2, val, z, 50)


def test_rejects_out_of_range():
    z, idx, val = _case()
    i2 = idx.copy()
    i2[3] = len(z)
    assert check_topk(i2, val, z, 50)


def test_near_tie_at_rank_k_accepts_either():
    z = np.array([5.0, 4.0, 3.0, 2.0005, 2.0, 1.0])
    # k = 4: s_4 - s_5 = 5e-4 < tol, so {0,1,2,4} is as good as {0,1,2,3}
    assert check_topk([0, 1, 2, 3], [5, 4, 3, 2.0005], z, 4) == []
    assert check_topk([0, 1, 2, 4], [5, 4, 3, 2.0], z, 4) == []
    assert check_topk([0, 1, 3, 4], [5, 4, 2.0005, 2.0], z, 4)


def test_equal_values_need_ascending_index():
    z = np.array([1.0, 3.0, 3.0, 0.0])
    assert check_topk([1, 2], [3.0, 3.0], z, 2) == []
    assert check_topk([2, 1], [3.0, 3.0], z, 2)


def test_partial_order_equals_full_order():
    """oracle_order_top is the prefix of the full (z desc, index asc) order,
    with exact ties at and around rank k, k = 1, k = V - 1 and k >= V."""
    import numpy as np
    from acceptance import oracle_order, oracle_order_top
    rng = np.random.default_rng(5)
    for trial in range(200):
        V = int(rng.integers(1, 300))
        z = rng.integers(-6, 6, size=V).astype(np.float64) if trial % 2 else rng.normal(size=V)
        full = oracle_order(z)
        for k in sorted({1, max(1, V // 3), max(1, V - 1), V, V + 2}):
            got = oracle_order_top(z, k)
            np.testing.assert_array_equal(got, full[:min(k + 1, V)])
