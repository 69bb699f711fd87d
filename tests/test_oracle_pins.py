"""Pins of the CPU oracle to things other than itself.

The paper prints no worked example for the dense head, so the oracle is
pinned to: a hand-worked V=16, d=4 case (tests/golden), exact integer and
exact rational brute force on small inputs, the Cauchy-Schwarz planted case,
library argmax / lexsort special cases (k = 1, k = V), a library bf16
decoder, and the sparse-softmax identity of Section 3.
"""
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as default_oracle
from paper_2608_27460_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "hand_v16_d4.txt")


def load_hand_case():
    W, h, z, rank = {}, {}, {}, {}
    V = d = None
    with open(GOLDEN) as f:
        for line in f:
            line = line.split("#", 1)[0].split()
            if not line:
                continue
            tag, rest = line[0], line[1:]
            if tag == "V":
                V = int(rest[0])
            elif tag == "d":
                d = int(rest[0])
            elif tag == "w":
                W[int(rest[0])] = [int(x, 16) for x in rest[1:]]
            elif tag == "h":
                h[int(rest[0])] = [float(x) for x in rest[1:]]
            elif tag == "z":
                z[int(rest[0])] = [float(x) for x in rest[1:]]
            elif tag == "rank":
                rank[int(rest[0])] = [int(x) for x in rest[1:]]
    Wb = np.array([W[i] for i in range(V)], dtype=np.uint16)
    hq = np.array([h[q] for q in sorted(h)], dtype=np.float32)
    zq = np.array([z[q] for q in sorted(z)], dtype=np.float64)
    rq = np.array([rank[q] for q in sorted(rank)], dtype=np.int32)
    assert Wb.shape == (V, d) and hq.shape[1] == d
    return Wb, hq, zq, rq


def pin_hand_worked_logits_and_ranking(o):
    W, h, z, rank = load_hand_case()
    zo = o.logits(W, h)
    np.testing.assert_array_equal(zo, z)
    for k in (1, 5, 9, 16):
        idx, val = o.topk(W, h, k)
        np.testing.assert_array_equal(idx, rank[:, :k])
        np.testing.assert_array_equal(val, np.take_along_axis(z, rank[:, :k].astype(np.int64), 1))


def pin_hand_worked_sparse_tensor(o):
    W, h, z, rank = load_hand_case()
    idx, val = o.topk(W, h, 5)
    out, ok = o.scatter(idx, val.astype(np.float32), 16)
    assert ok
    for q in range(2):
        finite = np.flatnonzero(np.isfinite(out[q]))
        assert sorted(finite) == sorted(rank[q, :5])
        for j in range(5):
            assert out[q, rank[q, j]] == z[q, rank[q, j]]
        assert np.all(out[q][~np.isfinite(out[q])] == -np.inf)


def pin_bf16_decode_matches_library(o):
    torch = pytest.importorskip("torch")
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    lib = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).to(torch.float64).numpy()
    finite = np.isfinite(lib)
    ours = np.array([o.bf16_to_double(int(b)) for b in bits[finite]])
    np.testing.assert_array_equal(ours, lib[finite])
    # infinities decode too
    assert o.bf16_to_double(0x7F80) == np.inf and o.bf16_to_double(0xFF80) == -np.inf


def exact_int_case(seed, V, d, wmax=8, hmax=5):
    rng = np.random.default_rng(seed)
    Wi = rng.integers(-wmax, wmax + 1, size=(V, d))
    hi = rng.integers(-hmax, hmax + 1, size=(2, d))
    Wb = synth.f32_to_bf16_bits(Wi.astype(np.float32))
    assert np.array_equal(synth.bf16_bits_to_f32(Wb), Wi.astype(np.float32))
    z = [[sum(int(Wi[i, j]) * int(hi[q, j]) for j in range(d)) for i in range(V)] for q in range(2)]
    return Wb, hi.astype(np.float32), z


def pin_exact_integer_brute_force(o, seed, V, d):
    W, h, z = exact_int_case(seed, V, d)
    np.testing.assert_array_equal(o.logits(W, h), np.array(z, dtype=np.float64))
    for k in (1, 7, 50, V):
        if k > V:
            continue
        idx, val = o.topk(W, h, k)
        for q in range(2):
            want = sorted(range(V), key=lambda i: (-z[q][i], i))[:k]
            assert idx[q].tolist() == want
            assert val[q].tolist() == [float(z[q][i]) for i in want]


def pin_exact_rational_general_values(o):
    """General bf16 weights and fp32 queries: each fp64 logit is within the
    sequential-summation error bound of the exact rational value."""
    rng = np.random.default_rng(7)
    V, d = 200, 37
    W = synth.f32_to_bf16_bits(rng.standard_normal((V, d)).astype(np.float32) * 0.3)
    h = (rng.standard_normal((1, d)) * 4).astype(np.float32)
    Wf = synth.bf16_bits_to_f32(W).astype(np.float64)
    zo = o.logits(W, h)[0]
    hq = [Fraction(float(x)) for x in h[0]]
    u = 2.0 ** -53
    exact = []
    for i in range(V):
        terms = [Fraction(float(Wf[i, j])) * hq[j] for j in range(d)]
        e = sum(terms, Fraction(0))
        exact.append(e)
        bound = d * u * float(sum(abs(t) for t in terms)) * 1.01
        assert abs(float(Fraction(zo[i]) - e)) <= bound
    idx, _ = o.topk(W, h, 20)
    want = sorted(range(V), key=lambda i: (-exact[i], i))[:20]
    assert idx[0].tolist() == want


def pin_planted_cauchy_schwarz(o):
    """Distinct rows of equal norm and h = c * w_j: row j is ranked first and
    z_j = c * |w_j|^2 (Cauchy-Schwarz, equality only for w_i = w_j)."""
    rng = np.random.default_rng(11)
    d, V = 16, 512
    base = np.array([0.5, -0.25, 1.0, 2.0, -1.5, 0.75, 0.125, -3.0, 1.25, 0.0, 0.5, -0.5,
                     1.0, 1.75, -2.5, 0.25], dtype=np.float32)
    rows = set()
    W = []
    while len(W) < V:
        r = rng.permutation(base) * rng.choice([-1.0, 1.0], size=d)
        key = r.tobytes()
        if key not in rows:
            rows.add(key)
            W.append(r.astype(np.float32))
    Wf = np.array(W, dtype=np.float32)
    Wb = synth.f32_to_bf16_bits(Wf)
    assert np.array_equal(synth.bf16_bits_to_f32(Wb), Wf)
    norm2 = float(np.sum(base.astype(np.float64) ** 2))
    for j in (0, 17, 255, 511):
        c = 3.0
        h = (c * Wf[j])[None, :].astype(np.float32)
        idx, val = o.topk(Wb, h, 3)
        assert idx[0, 0] == j
        assert val[0, 0] == c * norm2
        assert val[0, 1] < val[0, 0]


def pin_k1_is_library_argmax_and_kV_is_library_lexsort(o):
    W, h, z = exact_int_case(21, 700, 12, wmax=3, hmax=2)  # many exact ties
    zi = np.array(z, dtype=np.int64)
    idx1, _ = o.topk(W, h, 1)
    idxV, valV = o.topk(W, h, 700)
    for q in range(2):
        assert idx1[q, 0] == int(np.argmax(zi[q]))  # first maximum = smallest index
        order = np.lexsort((np.arange(700), -zi[q]))
        np.testing.assert_array_equal(idxV[q], order)
        np.testing.assert_array_equal(valV[q], zi[q][order].astype(np.float64))


def pin_topk_invariants_on_workload_shaped_inputs(o):
    """Returned logits are the k largest of the full product, descending."""
    W, meta = synth.make_weights(4096, 64, seed=5)
    h, _ = synth.make_queries(W, 3, seed=6)
    z = o.logits(W, h)
    idx, val = o.topk(W, h, 50)
    for q in range(3):
        assert np.all(np.diff(val[q]) <= 0)
        np.testing.assert_array_equal(val[q], z[q, idx[q]])
        rest = np.setdiff1d(np.arange(4096), idx[q])
        assert z[q, rest].max() <= val[q, -1]
        assert len(set(idx[q].tolist())) == 50


def pin_sparse_softmax_identity(o):
    """Exactly k finite entries; softmax over the sparse row equals the
    renormalised softmax of the top-k logits (Section 3's reconstruction)."""
    W, _ = synth.make_weights(3000, 32, seed=9)
    h, _ = synth.make_queries(W, 2, seed=10)
    k = 50
    idx, val = o.topk(W, h, k)
    out, ok = o.scatter(idx, val.astype(np.float32), 3000)
    assert ok
    for q in range(2):
        row = out[q].astype(np.float64)
        assert np.count_nonzero(np.isfinite(row)) == k
        m = row.max()
        p = np.exp(row - m)
        p /= p.sum()
        v = val[q].astype(np.float32).astype(np.float64)
        pk = np.exp(v - v.max())
        pk /= pk.sum()
        np.testing.assert_allclose(p[idx[q]], pk, rtol=1e-12, atol=0)
        assert np.all(p[np.setdiff1d(np.arange(3000), idx[q])] == 0)


def pin_scatter_rejects_out_of_range_index(o):
    # two rows, so a wrongly accepted index 9 of row 0 still lands inside the buffer
    idx = np.array([[0, 5, 9], [1, 2, 3]], dtype=np.int32)
    vals = np.array([[1.0, 2.0, 3.0], [4.0, 5.0, 6.0]], np.float32)
    out, ok = o.scatter(idx, vals, 9)
    assert not ok
    assert out[0, 0] == 1.0 and out[0, 5] == 2.0
    assert np.count_nonzero(np.isfinite(out[0])) == 2
    assert out[1, 1] == 4.0 and out[1, 2] == 5.0 and out[1, 3] == 6.0


def pin_oracle_rejects_bad_arguments(o):
    W = np.zeros((4, 2), np.uint16)
    h = np.zeros((1, 2), np.float32)
    with pytest.raises(ValueError):
        o.topk(W, h, 5)  # k > V
    with pytest.raises(ValueError):
        o.topk(W, h, 0)


# ---------------------------------------------------------------------------
# The battery: every pin, run against one compiled copy of the oracle.
INT_CASES = [(1, 64, 8), (2, 300, 17), (3, 1024, 24)]

PINS = [
    ("hand_worked_logits_and_ranking", lambda o: pin_hand_worked_logits_and_ranking(o)),
    ("hand_worked_sparse_tensor", lambda o: pin_hand_worked_sparse_tensor(o)),
    ("bf16_decode_matches_library", lambda o: pin_bf16_decode_matches_library(o)),
    ("exact_integer_brute_force", lambda o: [pin_exact_integer_brute_force(o, *c) for c in INT_CASES]),
    ("exact_rational_general_values", lambda o: pin_exact_rational_general_values(o)),
    ("planted_cauchy_schwarz", lambda o: pin_planted_cauchy_schwarz(o)),
    ("k1_argmax_kV_lexsort", lambda o: pin_k1_is_library_argmax_and_kV_is_library_lexsort(o)),
    ("topk_invariants", lambda o: pin_topk_invariants_on_workload_shaped_inputs(o)),
    ("sparse_softmax_identity", lambda o: pin_sparse_softmax_identity(o)),
    ("scatter_rejects_out_of_range", lambda o: pin_scatter_rejects_out_of_range_index(o)),
    ("rejects_bad_arguments", lambda o: pin_oracle_rejects_bad_arguments(o)),
]


@pytest.mark.parametrize("name,pin", PINS, ids=[n for n, _ in PINS])
def test_pin(name, pin):
    pin(default_oracle)
