"""Pins of the oracle's Recall@k bookkeeping (Section 4.3: the share of the
exact head's top-k tokens that an approximate search also retrieves).

Each pin checks the oracle against something other than itself: hand-worked
cases, set intersection on small random cases, invariants of the definition,
and the exact head's own top-k lists."""
import os

import numpy as np
import pytest

import oracle as default_oracle
from paper_2608_27460_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "recall_hand.txt")


def load_hand():
    cases = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        km, ex, ap, hits = [part.split() for part in line.split("|")]
        k, m = int(km[0]), int(km[1])
        ex, ap = [int(x) for x in ex], [int(x) for x in ap]
        assert len(ex) == k and len(ap) == m
        cases.append((ex, ap, int(hits[0])))
    return cases


def pin_hand_worked(lib):
    cases = load_hand()
    assert len(cases) == 9
    for ex, ap, want in cases:
        assert lib.recall_hits(np.array([ex]), np.array([ap]))[0] == want, (ex, ap)


def pin_set_intersection(lib):
    """Small random cases, repeats and empty slots included, against Python
    sets: hits = #{j : exact_j >= 0 and exact_j in set(candidates)}."""
    rng = np.random.default_rng(5)
    for _ in range(200):
        n, k, m = int(rng.integers(1, 6)), int(rng.integers(1, 9)), int(rng.integers(1, 12))
        ex = np.stack([rng.choice(30, k, replace=False) for _ in range(n)]).astype(np.int32)
        ap = rng.integers(-1, 30, (n, m)).astype(np.int32)
        got = lib.recall_hits(ex, ap)
        want = [sum(1 for e in ex[q] if e >= 0 and e in set(ap[q].tolist())) for q in range(n)]
        np.testing.assert_array_equal(got, want)


def pin_invariants(lib):
    rng = np.random.default_rng(6)
    ex = np.stack([rng.choice(1000, 50, replace=False) for _ in range(8)]).astype(np.int32)
    k = ex.shape[1]
    assert np.all(lib.recall_hits(ex, ex) == k)                               # itself
    assert np.all(lib.recall_hits(ex, ex[:, ::-1].copy()) == k)              # any order
    assert np.all(lib.recall_hits(ex, np.concatenate([ex, ex], 1)) == k)     # repeats count once
    assert np.all(lib.recall_hits(ex, ex + 1000) == 0)                       # disjoint
    assert np.all(lib.recall_hits(ex, np.full((8, 7), -1, np.int32)) == 0)   # all slots empty
    assert np.all(lib.recall_hits(np.full((8, 3), -1, np.int32), np.full((8, 3), -1, np.int32)) == 0)
    # the first c candidates of the exact list give c hits; adding candidates never loses one
    for c in (1, 7, 49):
        assert np.all(lib.recall_hits(ex, ex[:, :c].copy()) == c)
    base = lib.recall_hits(ex, ex[:, :20].copy())
    more = lib.recall_hits(ex, np.concatenate([ex[:, :20], rng.integers(0, 2000, (8, 30))], 1).astype(np.int32))
    assert np.all(more >= base)
    # the candidate row of query q is matched against query q only
    shifted = np.roll(ex, 1, axis=0)
    want = [len(set(ex[q].tolist()) & set(shifted[q].tolist())) for q in range(8)]
    np.testing.assert_array_equal(lib.recall_hits(ex, shifted), want)


def pin_recall_at_k_value(lib):
    """Hits 2, 1, 0, 2 of k = 2 over four queries: Recall@2 = 5 / 8."""
    ex = np.array([[1, 2], [1, 2], [1, 2], [1, 2]], np.int32)
    ap = np.array([[2, 1, 7], [2, 9, 9], [5, 6, 7], [1, 2, -1]], np.int32)
    np.testing.assert_array_equal(lib.recall_hits(ex, ap), [2, 1, 0, 2])
    assert lib.recall_at_k(ex, ap) == 0.625


def pin_exact_head_lists(lib):
    """The exact head's top-k against its own top-(k + 8): every hit found;
    against the top-k of other queries: only the shared tokens."""
    W, _ = synth.make_weights(3000, 64, seed=12)
    h = np.random.default_rng(13).normal(0, 1, (6, 64)).astype(np.float32)
    top2, _ = lib.topk(W, h, 2)
    top10, _ = lib.topk(W, h, 10)
    assert np.all(lib.recall_hits(top2, top10) == 2)
    assert lib.recall_at_k(top10, top2) == 2 / 10
    other = np.roll(top10, 1, axis=0)
    want = [len(set(top10[q].tolist()) & set(other[q].tolist())) for q in range(6)]
    np.testing.assert_array_equal(lib.recall_hits(top10, other), want)


def pin_argument_errors(lib):
    with pytest.raises(ValueError):
        lib.recall_hits(np.zeros((2, 2), np.int32), np.zeros((3, 2), np.int32))


RECALL_PINS = [(f.__name__, f) for f in (
    pin_hand_worked, pin_set_intersection, pin_invariants, pin_recall_at_k_value, pin_exact_head_lists,
    pin_argument_errors)]


@pytest.mark.parametrize("name,pin", RECALL_PINS, ids=[n for n, _ in RECALL_PINS])
def test_recall_pin(name, pin):
    pin(default_oracle._default())
