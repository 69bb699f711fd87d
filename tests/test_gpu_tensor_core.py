"""GPU parity of the batched (tensor-core) path and of its merge in the last
CTA: path selection, the largest k of the path, two query groups, and inputs
whose winners crowd into a few per-CTA lists, which the warp merge cannot
settle from the lists' heads and hands to the full merge."""
import numpy as np
import pytest

from gpu_cases import assert_parity, run_head, to_device_bits, workload
from paper_2608_27460_gb300 import synth

pytestmark = pytest.mark.gpu


def test_plan_selects_paths(vie):
    W, _ = workload(20011, 640, 1, seed=3)
    with vie.Head(to_device_bits(W)) as head:
        p = head.plan(1, 50)
        assert (p.path, p.groups, p.launches) == (0, 1, 1)
        p = head.plan(2, 50)  # query prep, then the projection
        assert (p.path, p.groups, p.launches) == (1, 1, 2)
        p = head.plan(40, 50)  # one 64-query group: one pass over W
        assert (p.path, p.groups, p.launches) == (1, 1, 2)
        p = head.plan(40, 65)  # k above the 64-query tile's lists: 32 + 8
        assert (p.path, p.groups, p.launches) == (1, 2, 4)
        p = head.plan(100, 50)  # 64 + 36
        assert (p.path, p.groups, p.launches) == (1, 2, 4)
        p = head.plan(4, 129)  # above the tensor-core path's k
        assert p.path == 0


@pytest.mark.parametrize("V,d,batch,k", [
    (20011, 512, 3, 128),    # largest k of the tensor-core path
    (20011, 512, 3, 129),    # smallest k above it (streaming path)
    (30011, 256, 40, 50),    # 64-query tile, four queries per selector warp
    (30011, 256, 64, 64),    # full 64-query tile at its largest k
    (30011, 256, 40, 65),    # two 32-query groups, two queries per selector warp
    (20011, 1152, 100, 50),  # 64 + 36 queries
    (30011, 256, 32, 1),     # greedy, full group of 32
    (50021, 1024, 17, 77),
    (100, 64, 4, 50),        # one tile: most CTAs draw nothing and write empty lists
    (64, 128, 2, 64),        # k = V on one CTA
    (200, 256, 40, 64),      # 64-query tile over two tiles
    (129, 128, 8, 128),      # largest k, a one-row last tile
])
def test_tensor_core_parity(vie, V, d, batch, k):
    W, h = workload(V, d, batch, seed=V + batch + k)
    assert_parity(vie, W, h, k, reps=2)


def _crowded(V, d, batch, rows, seed):
    """Rows `rows` scaled by 64 (exact in bf16): the winners of every query
    sit in one or two 128-row tiles, so in one or two per-CTA lists."""
    W, h = workload(V, d, batch, seed=seed)
    f = synth.bf16_bits_to_f32(W)
    f[rows] *= 64.0
    return synth.f32_to_bf16_bits(f), h


@pytest.mark.parametrize("batch,k", [(1, 50), (4, 50), (4, 128), (20, 50), (40, 50)])
@pytest.mark.parametrize("where", ["head", "tail"])
def test_crowded_winners_take_the_full_merge(vie, batch, k, where):
    V, d = 40009, 256
    rows = np.arange(0, 200) if where == "head" else np.arange(V - 200, V)
    W, h = _crowded(V, d, batch, rows, seed=11 + batch + k)
    idx, _, _ = assert_parity(vie, W, h, k)
    assert np.isin(idx[:, :20], rows).all()  # the scaled rows do win


def test_all_rows_equal_full_groups(vie):
    """Every logit equal, in 32- and 64-query tiles: every query leaves the
    fast merge for the full merge, which ranks by index."""
    V, d = 30011, 64
    row = synth.f32_to_bf16_bits(np.full(d, 0.25, np.float32))
    W = np.tile(row, (V, 1))
    for b, k in ((20, 1), (20, 128), (48, 64)):
        h = np.ones((b, d), np.float32)
        idx, val = run_head(vie, W, h, k)
        np.testing.assert_array_equal(idx, np.tile(np.arange(k, dtype=np.int32), (b, 1)))
        assert np.all(val == np.float32(0.25 * d))
