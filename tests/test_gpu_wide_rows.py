"""The widest rows the library serves, on every path, against the oracle.

At d = VIE_D_MAX = 16384 a bf16 row is 32 KB, so the streaming kernel's
weight stages shrink to two rows (five for e4m3 rows) beside the 64 KB of
staged query; the tensor-core kernel walks 256 K-blocks per tile.  e4m3
rows wider than 3072 codes no longer let the 4-query tile hold its query
pieces in shared memory, so those calls take the piece-prep kernel and two
launches.  V is odd and not a multiple of 128: the last stage and the last
tile are partial."""
import pytest

from gpu_cases import assert_parity, to_device_bits, workload
from test_gpu_e4m3 import _parity as e4m3_parity

pytestmark = pytest.mark.gpu

V = 3001


@pytest.mark.parametrize("batch,k,path", [(1, 50, 0), (3, 50, 1), (2, 300, 0)])
def test_widest_bf16_rows(vie, batch, k, path):
    d = vie.VIE_D_MAX
    W, h = workload(V, d, batch, seed=d + 7 * batch + k)
    with vie.Head(to_device_bits(W)) as head:
        assert head.plan(batch, k).path == path
    assert_parity(vie, W, h, k, reps=2)


@pytest.mark.parametrize("d,batch,k,path,launches", [
    (4104, 1, 50, 1, 2),     # 4-query tile, pieces from the prep kernel
    (4104, 4, 50, 1, 2),
    (16384, 3, 50, 1, 2),
    (16384, 1, 200, 0, 1),   # streaming kernel, five-row stages
])
def test_wide_e4m3_rows(vie, d, batch, k, path, launches):
    W, h = workload(V, d, batch, seed=d + 5 * batch + k)
    with vie.Head(to_device_bits(W), storage="e4m3") as head:
        plan = head.plan(batch, k)
        assert (plan.path, plan.launches) == (path, launches)
    e4m3_parity(vie, W, h, k, reps=2)
