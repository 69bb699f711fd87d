"""Wide lists (k > 64) on the streaming kernel.  Each query's candidates
collect in a shared-memory buffer; whenever it fills, a bisection cuts it back
to its best k and raises the entry bound; after the stream the whole CTA sorts
it into the CTA's list.  The cases make buffers fill during the stream (many
rows per CTA against the buffer), fill groups of 8, 4 + 1 and 2 queries, tie on
the k-th logit (small-integer inputs: exact logits shared by many rows, ranked
by row), and run on e4m3 rows and through the no-alloc entry point."""
import numpy as np
import pytest

import oracle
from acceptance import check_topk
from gpu_cases import assert_parity, run_head, to_device_bits, workload
from paper_2608_27460_gb300 import synth

pytestmark = pytest.mark.gpu

def streaming(vie):
    """Every batch on the streaming kernel (the tensor cores take k <= 128 from batch 2)."""
    return vie.launch_options({vie.VIE_OPT_TC_MIN_BATCH: 100000, vie.VIE_OPT_TC_MIN_BATCH_E4M3: 100000})


@pytest.mark.parametrize("V,d,batch,k,launches", [
    (151936, 64, 1, 100, 1),    # ~1000 rows per CTA against a 256-key buffer: cut-backs
    (262144, 32, 1, 700, 1),    # ~1725 rows per CTA, a 1408-key buffer: a cut-back
    (200003, 64, 8, 129, 1),    # eight 320-key buffers
    (120011, 64, 8, 65, 1),     # the smallest wide k, eight queries
    (100003, 128, 5, 300, 2),   # groups of 4 + 1 (640-key buffers)
    (50021, 256, 2, 1024, 1),   # two 2048-key buffers, k = 1024
    (7001, 640, 1, 65, 1),      # fewer rows per CTA than the buffer holds
])
def test_wide_lists_match_the_oracle(vie, V, d, batch, k, launches):
    W, h = workload(V, d, batch, seed=V + k)
    with streaming(vie):
        with vie.Head(to_device_bits(W)) as head:
            plan = head.plan(batch, k)
            assert (plan.path, plan.launches) == (0, launches)
        assert_parity(vie, W, h, k, reps=2)


@pytest.mark.parametrize("batch,k", [(1, 200), (3, 500), (8, 129)])
def test_wide_lists_rank_exact_ties_by_row(vie, batch, k):
    """Weights in -3..3 and queries in -2..2: every logit is an exact small
    integer shared by thousands of rows, so the k-th logit is tied and the
    ranking rule (equal logits: smaller row first) decides the list, in the
    cut-backs as in the final sort."""
    rng = np.random.default_rng(11 + k)
    V, d = 120011, 48
    W = synth.f32_to_bf16_bits(rng.integers(-3, 4, size=(V, d)).astype(np.float32))
    h = rng.integers(-2, 3, size=(batch, d)).astype(np.float32)
    with streaming(vie):
        idx, val = run_head(vie, W, h, k, reps=2)
    oi, ov = oracle.topk(W, h, k)
    np.testing.assert_array_equal(idx, oi)
    np.testing.assert_array_equal(val.astype(np.float64), ov)


@pytest.mark.parametrize("V,d,batch,k", [(151936, 128, 1, 100), (100003, 256, 5, 300)])
def test_wide_lists_on_e4m3_rows(vie, V, d, batch, k):
    import torch
    W, h = workload(V, d, batch, seed=V + 3 * k)
    q, sc = oracle.quantize_e4m3(W)
    z = oracle.logits_e4m3(q, sc, h)
    with streaming(vie):
        with vie.Head(to_device_bits(W), storage="e4m3") as head:
            assert head.plan(batch, k).path == 0
            hd = torch.from_numpy(h).cuda()
            idx, val = head.topk(hd, k)
            torch.cuda.synchronize()
            assert head.device_status() == vie.VIE_OK, vie.vie_last_error()
    idx, val = idx.cpu().numpy(), val.cpu().numpy()
    fails = {b: e for b in range(batch) if (e := check_topk(idx[b], val[b], z[b], k))}
    assert not fails, next(iter(fails.items()))
