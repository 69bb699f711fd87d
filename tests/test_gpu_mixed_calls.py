"""Back-to-back calls on one handle that switch between the streaming and the
tensor-core kernels (and their batch tiles) on one stream, with no
synchronisation in between: the per-handle counters that each launch re-arms
in its last CTA, and programmatic dependent launch across kernels, must leave
every result equal to what the same call gives alone."""
import numpy as np
import pytest

import oracle
from acceptance import check_topk
from gpu_cases import to_device_bits, workload

pytestmark = pytest.mark.gpu

CALLS = [(1, 50), (4, 50), (1, 300), (40, 50), (1, 50), (9, 128), (2, 1), (64, 64), (3, 300), (1, 7)]


@pytest.mark.parametrize("storage", ["bf16", "e4m3"])
def test_mixed_paths_back_to_back(vie, storage):
    import torch
    V, d = 30011, 512
    W, h = workload(V, d, 64, seed=83)
    hd = torch.from_numpy(h).cuda()
    with vie.Head(to_device_bits(W), storage=storage) as head:
        # each call alone first
        alone = []
        for b, k in CALLS:
            i, v = head.topk(hd[:b], k)
            torch.cuda.synchronize()
            alone.append((i.cpu().numpy(), v.cpu().numpy()))
        paths = {head.plan(b, k).path for b, k in CALLS}
        assert paths == {0, 1}
        # then all of them back to back, twice over, sparse tensors included
        outs = []
        for rep in range(2):
            for b, k in CALLS:
                if rep:
                    outs.append(head.topk_sparse(hd[:b], k))
                else:
                    outs.append(head.topk(hd[:b], k))
        torch.cuda.synchronize()
        assert head.device_status() == vie.VIE_OK
    for n, out in enumerate(outs):
        ai, av = alone[n % len(CALLS)]
        np.testing.assert_array_equal(out[0].cpu().numpy(), ai)
        np.testing.assert_array_equal(out[1].cpu().numpy().view(np.uint32), av.view(np.uint32))
    if storage == "e4m3":
        q, sc = oracle.quantize_e4m3(W)
        z = oracle.logits_e4m3(q, sc, h)
    else:
        z = oracle.logits(W, h)
    for (b, k), (ai, av) in zip(CALLS, alone):
        for r in range(b):
            assert not check_topk(ai[r], av[r], z[r], k), (b, k, r)
