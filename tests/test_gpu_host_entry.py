"""vie_head_topk_host: the whole step from host memory (h in, top-k out,
ready on return) gives the same bits as the device entry points, on both
paths, with pinned buffers (read and written in place by the kernels) and
pageable ones (staged through device buffers), with and without the sparse
tensor, and when a later call needs larger staging buffers."""
import numpy as np
import pytest

import oracle
from acceptance import check_topk
from gpu_cases import to_device_bits, workload

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("batch,k", [(1, 50), (4, 50), (3, 300), (40, 64)])
@pytest.mark.parametrize("pinned", ["both", "h", "out", "none"])
@pytest.mark.parametrize("storage", ["bf16", "e4m3"])
def test_host_entry_matches_device_entry(vie, batch, k, pinned, storage):
    import torch
    if storage == "e4m3" and pinned in ("h", "out"):
        pytest.skip("the e4m3 head covers the all-pinned and all-pageable cases")
    V, d = 30011, 512
    W, h = workload(V, d, batch, seed=batch * 7 + k)
    with vie.Head(to_device_bits(W), storage=storage) as head:
        hd = torch.from_numpy(h).cuda()
        ref_i, ref_v = head.topk(hd, k)
        ref_i2, ref_v2, ref_sp = head.topk_sparse(hd, k)
        torch.cuda.synchronize()
        hh = torch.from_numpy(h)
        if pinned in ("both", "h"):
            hh = hh.pin_memory()
        oi = torch.empty((batch, k), dtype=torch.int32)
        ol = torch.empty((batch, k), dtype=torch.float32)
        if pinned in ("both", "out"):
            oi, ol = oi.pin_memory(), ol.pin_memory()
        gi, gv = head.topk_host(hh, k, out_idx=oi, out_logits=ol)  # ready on return
        np.testing.assert_array_equal(gi.numpy(), ref_i.cpu().numpy())
        np.testing.assert_array_equal(gv.numpy().view(np.uint32), ref_v.cpu().numpy().view(np.uint32))
        sp = torch.empty((batch, V), dtype=torch.float32, device="cuda")
        gi, gv = head.topk_host(hh, k, out_sparse=sp)
        np.testing.assert_array_equal(gi.numpy(), ref_i2.cpu().numpy())
        torch.cuda.synchronize()
        np.testing.assert_array_equal(sp.cpu().numpy().view(np.uint32), ref_sp.cpu().numpy().view(np.uint32))
        assert head.device_status() == vie.VIE_OK
    if storage == "e4m3":
        q8, sc = oracle.quantize_e4m3(W)
        z = oracle.logits_e4m3(q8, sc, h)
    else:
        z = oracle.logits(W, h)
    for q in range(batch):
        assert not check_topk(gi.numpy()[q], gv.numpy()[q], z[q], k)


def test_host_entry_grows_its_staging(vie):
    import torch
    V, d = 20011, 256
    W, h = workload(V, d, 24, seed=5)
    with vie.Head(to_device_bits(W)) as head:
        for batch, k in ((1, 5), (24, 64), (2, 1000), (1, 5)):
            gi, gv = head.topk_host(torch.from_numpy(h[:batch]), k)
            ri, rv = head.topk(torch.from_numpy(h[:batch]).cuda(), k)
            torch.cuda.synchronize()
            np.testing.assert_array_equal(gi.numpy(), ri.cpu().numpy())
            np.testing.assert_array_equal(gv.numpy().view(np.uint32), rv.cpu().numpy().view(np.uint32))
        assert head.device_status() == vie.VIE_OK
