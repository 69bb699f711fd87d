"""The top-k calls are safe to capture in a CUDA graph (no allocation and no
synchronisation inside them): replaying a captured call gives bit for bit
what the call gives eagerly, on the streaming kernel, the tensor-core path
(bf16 and e4m3) and the sampling chain."""
import numpy as np
import pytest

from gpu_cases import to_device_bits, workload

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("storage,batch,k", [("bf16", 1, 50), ("bf16", 4, 50), ("bf16", 40, 64),
                                             ("e4m3", 1, 50), ("e4m3", 12, 50), ("bf16", 3, 300)])
def test_graph_replay_equals_eager(vie, storage, batch, k):
    import torch
    V, d = 30011, 512
    W, h = workload(V, d, batch, seed=91 + batch)
    hd = torch.from_numpy(h).cuda()
    with vie.Head(to_device_bits(W), storage=storage) as head:
        ei, ev, es = head.topk_sparse(hd, k)
        torch.cuda.synchronize()
        oi = torch.empty_like(ei)
        ov = torch.empty_like(ev)
        osp = torch.empty_like(es)
        tok = torch.empty((batch,), dtype=torch.int32, device="cuda")
        prob = torch.empty((batch,), dtype=torch.float32, device="cuda")
        cap = torch.cuda.Stream()
        cap.wait_stream(torch.cuda.current_stream())
        g = torch.cuda.CUDAGraph()
        with torch.cuda.stream(cap):
            with torch.cuda.graph(g, stream=cap):
                head.topk_sparse(hd, k, out_idx=oi, out_logits=ov, out_sparse=osp, stream=cap)
                vie.sample_topk(oi, ov, 0.8, 0.9, 0.05, seed=3, step=1, out_token=tok, out_prob=prob, stream=cap)
        torch.cuda.current_stream().wait_stream(cap)
        for _ in range(3):
            oi.zero_()
            osp.zero_()
            g.replay()
            torch.cuda.synchronize()
            np.testing.assert_array_equal(oi.cpu().numpy(), ei.cpu().numpy())
            np.testing.assert_array_equal(ov.cpu().numpy().view(np.uint32), ev.cpu().numpy().view(np.uint32))
            np.testing.assert_array_equal(osp.cpu().numpy().view(np.uint32), es.cpu().numpy().view(np.uint32))
        t2, p2 = vie.sample_topk(ei, ev, 0.8, 0.9, 0.05, seed=3, step=1)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(tok.cpu().numpy(), t2.cpu().numpy())
        assert head.device_status() == vie.VIE_OK
