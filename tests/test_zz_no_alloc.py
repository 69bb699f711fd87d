"""vie_head_topk_noalloc: top-k for callers that must not allocate device
memory -- serving engines that carve all device memory out of one budget
fixed at start-up, and decode loops that cannot afford the device
synchronisation an allocation may cause.

Its results must pass the oracle's acceptance rule and agree with
vie_head_topk on the same inputs, call after call, with its scratch held in
the library's fixed array.  The cases include a batch that takes two launches
(two query groups sharing the array's counters and lists) and list areas of
an odd number of keys (the heads area behind them must still start on a
16-byte boundary).  This file is collected last so that a failure here stops
a run only after every other test has run."""
import numpy as np
import pytest

import oracle
from acceptance import check_topk
from gpu_cases import to_device_bits, workload

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("V,d,batch,k", [
    (151936, 1024, 1, 50),   # Qwen3-0.6B-shaped, one launch
    (20011, 640, 3, 1),
    (70001, 512, 8, 64),
    (70001, 1024, 13, 50),   # two query groups: launches of 8 and 5 queries
    (5000, 64, 1, 1),        # 79 CTAs x k = 1: an odd number of list keys
    (5000, 64, 1, 3),        # 79 x 3 keys: odd again
    (5000, 64, 3, 3),        # 4 slots x 79 x 3: even, three queries
    (30011, 64, 3, 150),     # wide lists: 320-key candidate buffers, 4 slots
    (30011, 64, 1, 600),     # wide lists, one 1216-key buffer
])
def test_noalloc_matches_oracle_and_head_topk_twice(vie, V, d, batch, k):
    import torch
    W, h = workload(V, d, batch, seed=V + 11 * k + batch)
    z = oracle.logits(W, h)
    Wd = to_device_bits(W)
    hd = torch.from_numpy(h).cuda()
    s = torch.cuda.current_stream().cuda_stream
    with vie.Head(Wd) as head:
        ref_idx, ref_val = head.topk(hd, k)
    torch.cuda.synchronize()
    ref_idx, ref_val = ref_idx.cpu().numpy(), ref_val.cpu().numpy()
    for call in range(2):
        idx = torch.full((batch, k), -1, dtype=torch.int32, device="cuda")
        val = torch.full((batch, k), float("nan"), dtype=torch.float32, device="cuda")
        st = vie.vie_head_topk_noalloc(Wd.data_ptr(), V, d, hd.data_ptr(), batch, k,
                                       idx.data_ptr(), val.data_ptr(), s)
        assert st == vie.VIE_OK, vie.vie_last_error()
        assert vie.vie_device_status(s) == vie.VIE_OK, vie.vie_last_error()
        got_idx, got_val = idx.cpu().numpy(), val.cpu().numpy()
        for q in range(batch):
            errs = check_topk(got_idx[q], got_val[q], z[q], k)
            assert not errs, f"call {call}, query {q}: {errs}"
        # against the existing entry point: the same indices, logits within
        # the parity tolerance (the same kernel computes both, so in practice
        # they agree bit for bit)
        np.testing.assert_array_equal(got_idx, ref_idx, err_msg=f"call {call}")
        assert np.all(np.abs(got_val - ref_val) <= 2e-3 + 1e-3 * np.abs(ref_val)), f"call {call}"


def test_noalloc_rejects_what_it_cannot_serve(vie):
    import torch
    W = torch.zeros((1000, 12), dtype=torch.int16, device="cuda")  # d not a multiple of 8
    h = torch.zeros((1, 12), dtype=torch.float32, device="cuda")
    i = torch.empty((1, 4), dtype=torch.int32, device="cuda")
    v = torch.empty((1, 4), dtype=torch.float32, device="cuda")
    s = torch.cuda.current_stream().cuda_stream
    assert vie.vie_head_topk_noalloc(W.data_ptr(), 1000, 12, h.data_ptr(), 1, 4, i.data_ptr(),
                                     v.data_ptr(), s) == vie.VIE_ERR_INVALID_ARG
    # weights in host memory are refused before anything is enqueued
    Wh = torch.zeros((1000, 16), dtype=torch.int16).pin_memory()
    h16 = torch.zeros((1, 16), dtype=torch.float32, device="cuda")
    assert vie.vie_head_topk_noalloc(Wh.data_ptr(), 1000, 16, h16.data_ptr(), 1, 4, i.data_ptr(),
                                     v.data_ptr(), s) == vie.VIE_ERR_INVALID_ARG
    assert "device memory" in vie.vie_last_error()
    W2 = torch.zeros((200000, 16), dtype=torch.int16, device="cuda")
    h2 = torch.zeros((8, 16), dtype=torch.float32, device="cuda")
    i2 = torch.empty((8, 1024), dtype=torch.int32, device="cuda")
    v2 = torch.empty((8, 1024), dtype=torch.float32, device="cuda")
    st = vie.vie_head_topk_noalloc(W2.data_ptr(), 200000, 16, h2.data_ptr(), 8, 1024,
                                   i2.data_ptr(), v2.data_ptr(), s)
    assert st == vie.VIE_ERR_UNSUPPORTED and "scratch" in vie.vie_last_error()
    torch.cuda.synchronize()
