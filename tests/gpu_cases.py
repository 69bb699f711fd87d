"""Shared helpers of the GPU parity tests: run the CUDA head through the C ABI
on seeded inputs and compare with the oracle."""
import numpy as np

import oracle
from acceptance import check_topk
from paper_2608_27460_gb300 import synth


def to_device_bits(W_bits):
    import torch
    return torch.from_numpy(np.ascontiguousarray(W_bits).view(np.int16)).cuda()


def run_head(vie, W_bits, h, k, reps=1):
    """Top-k on the GPU; returns (idx int32 [b,k], val fp32 [b,k])."""
    import torch
    Wd = to_device_bits(W_bits)
    hd = torch.from_numpy(np.ascontiguousarray(h)).cuda()
    with vie.Head(Wd) as head:
        del Wd
        out = None
        for _ in range(reps):
            idx, val = head.topk(hd, k)
            torch.cuda.synchronize()
            cur = (idx.cpu().numpy(), val.cpu().numpy())
            if out is not None:
                assert np.array_equal(out[0], cur[0]) and np.array_equal(out[1].view(np.uint32), cur[1].view(np.uint32)), \
                    "repeated launches disagree"
            out = cur
        assert head.device_status() == vie.VIE_OK, vie.vie_last_error()
    return out


def assert_parity(vie, W_bits, h, k, reps=1, z=None):
    idx, val = run_head(vie, W_bits, h, k, reps=reps)
    if z is None:
        z = oracle.logits(W_bits, h)
    failures = {}
    for q in range(h.shape[0]):
        e = check_topk(idx[q], val[q], z[q], k)
        if e:
            failures[q] = e
    assert not failures, f"{len(failures)} queries fail, e.g. {next(iter(failures.items()))}"
    return idx, val, z


def workload(V, d, n, seed, dup_frac=0.0, planted=0.0):
    W, meta = synth.make_weights(V, d, seed, dup_frac=dup_frac)
    h, rows = synth.make_queries(W, n, seed + 1, planted_frac=planted, dup_src=meta["dup_src"])
    return W, h
