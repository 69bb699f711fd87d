"""GPU parity of top-k sampling (vie_sample_topk, vie_head_topk_sample)
against the oracle's fp64 definition: each draw must be one the oracle's
distribution allows at the same uniform (tests/acceptance.check_draw), the
generator must give the same uniforms, and many draws must follow the
distribution."""
import numpy as np
import pytest

import oracle
from acceptance import check_draw, check_topk
from gpu_cases import to_device_bits, workload
from paper_2608_27460_gb300 import synth

pytestmark = pytest.mark.gpu


def _draw(vie, idx, z, T, top_p, min_p, seed, step):
    import torch
    ti = torch.from_numpy(idx).cuda()
    tz = torch.from_numpy(z).cuda()
    tok, prob = vie.sample_topk(ti, tz, T, top_p, min_p, seed, step)
    torch.cuda.synchronize()
    return tok.cpu().numpy(), prob.cpu().numpy()


@pytest.mark.parametrize("k,T,top_p,min_p,spread", [
    (50, 1.0, 1.0, 0.0, 1.0),
    (50, 0.7, 0.9, 0.05, 1.0),     # the paper's k with both processors
    (1, 1.0, 1.0, 0.0, 1.0),
    (64, 1.3, 0.5, 0.0, 0.5),
    (65, 1.0, 1.0, 0.1, 0.5),      # first k of the 8-per-lane kernel
    (256, 0.5, 0.95, 0.0, 0.3),
    (257, 1.0, 1.0, 0.0, 0.3),     # first k of the 32-per-lane kernel
    (1024, 1.0, 0.99, 0.01, 0.2),  # largest k
    (50, 1e-3, 1.0, 0.0, 1.0),     # near-greedy
    (50, 50.0, 1.0, 0.0, 1.0),     # near-uniform
    (50, 1.0, 1e-6, 0.0, 1.0),     # top-p keeps one
    (50, 1.0, 1.0, 1.0, 1.0),      # min-p keeps the best only
])
def test_draws_match_the_oracle(vie, k, T, top_p, min_p, spread):
    batch, seed = 37, 1234  # 37 queries: a ragged last block of warps
    idx, z = synth.make_candidates(batch, k, 200000, seed=k * 31 + 7, spread=spread)
    pos = {(q, int(t)): j for q in range(batch) for j, t in enumerate(idx[q])}
    for step in range(4):
        tok, prob = _draw(vie, idx, z, T, top_p, min_p, seed, step)
        for q in range(batch):
            j = pos[(q, int(tok[q]))]
            u = oracle.uniform(seed, step, q)
            e = check_draw(z[q], T, top_p, min_p, u, j, float(prob[q]))
            assert not e, (q, step, e)


def test_tied_logits(vie):
    idx, z = synth.make_candidates(64, 50, 50000, seed=5, spread=0.5, ties=0.3)
    pos = {(q, int(t)): j for q in range(64) for j, t in enumerate(idx[q])}
    tok, prob = _draw(vie, idx, z, 0.9, 0.8, 0.02, 77, 3)
    for q in range(64):
        e = check_draw(z[q], 0.9, 0.8, 0.02, oracle.uniform(77, 3, q), pos[(q, int(tok[q]))], float(prob[q]))
        assert not e, (q, e)


@pytest.mark.parametrize("seed,step", [(0, 0), (1, 2), (2**32 + 5, 7), (123, 2**32 + 9),
                                       (2**64 - 1, 2**64 - 1)])
def test_generator_matches_the_oracle(vie, seed, step):
    """Equal logits and k = 1024: every cumulative sum is exact in fp32, so
    the draw is floor(u * 1024) and exposes 10 bits of each uniform."""
    batch, k = 200, 1024
    idx = np.tile(np.arange(k, dtype=np.int32), (batch, 1))
    z = np.zeros((batch, k), np.float32)
    tok, prob = _draw(vie, idx, z, 1.0, 1.0, 0.0, seed, step)
    want = np.array([int(oracle.uniform(seed, step, q) * k) for q in range(batch)])
    np.testing.assert_array_equal(tok, want)
    assert np.all(prob == np.float32(1.0 / k))


def test_frequencies_follow_the_distribution(vie):
    import torch
    k, T, top_p, min_p = 8, 0.8, 0.95, 0.02
    z = np.sort(np.array([2.0, 1.7, 1.6, 1.0, 0.5, 0.1, -0.8, -2.0], np.float32))[::-1].copy()
    batch = 1024
    idx = np.tile(np.arange(k, dtype=np.int32), (batch, 1))
    zz = np.tile(z, (batch, 1))
    ti, tz = torch.from_numpy(idx).cuda(), torch.from_numpy(zz).cuda()
    counts = np.zeros(k, int)
    for step in range(8):
        tok, _ = vie.sample_topk(ti, tz, T, top_p, min_p, 4242, step)
        counts += np.bincount(tok.cpu().numpy(), minlength=k)
    p = np.exp((z - z[0]) / T)
    p /= p.sum()
    n = min(next(i + 1 for i in range(k) if p[:i + 1].sum() >= top_p), int(np.sum(p >= min_p * p[0])))
    want = np.zeros(k)
    want[:n] = p[:n] / p[:n].sum()
    N = counts.sum()
    sd = np.sqrt(want * (1 - want) / N)
    assert np.all(np.abs(counts / N - want) <= 5 * sd + 1e-4), (counts / N, want)


def test_head_then_sample_in_one_call(vie):
    import torch
    V, d, b, k = 30011, 256, 6, 50
    W, h = workload(V, d, b, seed=19)
    z_or = oracle.logits(W, h)
    oi, ov = oracle.topk(W, h, k)
    with vie.Head(to_device_bits(W)) as head:
        hd = torch.from_numpy(h).cuda()
        sp = torch.empty((b, V), dtype=torch.float32, device="cuda")
        for step in range(3):
            idx, val, tok, prob = head.topk_sample(hd, k, 0.8, 0.9, 0.02, seed=5, step=step, out_sparse=sp)
            torch.cuda.synchronize()
            idx, val, tok, prob = idx.cpu().numpy(), val.cpu().numpy(), tok.cpu().numpy(), prob.cpu().numpy()
            for q in range(b):
                assert not check_topk(idx[q], val[q], z_or[q], k)
                assert tok[q] in idx[q]
                if set(idx[q]) == set(oi[q]):  # same candidates: the oracle's fp64 logits decide
                    j = list(oi[q]).index(tok[q])
                    e = check_draw(ov[q], 0.8, 0.9, 0.02, oracle.uniform(5, step, q), j, float(prob[q]))
                    assert not e, (q, step, e)
            # the sparse tensor came with it
            spc = sp.cpu().numpy()
            assert np.all(np.isfinite(spc).sum(axis=1) == k)
        assert head.device_status() == vie.VIE_OK
