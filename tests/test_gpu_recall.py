"""GPU parity of the Recall@k pieces (Section 4.3): vie_recall_hits counts
bit for bit what the oracle counts on the same index lists, and
vie_head_topk_many gives every block of hidden states the same exact top-k
as vie_head_topk, within the acceptance rule against the oracle."""
import numpy as np
import pytest

import oracle
from acceptance import check_topk
from gpu_cases import to_device_bits, workload

pytestmark = pytest.mark.gpu


def _lists(n, k, m, seed, V=5000, share=0.5, empty=0.1, repeats=0.1, neg_exact=False):
    """Exact lists of distinct indices; candidate lists mixing some of the
    query's exact indices, other indices, repeats and empty slots."""
    rng = np.random.default_rng(seed)
    ex = np.stack([rng.choice(V, k, replace=False) for _ in range(n)]).astype(np.int32)
    if neg_exact:
        ex[rng.random((n, k)) < 0.1] = -1
    ap = rng.integers(0, V, (n, m)).astype(np.int32)
    take = rng.random((n, m)) < share
    ap[take] = ex[np.arange(n)[:, None].repeat(m, 1)[take], rng.integers(0, k, (n, m))[take]]
    rep = rng.random((n, m)) < repeats
    ap[:, 1:][rep[:, 1:]] = ap[:, :-1][rep[:, 1:]]
    ap[rng.random((n, m)) < empty] = -1
    return ex, ap


@pytest.mark.parametrize("n,k,m", [
    (1, 1, 1), (37, 2, 2), (20000, 2, 2),     # Recall@2 over 20k states, as in Section 4.3
    (257, 50, 64), (64, 33, 500),             # first k of 4 entries per lane
    (20, 129, 1000),                          # first k of 32 entries per lane
    (5, 1024, 4096), (3, 1024, 1), (9, 32, 70000)])
def test_hits_match_the_oracle(vie, n, k, m):
    import torch
    ex, ap = _lists(n, k, m, seed=n * 7 + k * 3 + m, neg_exact=(k == 33))
    got = vie.recall_hits(torch.from_numpy(ex).cuda(), torch.from_numpy(ap).cuda())
    torch.cuda.synchronize()
    np.testing.assert_array_equal(got.cpu().numpy(), oracle.recall_hits(ex, ap))


def test_hits_edge_lists(vie):
    import torch
    ex = np.arange(64, dtype=np.int32).reshape(2, 32)
    cases = [ex.copy(), ex[:, ::-1].copy(), np.full((2, 5), -1, np.int32), ex + 64,
             np.concatenate([ex, ex, ex], 1)]
    for ap in cases:
        got = vie.recall_hits(torch.from_numpy(ex).cuda(), torch.from_numpy(ap).cuda())
        torch.cuda.synchronize()
        np.testing.assert_array_equal(got.cpu().numpy(), oracle.recall_hits(ex, ap))


def test_topk_many_is_topk_per_block(vie):
    import torch
    V, d, n, k = 20011, 256, 2500, 2
    W, h = workload(V, d, n, seed=41)
    hd = torch.from_numpy(h).cuda()
    with vie.Head(to_device_bits(W)) as head:
        idx, val = head.topk_many(hd, k)
        for q0 in range(0, n, vie.VIE_BATCH_MAX):
            bi, bv = head.topk(hd[q0:q0 + vie.VIE_BATCH_MAX], k)
            torch.cuda.synchronize()
            np.testing.assert_array_equal(bi.cpu().numpy(), idx[q0:q0 + vie.VIE_BATCH_MAX].cpu().numpy())
            np.testing.assert_array_equal(bv.cpu().numpy().view(np.uint32),
                                          val[q0:q0 + vie.VIE_BATCH_MAX].cpu().numpy().view(np.uint32))
        assert head.device_status() == vie.VIE_OK
    sample = np.arange(0, n, 7)
    z = oracle.logits(W, h[sample])
    idx, val = idx.cpu().numpy(), val.cpu().numpy()
    fails = [q for r, q in enumerate(sample) if check_topk(idx[q], val[q], z[r], k)]
    assert not fails, fails[:5]


def test_recall_of_the_e4m3_head(vie):
    """The e4m3 head as the approximate head, the bf16 head as the ground
    truth: the device's Recall@2 equals the oracle's count on the same lists,
    and is close to the Recall@2 of the oracle's own two heads."""
    import torch
    V, d, n, k = 30011, 512, 3000, 2
    W, h = workload(V, d, n, seed=43)
    hd = torch.from_numpy(h).cuda()
    with vie.Head(to_device_bits(W)) as exact_head, vie.Head(to_device_bits(W), storage="e4m3") as q_head:
        ei, _ = exact_head.topk_many(hd, k)
        ai, _ = q_head.topk_many(hd, k)
        hits = vie.recall_hits(ei, ai)
        torch.cuda.synchronize()
    ei, ai, hits = ei.cpu().numpy(), ai.cpu().numpy(), hits.cpu().numpy()
    np.testing.assert_array_equal(hits, oracle.recall_hits(ei, ai))
    sample = np.arange(0, n, 10)
    q, sc = oracle.quantize_e4m3(W)
    o_exact, _ = oracle.topk(W, h[sample], k)
    o_q, _ = oracle.topk_e4m3(q, sc, h[sample], k)
    r_dev = hits[sample].sum() / (len(sample) * k)
    r_or = oracle.recall_at_k(o_exact, o_q)
    assert abs(r_dev - r_or) <= 0.02, (r_dev, r_or)
