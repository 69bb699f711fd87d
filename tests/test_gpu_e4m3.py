"""GPU parity of the e4m3-quantised head (vie_head_create_e4m3): the
device quantiser gives the oracle's codes and scales bit for bit, and every
top-k call on the handle matches the oracle's head on those codes
(z_i = scale_i * sum_j e4m3(q_ij) h_j) under the usual acceptance rule, on
the tensor-core path (kind::f8f6f4, queries split into four e4m3 pieces) and
on the streaming CUDA-core kernel."""
import numpy as np
import pytest

import oracle
from acceptance import check_topk
from gpu_cases import to_device_bits, workload
from paper_2608_27460_gb300 import synth

pytestmark = pytest.mark.gpu


def _head(vie, W):
    return vie.Head(to_device_bits(W), storage="e4m3")


@pytest.mark.parametrize("V,d", [(3001, 100), (2003, 640), (1009, 1024), (257, 16)])
def test_quantiser_is_bit_exact(vie, V, d):
    W, _ = workload(V, d, 1, seed=V + d)
    W[7] = 0  # an all-zero row
    oq, osc = oracle.quantize_e4m3(W)
    with _head(vie, W) as head:
        codes, scales = head.export_e4m3()
        np.testing.assert_array_equal(codes.cpu().numpy(), oq)
        np.testing.assert_array_equal(scales.cpu().numpy().view(np.uint32), osc.view(np.uint32))
        p = head.props
        assert p.d_pad == (d + 15) // 16 * 16 and p.weight_bytes == V * p.d_pad + V * 4
        # the tensor-core path takes e4m3 rows of at least 128 codes, k <= 128
        assert head.plan(16, 50).path == (1 if p.d_pad >= 128 else 0)
        assert head.plan(1, 50).path == (1 if p.d_pad >= 128 else 0)
        assert head.plan(4, 129).path == 0
        if p.d_pad >= 128:  # up to 4 queries: the CTAs build the pieces themselves, one launch
            assert head.plan(4, 50).launches == 1 and head.plan(5, 50).launches == 2


def _parity(vie, W, h, k, reps=1, batch=None):
    """Top-k of every query of h on an e4m3 handle against the oracle's e4m3
    head; `batch` queries per call (all of them in one call by default)."""
    import torch
    q, sc = oracle.quantize_e4m3(W)
    z = oracle.logits_e4m3(q, sc, h)
    n = h.shape[0]
    batch = batch or n
    with _head(vie, W) as head:
        hd = torch.from_numpy(h).cuda()
        prev = None
        for _ in range(reps):
            parts = [head.topk(hd[q0:q0 + batch], k) for q0 in range(0, n, batch)]
            torch.cuda.synchronize()
            cur = (np.concatenate([i.cpu().numpy() for i, _ in parts]),
                   np.concatenate([v.cpu().numpy() for _, v in parts]))
            if prev is not None:
                assert np.array_equal(prev[0], cur[0]) and np.array_equal(prev[1].view(np.uint32),
                                                                           cur[1].view(np.uint32))
            prev = cur
        assert head.device_status() == vie.VIE_OK
    fails = {q_: e for q_ in range(n) if (e := check_topk(prev[0][q_], prev[1][q_], z[q_], k))}
    assert not fails, next(iter(fails.items()))
    return prev, z


@pytest.mark.parametrize("V,d,batch,k", [
    (20011, 640, 1, 50),
    (20011, 640, 9, 128),    # 16-query group at the path's largest k
    (30011, 1024, 32, 50),   # full 32-query group
    (30011, 2048, 45, 7),    # two groups: 32 + 13
    (10007, 200, 2, 50),     # d_pad 208: a partial last K-block of 128 codes
    (130, 128, 1, 50),       # one and a bit tiles: most CTAs write empty lists
    (300, 512, 12, 100),     # 16-query group over three tiles
    (64, 256, 3, 64),        # k = V
    (20011, 1024, 1, 50),
    (4099, 100, 3, 50),      # padded rows
    (33333, 2048, 4, 1),
    (30011, 512, 8, 64),
    (30011, 512, 13, 50),    # two query groups
    (9973, 256, 2, 300),
    (5000, 1152, 1, 1024),
])
def test_e4m3_head_matches_the_oracle(vie, V, d, batch, k):
    W, h = workload(V, d, batch, seed=V + d + batch)
    _parity(vie, W, h, k, reps=2)


def test_duplicate_rows_tie_by_index(vie):
    W, h = workload(40009, 640, 4, seed=23, dup_frac=0.05, planted=0.5)
    (idx, val), _ = _parity(vie, W, h, 50)
    for q in range(4):
        for j in range(1, 50):
            if val[q, j] == val[q, j - 1]:
                assert idx[q, j] > idx[q, j - 1]


@pytest.mark.parametrize("name,batch,k,n", [("qwen3-0.6b", 1, 50, 2), ("gemma3-270m", 1, 50, 2),
                                            ("llama3.2-1b", 4, 50, 4)])
def test_e4m3_full_size(vie, name, batch, k, n):
    shape = synth.HEADS[name]
    W, h, _, _ = synth.make_head(shape, seed=0, n_queries=n)
    _parity(vie, W, h[:n], k, batch=batch)  # one call per decode step of `batch` queries


def test_host_entry_and_sampling_on_e4m3(vie):
    import torch
    W, h = workload(20011, 512, 3, seed=3)
    with _head(vie, W) as head:
        ri, rv = head.topk(torch.from_numpy(h).cuda(), 50)
        gi, gv = head.topk_host(torch.from_numpy(h), 50)
        torch.cuda.synchronize()
        np.testing.assert_array_equal(gi.numpy(), ri.cpu().numpy())
        idx, val, tok, prob = head.topk_sample(torch.from_numpy(h).cuda(), 50, 0.8, 0.9, 0.05, seed=1, step=2)
        torch.cuda.synchronize()
        for q in range(3):
            assert tok[q].item() in idx[q].cpu().numpy()
        assert head.device_status() == vie.VIE_OK


def _wide_range_weights(V, d, seed):
    """Rows whose magnitudes span 2^-18 .. 1: after the per-row scale they land
    on every e4m3 binade, subnormal codes and zero included."""
    rng = np.random.default_rng(seed)
    mag = np.exp2(rng.uniform(-18.0, 0.0, (V, d)))
    sign = np.where(rng.random((V, d)) < 0.5, -1.0, 1.0)
    return synth.f32_to_bf16_bits((sign * mag).astype(np.float32))


@pytest.mark.parametrize("hval", [1.0, -0.375, 2.0**40, 2.0**-30, 1.5 * 2.0**70])
def test_one_hot_queries_give_exact_products(vie, hval):
    """With h = hval * e_j every logit is one product scale_i * e4m3(q_ij) *
    hval, which the kernel must return rounded once to fp32: equal, bit for
    bit, to the oracle's fp64 value rounded to fp32, for normal and subnormal
    codes alike."""
    import torch
    V, d, k = 4096, 48, 1024
    W = _wide_range_weights(V, d, seed=17)
    q, sc = oracle.quantize_e4m3(W)
    assert ((q & 0x78) == 0).mean() > 0.05  # subnormal codes (and zeros) are common
    cols = [0, 5, 16, 31, 47]
    h = np.zeros((len(cols), d), np.float32)
    for r, j in enumerate(cols):
        h[r, j] = hval
    z = oracle.logits_e4m3(q, sc, h)
    with _head(vie, W) as head:
        idx, val = head.topk(torch.from_numpy(h).cuda(), k)
        torch.cuda.synchronize()
        assert head.device_status() == vie.VIE_OK
    idx, val = idx.cpu().numpy(), val.cpu().numpy()
    for r in range(len(cols)):
        want = z[r][idx[r]].astype(np.float32)
        np.testing.assert_array_equal(val[r].view(np.uint32), want.view(np.uint32))
        assert not check_topk(idx[r], val[r], z[r], k)


@pytest.mark.parametrize("batch", [1, 16, 32])
def test_tensor_core_error_against_the_sum_of_magnitudes(vie, batch):
    """The four-piece split keeps each h_j to within 2^-16 |h_j|, the products
    are exact and the accumulation is fp32, so a returned logit is within a
    small multiple of 2^-16 of scale_i * sum_j |e4m3(q_ij)| |h_j| from the
    oracle's value."""
    import torch
    V, d, k = 30011, 1024, 128
    W, h = workload(V, d, batch, seed=57 + batch)
    q, sc = oracle.quantize_e4m3(W)
    z = oracle.logits_e4m3(q, sc, h)
    mag = oracle.logits_e4m3(q & 0x7F, sc, np.abs(h))
    with _head(vie, W) as head:
        assert head.plan(batch, k).path == 1
        idx, val = head.topk(torch.from_numpy(h).cuda(), k)
        torch.cuda.synchronize()
        assert head.device_status() == vie.VIE_OK
    idx, val = idx.cpu().numpy(), val.cpu().numpy()
    rel = np.array([np.abs(val[b] - z[b][idx[b]]) / mag[b][idx[b]] for b in range(batch)])
    print(f"batch {batch}: largest error / sum of magnitudes = 2^{np.log2(rel.max()):.2f}")
    assert rel.max() <= 2.0**-14


def test_streaming_kernel_on_e4m3_rows(vie):
    """The same parity with every call forced onto the streaming CUDA-core
    kernel through the launch-option hook."""
    with vie.launch_options({vie.VIE_OPT_TC_MIN_BATCH_E4M3: 100000}):
        for V, d, b, k in [(20011, 640, 1, 50), (30011, 1024, 8, 64), (20011, 2048, 3, 1)]:
            W, h = workload(V, d, b, seed=V + b)
            with _head(vie, W) as head:
                assert head.plan(b, k).path == 0
            _parity(vie, W, h, k, reps=2)


@pytest.mark.parametrize("batch", [1, 3, 12])
def test_zero_and_tiny_queries(vie, batch):
    """An all-zero query (every logit 0: the first k indices) and queries of
    very small or very large magnitude next to ordinary ones."""
    W, h = workload(20011, 1024, batch, seed=71 + batch)
    h[0] = 0.0
    if batch > 1:
        h[1] *= 1e-30
    if batch > 2:
        h[2] *= 1e30
    (idx, val), _ = _parity(vie, W, h, 50)
    np.testing.assert_array_equal(idx[0], np.arange(50))
    assert not np.any(val[0])
