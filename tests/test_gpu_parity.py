"""GPU parity: the CUDA head (through the C ABI) against the fp64 oracle.

Small cases span several stages and CTAs with ragged tails; the full-size
cases use the five workload shapes with the launch configuration the bench
times.  Acceptance rules are in tests/acceptance.py."""
import functools

import numpy as np
import pytest

import oracle
from acceptance import check_topk
from gpu_cases import assert_parity, run_head, to_device_bits, workload
from paper_2608_27460_gb300 import synth
from test_oracle_pins import load_hand_case

pytestmark = pytest.mark.gpu


def test_hand_worked_case_exact(vie):
    W, h, z, rank = load_hand_case()
    for k in (1, 5, 9, 16):
        idx, val = run_head(vie, W, h, k)
        np.testing.assert_array_equal(idx, rank[:, :k])
        np.testing.assert_array_equal(val, np.take_along_axis(z, rank[:, :k].astype(np.int64), 1))


@pytest.mark.parametrize("V,d,batch,k", [
    (1000, 64, 1, 50),
    (4099, 100, 1, 50),      # d not a multiple of 8: padded rows
    (20011, 640, 1, 50),     # ragged CTA slices and stages
    (20011, 640, 3, 1),      # greedy, odd batch
    (33333, 1024, 2, 64),    # largest short-list k
    (33333, 1152, 4, 65),    # k = 65 on the tensor cores (batch 4)
    (9973, 256, 5, 256),
    (9973, 256, 1, 257),     # streaming wide lists, a 576-key buffer
    (70001, 512, 8, 50),     # widest query group
    (70001, 512, 13, 50),    # two query groups
    (5000, 2048, 1, 1024),   # largest k
    (777, 24, 2, 777),       # k = V
    (131, 8, 1, 7),          # fewer rows than CTAs would like
    (40000, 3072, 3, 50),
    (20000, 4104, 1, 50),    # wide rows
])
def test_parity_small(vie, V, d, batch, k):
    W, h = workload(V, d, batch, seed=V + d + batch + k)
    assert_parity(vie, W, h, k, reps=2)


def test_exact_integer_inputs_are_exact(vie):
    """Small-integer weights and queries: every fp32 partial sum is exact, so
    the GPU logits equal the exact values bit for bit."""
    rng = np.random.default_rng(5)
    V, d = 30011, 136
    Wi = rng.integers(-8, 9, size=(V, d))
    hi = rng.integers(-4, 5, size=(3, d)).astype(np.float32)
    W = synth.f32_to_bf16_bits(Wi.astype(np.float32))
    idx, val = run_head(vie, W, hi, 100)
    oi, ov = oracle.topk(W, hi, 100)
    np.testing.assert_array_equal(idx, oi)
    np.testing.assert_array_equal(val.astype(np.float64), ov)


def test_all_rows_equal_ranks_by_index(vie):
    """Every logit equal: the ranking is the index order (tie rule), which
    also drives the merge through its many-candidates path."""
    V, d = 50000, 64
    row = synth.f32_to_bf16_bits(np.full(d, 0.5, np.float32))
    W = np.tile(row, (V, 1))
    h = np.ones((2, d), np.float32)
    for k in (1, 50, 1000):
        idx, val = run_head(vie, W, h, k)
        np.testing.assert_array_equal(idx, np.tile(np.arange(k, dtype=np.int32), (2, 1)))
        assert np.all(val == np.float32(0.5 * d))


def test_tie_stress_duplicate_rows(vie):
    W, h = workload(100003, 1152, 8, seed=17, dup_frac=0.05, planted=0.5)
    idx, val, z = assert_parity(vie, W, h, 50)
    # duplicated rows give bit-identical logits, ranked by ascending index
    for q in range(h.shape[0]):
        for j in range(1, 50):
            if val[q, j] == val[q, j - 1]:
                assert idx[q, j] > idx[q, j - 1]


@pytest.mark.parametrize("half_rows", [0, 1])
def test_streaming_row_mappings(vie, half_rows):
    """Both ways the streaming kernel spreads a stage over a warp (whole-warp
    rows, or one row per half-warp), forced through the launch-option hook for
    every shape, with every batch on the streaming kernel; duplicated rows
    must still tie bit for bit."""
    opts = {vie.VIE_OPT_HALF_ROWS: half_rows, vie.VIE_OPT_TC_MIN_BATCH: 100000}
    with vie.launch_options(opts):
        for V, d, b, k, dup in [(20011, 640, 1, 50, 0.0), (20011, 640, 3, 1, 0.0),
                                (33333, 1152, 4, 50, 0.05), (4099, 100, 2, 50, 0.0),
                                (70001, 512, 8, 50, 0.05), (20011, 2048, 1, 64, 0.0)]:
            W, h = workload(V, d, b, seed=V + d + b, dup_frac=dup, planted=0.5 if dup else 0.0)
            with vie.Head(to_device_bits(W)) as head:
                assert head.plan(b, k).path == 0
            idx, val, _ = assert_parity(vie, W, h, k, reps=2)
            for q in range(b):
                for j in range(1, k):
                    if val[q, j] == val[q, j - 1]:
                        assert idx[q, j] > idx[q, j - 1]


def test_negative_zero_ranks_as_zero(vie):
    """Rows whose logit is -0.0 or +0.0 tie and are ranked by index."""
    d = 8
    W = np.zeros((64, d), np.float32)
    W[:, 0] = np.where(np.arange(64) % 2 == 0, 1.0, 0.0)
    W[5, 0] = 2.0
    Wb = synth.f32_to_bf16_bits(W)
    h = np.zeros((1, d), np.float32)
    h[0, 0] = -1.0  # even rows: -1 (row 5: -2); odd rows: -0.0
    idx, val = run_head(vie, Wb, h, 40)
    want = [i for i in range(64) if i % 2 == 1 and i != 5]
    want = want + [i for i in range(64) if i % 2 == 0]
    np.testing.assert_array_equal(idx[0], np.array(want[:40], np.int32))
    assert np.all(val[0, :31].view(np.uint32) == 0)


def test_scatter_is_bit_exact(vie):
    import torch
    W, h = workload(50021, 256, 4, seed=3)
    Wd = to_device_bits(W)
    with vie.Head(Wd) as head:
        idx, val = head.topk(torch.from_numpy(h).cuda(), 50)
        out = head.sparse_logits(idx, val)
        torch.cuda.synchronize()
        assert vie.vie_device_status() == vie.VIE_OK
        want, ok = oracle.scatter(idx.cpu().numpy(), val.cpu().numpy(), 50021)
        assert ok
        np.testing.assert_array_equal(out.cpu().numpy().view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("V,d,batch,k", [(50021, 256, 4, 50), (20011, 640, 1, 1), (4099, 100, 3, 300),
                                         (151936, 1024, 1, 50), (70001, 512, 13, 64)])
def test_fused_sparse_equals_topk_then_scatter(vie, V, d, batch, k):
    """One-launch top-k + sparse tensor: same top-k as vie_head_topk and the
    sparse rows bit-equal to the oracle's scatter of those results."""
    import torch
    W, h = workload(V, d, batch, seed=V + k)
    with vie.Head(to_device_bits(W)) as head:
        hd = torch.from_numpy(h).cuda()
        i1, v1 = head.topk(hd, k)
        base = torch.empty(batch * V + 1, dtype=torch.float32, device="cuda")
        sp_out = base[1:].view(batch, V)  # rows that start off 16-byte alignment
        sp_out.fill_(7.0)
        i2, v2, sp = head.topk_sparse(hd, k, out_sparse=sp_out)
        torch.cuda.synchronize()
        assert head.device_status() == vie.VIE_OK
        np.testing.assert_array_equal(i1.cpu().numpy(), i2.cpu().numpy())
        np.testing.assert_array_equal(v1.cpu().numpy().view(np.uint32), v2.cpu().numpy().view(np.uint32))
        want, ok = oracle.scatter(i2.cpu().numpy(), v2.cpu().numpy(), V)
        assert ok
        np.testing.assert_array_equal(sp.cpu().numpy().view(np.uint32), want.view(np.uint32))
    z = oracle.logits(W, h)
    for q in range(batch):
        assert not check_topk(i2.cpu().numpy()[q], v2.cpu().numpy()[q], z[q], k)


@pytest.mark.parametrize("V,batch,k,offset", [(1, 1, 1, 0), (7, 3, 7, 1), (262144, 2, 50, 3),
                                               (151936, 1, 1024, 1), (100000, 70, 5, 2)])
def test_scatter_shapes_and_alignment(vie, V, batch, k, offset):
    """Rows that start off 16-byte alignment, a single slot, many CTAs."""
    import torch
    rng = np.random.default_rng(V + k)
    idx = np.stack([rng.choice(V, size=k, replace=False) for _ in range(batch)]).astype(np.int32)
    val = rng.standard_normal((batch, k)).astype(np.float32)
    base = torch.empty(batch * V + offset, dtype=torch.float32, device="cuda")
    out = base[offset:]
    idx_d = torch.from_numpy(idx).cuda()  # keep both alive while the kernel runs
    val_d = torch.from_numpy(val).cuda()
    st = vie.vie_scatter_sparse_logits(idx_d.data_ptr(), val_d.data_ptr(), batch, k, V,
                                       out.data_ptr(), torch.cuda.current_stream().cuda_stream)
    assert st == vie.VIE_OK
    assert vie.vie_device_status() == vie.VIE_OK
    want, ok = oracle.scatter(idx, val, V)
    np.testing.assert_array_equal(out.view(batch, V).cpu().numpy().view(np.uint32),
                                  want.view(np.uint32))


def test_scatter_out_of_range_index_sets_device_flag(vie):
    import torch
    idx = torch.tensor([[0, 3, 12]], dtype=torch.int32, device="cuda")
    val = torch.tensor([[1.0, 2.0, 3.0]], dtype=torch.float32, device="cuda")
    out = torch.empty((1, 12), dtype=torch.float32, device="cuda")
    assert vie.vie_device_status() == vie.VIE_OK
    st = vie.vie_scatter_sparse_logits(idx.data_ptr(), val.data_ptr(), 1, 3, 12, out.data_ptr(),
                                       torch.cuda.current_stream().cuda_stream)
    assert st == vie.VIE_OK
    assert vie.vie_device_status() == vie.VIE_ERR_DEVICE
    assert "scatter index" in vie.vie_last_error()
    assert vie.vie_device_status() == vie.VIE_OK  # the flag was cleared
    o = out.cpu().numpy()[0]
    assert o[0] == 1.0 and o[3] == 2.0 and np.count_nonzero(np.isfinite(o)) == 2


def test_invalid_arguments_on_gpu(vie):
    import torch
    W = to_device_bits(synth.make_weights(100, 16, 1)[0])
    with vie.Head(W) as head:
        h = torch.zeros((1, 16), dtype=torch.float32, device="cuda")
        i = torch.empty((1, 200), dtype=torch.int32, device="cuda")
        v = torch.empty((1, 200), dtype=torch.float32, device="cuda")
        s = torch.cuda.current_stream().cuda_stream
        assert vie.vie_head_topk(head.handle, h.data_ptr(), 1, 101, i.data_ptr(), v.data_ptr(), s) \
            == vie.VIE_ERR_INVALID_ARG
        assert vie.vie_head_topk(head.handle, h.data_ptr(), 0, 1, i.data_ptr(), v.data_ptr(), s) \
            == vie.VIE_ERR_INVALID_ARG
        assert vie.vie_head_topk(head.handle, h.data_ptr(), vie.VIE_BATCH_MAX + 1, 1, i.data_ptr(),
                                 v.data_ptr(), s) == vie.VIE_ERR_INVALID_ARG
        assert vie.vie_head_topk(head.handle, h.data_ptr() + 2, 1, 1, i.data_ptr(), v.data_ptr(), s) \
            == vie.VIE_ERR_INVALID_ARG
    host = np.zeros((10, 8), np.uint16)
    st, hd = vie.vie_head_create(host.ctypes.data, 10, 8)
    assert st == vie.VIE_ERR_INVALID_ARG and hd is None
    assert torch.cuda.current_stream().query() or True
    torch.cuda.synchronize()  # no sticky CUDA error was left behind


def test_props(vie):
    W = to_device_bits(synth.make_weights(5000, 100, 1)[0])
    with vie.Head(W) as head:
        p = head.props
        assert (p.V, p.d, p.d_pad) == (5000, 100, 104)
        assert p.weight_bytes == 5000 * 104 * 2
        assert 1 <= p.ctas <= 1024


# ---------------------------------------------------------------------------
# Full-size workloads in the launch configuration the bench times: one fused
# call (top-k and the sparse tensor) per decode step of `batch` queries, so
# batch 1 runs on the streaming kernel and batches of 2 or more on the tensor
# cores.  The sampled queries are computed in full by the oracle.
FULL = [("gemma3-270m", 1, 50, 3), ("qwen3-0.6b", 1, 50, 3), ("llama3.2-1b", 1, 50, 2),
        ("llama3.2-1b", 1, 1, 2), ("llama3.2-1b", 4, 1, 4), ("llama3.2-1b", 4, 50, 4),
        ("gemma3-1b", 1, 50, 2), ("gemma3-1b", 2, 50, 2), ("gemma3-1b", 4, 50, 4),
        ("gemma3-1b", 8, 50, 8), ("gemma3-1b-ties", 1, 50, 4), ("gemma3-1b-ties", 4, 50, 4),
        ("llama3.2-3b", 16, 50, 16), ("llama3.2-3b", 64, 50, 64)]


@functools.lru_cache(maxsize=1)
def _full_head(name):
    """Weights and 64 queries of one workload (kept while the cases of that
    workload run; they are listed together)."""
    W, h, _, _ = synth.make_head(synth.HEADS[name], seed=0, n_queries=64)
    return W, h


@pytest.mark.parametrize("name,batch,k,n", FULL, ids=[f"{a}-b{b}-k{c}" for a, b, c, _ in FULL])
def test_parity_full_size(vie, name, batch, k, n):
    import torch
    W, h = _full_head(name)
    V = W.shape[0]
    z = oracle.logits(W, h[:n])
    with vie.Head(to_device_bits(W)) as head:
        want_path = 0 if batch == 1 else 1
        assert head.plan(batch, k).path == want_path
        hd = torch.from_numpy(np.ascontiguousarray(h[:n])).cuda()
        for q0 in range(0, n, batch):
            idx, val, sparse = head.topk_sparse(hd[q0:q0 + batch], k)
            torch.cuda.synchronize()
            idx, val, sparse = idx.cpu().numpy(), val.cpu().numpy(), sparse.cpu().numpy()
            for q in range(batch):
                e = check_topk(idx[q], val[q], z[q0 + q], k)
                assert not e, (q0 + q, e)
            want, ok = oracle.scatter(idx, val, V)
            assert ok and np.array_equal(want.view(np.uint32), sparse.view(np.uint32))
        assert head.device_status() == vie.VIE_OK, vie.vie_last_error()


@pytest.mark.parametrize("early", [0, 1])
def test_batch1_merge_modes(vie, early):
    """Single-query launches merged early (CTA 0 streams only its round-robin
    chunks, then takes the other CTAs' lists as they are published) or by
    the last CTA to finish: the same parity, the sparse tensor equal to the
    oracle's scatter of the returned top-k, and many back-to-back calls on
    one handle (the early merge keys each launch's publications by an epoch
    that advances every launch).  Covered: vocabularies so small that CTA 0
    streams nothing (V = 200, 2 CTAs at V = 128), k = 1 and k = 64 (the
    largest early-merged k), duplicate rows, and the full Gemma-3-1B shape."""
    import torch
    with vie.launch_options({vie.VIE_OPT_EARLY_MERGE: early}):
        for V, d, k, dup in [(151936, 1024, 50, 0.0), (20011, 640, 64, 0.05), (9000, 256, 1, 0.0),
                             (4099, 100, 50, 0.0), (200, 64, 50, 0.0), (128, 16, 64, 0.0),
                             (262144, 1152, 50, 0.05)]:
            n = 4
            W, h = workload(V, d, n, seed=V + d + k, dup_frac=dup, planted=0.5 if dup else 0.0)
            z = oracle.logits(W, h)
            hd = torch.from_numpy(h).cuda()
            with vie.Head(to_device_bits(W)) as head:
                assert head.plan(1, k).path == 0
                first = None
                for rep in range(3):
                    for q in range(n):
                        idx, val, sp = head.topk_sparse(hd[q:q + 1], k)
                        torch.cuda.synchronize()
                        idx, val, sp = idx.cpu().numpy(), val.cpu().numpy(), sp.cpu().numpy()
                        errs = check_topk(idx[0], val[0], z[q], k)
                        assert not errs, (V, d, k, early, rep, q, errs)
                        want, ok = oracle.scatter(idx, val, V)
                        assert ok and np.array_equal(want.view(np.uint32), sp.view(np.uint32))
                        if q == 0:
                            if first is None:
                                first = (idx, val)
                            else:  # a repeated call returns the same bits
                                assert np.array_equal(first[0], idx)
                                assert np.array_equal(first[1].view(np.uint32), val.view(np.uint32))
                assert head.device_status() == vie.VIE_OK, vie.vie_last_error()
