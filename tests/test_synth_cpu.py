"""The seeded input generator: determinism, shapes, distributions, ties."""
import numpy as np

from paper_2608_27460_gb300 import synth


def test_bf16_rounding_is_nearest_even():
    x = np.array([1.0, 1.00390625, 1.005859375, 1.0078125, -2.5, 3.0e-3], dtype=np.float32)
    b = synth.f32_to_bf16_bits(x)
    back = synth.bf16_bits_to_f32(b)
    # 1 + 2^-8 is halfway between 1 and 1 + 2^-7: ties to even (1.0)
    assert back[1] == 1.0
    assert back[2] == 1.0078125
    assert back[3] == 1.0078125
    assert back[4] == -2.5
    assert abs(back[5] - 3.0e-3) <= 3.0e-3 * 2 ** -8


def test_weights_deterministic_and_distributed():
    W1, _ = synth.make_weights(20000, 64, seed=4)
    W2, _ = synth.make_weights(20000, 64, seed=4)
    assert np.array_equal(W1, W2)
    Wf = synth.bf16_bits_to_f32(W1).astype(np.float64)
    norms = np.sqrt((Wf ** 2).sum(1)) / (0.02 * np.sqrt(64))
    # log of the row scale is N(0, 0.3^2) (chi noise adds a little spread)
    assert abs(np.median(np.log(norms))) < 0.03
    assert 0.28 < np.std(np.log(norms)) < 0.36


def test_queries_built_from_three_rows():
    W, _ = synth.make_weights(1000, 4096, seed=1)
    h, rows = synth.make_queries(W, 8, seed=2)
    assert h.dtype == np.float32 and h.shape == (8, 4096)
    for q in range(8):
        assert len(set(rows[q].tolist())) == 3
        Wr = synth.bf16_bits_to_f32(W[rows[q]]).astype(np.float64)
        # least squares recovers coefficients near N(20, 2^2)
        c, *_ = np.linalg.lstsq(Wr.T, h[q].astype(np.float64), rcond=None)
        assert np.all(np.abs(c - 20) < 10)
    # the noise is N(0, 1) per component
    resid = h[q] - c @ Wr
    assert 0.9 < np.std(resid) < 1.1


def test_tie_stress_rows_are_exact_copies():
    W, meta = synth.make_weights(4000, 16, seed=3, dup_frac=0.05)
    dst, src = meta["dup_dst"], meta["dup_src"]
    assert len(dst) == 200 and len(np.unique(dst)) == 200
    assert not set(src.tolist()) & set(dst.tolist())
    assert np.array_equal(W[dst], W[src])
    h, rows = synth.make_queries(W, 8, seed=5, planted_frac=0.25, dup_src=src)
    assert sum(int(r in set(src.tolist())) for r in rows[:2, 0]) == 2


def test_head_shapes_match_the_paper_models():
    s = synth.HEADS
    assert (s["gemma3-270m"].V, s["gemma3-270m"].d) == (262144, 640)
    assert (s["qwen3-0.6b"].V, s["qwen3-0.6b"].d) == (151936, 1024)
    assert (s["llama3.2-1b"].V, s["llama3.2-1b"].d) == (128256, 2048)
    assert (s["gemma3-1b"].V, s["gemma3-1b"].d) == (262144, 1152)
    assert (s["llama3.2-3b"].V, s["llama3.2-3b"].d) == (128256, 3072)
