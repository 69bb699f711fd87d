"""Pins of the oracle's quantised head: W_out rows stored as e4m3 codes with
one fp32 scale per row (weight quantisation, named in Section 4 as
orthogonal to the method), z_i = scale_i * sum_j e4m3(q_ij) h_j.

The e4m3 format is pinned to a library's implementation of it (torch's
float8_e4m3fn), the quantisation to the format's own error bound, the logits
to numpy's fp64 dot product and the top-k to a full sort."""
import numpy as np
import pytest

import oracle as default_oracle
from paper_2608_27460_gb300 import synth


def _torch_codes():
    import torch
    return torch.arange(256, dtype=torch.uint8).view(torch.float8_e4m3fn).float().numpy().astype(np.float64)


def pin_e4m3_decode_matches_library(lib):
    want = _torch_codes()
    got = np.array([lib.e4m3_to_double(c) for c in range(256)])
    assert np.array_equal(np.isnan(want), np.isnan(got))
    assert np.array_equal(want[~np.isnan(want)], got[~np.isnan(got)])
    assert got[0x7E] == 448.0 and got[0x01] == 2.0**-9 and got[0x08] == 2.0**-6


def pin_e4m3_encode_matches_library(lib):
    import torch
    vals = _torch_codes()[:0x7F]  # positive finite codes, increasing
    xs = [0.0, 1e-4, 2.0**-10, 3 * 2.0**-11, 448.0, 447.0, 460.0, 464.0]
    for a, b in zip(vals[:-1], vals[1:]):
        mid = np.float32((a + b) / 2)  # exact: a tie, to the even code
        xs += [mid, np.nextafter(mid, np.float32(0)), np.nextafter(mid, np.float32(1e9)), np.float32(a)]
    rng = np.random.default_rng(2)
    xs = np.array(xs + list(rng.normal(0, 40, 3000)) + list(rng.normal(0, 0.02, 3000)), np.float32)
    xs = np.concatenate([xs, -xs])
    xs = xs[np.abs(xs) <= 464.0]  # the library maps larger values to NaN; here they saturate
    want = torch.from_numpy(xs).to(torch.float8_e4m3fn).view(torch.uint8).numpy()
    got = np.array([lib.f32_to_e4m3(x) for x in xs], np.uint8)
    bad = np.flatnonzero(want != got)
    assert bad.size == 0, [(float(xs[i]), int(want[i]), int(got[i])) for i in bad[:5]]
    assert lib.f32_to_e4m3(1e6) == 0x7E and lib.f32_to_e4m3(-1e6) == 0xFE  # saturation


def pin_quantisation_error_bound(lib):
    """Every dequantised weight is within half an e4m3 step of the scaled
    weight: 2^-4 relative for normals, 2^-10 absolute (times the scale) for
    subnormals, plus one fp32 rounding of the quotient."""
    W, _ = synth.make_weights(300, 96, seed=4)
    q, s = lib.quantize_e4m3(W)
    table = np.array([lib.e4m3_to_double(c) for c in range(256)])
    w = synth.bf16_bits_to_f32(W).astype(np.float64)
    deq = table[q] * s[:, None].astype(np.float64)
    bound = np.maximum(2.0**-4 * np.abs(w), 2.0**-10 * s[:, None]) * (1 + 2.0**-20) + 1e-30
    assert np.all(np.abs(w - deq) <= bound)
    # the largest magnitude of a row lands on +-448, the scale is its fp32 quotient
    amax = np.max(np.abs(w), axis=1).astype(np.float32)
    assert np.array_equal(s, amax / np.float32(448.0))
    assert np.all(np.max(np.abs(table[q]), axis=1) == 448.0)


def pin_zero_row(lib):
    W = np.zeros((3, 16), np.uint16)
    W[1, 5] = synth.f32_to_bf16_bits(np.array([0.5], np.float32))[0]
    q, s = lib.quantize_e4m3(W)
    assert s[0] == 1.0 and s[2] == 1.0 and not q[0].any() and not q[2].any()
    assert s[1] == np.float32(0.5) / np.float32(448.0) and q[1, 5] == 0x7E


def pin_logits_match_numpy(lib):
    W, _ = synth.make_weights(500, 64, seed=6)
    q, s = lib.quantize_e4m3(W)
    h = np.random.default_rng(7).normal(0, 1, (3, 64)).astype(np.float32)
    table = _torch_codes()
    want = (table[q] @ h.astype(np.float64).T).T * s.astype(np.float64)
    got = lib.logits_e4m3(q, s, h)
    assert np.allclose(got, want, rtol=1e-12, atol=1e-12)


def pin_topk_is_a_full_sort(lib):
    W, _ = synth.make_weights(400, 32, seed=8)
    q, s = lib.quantize_e4m3(W)
    h = np.random.default_rng(9).normal(0, 1, (2, 32)).astype(np.float32)
    z = lib.logits_e4m3(q, s, h)
    for k in (1, 17, 400):
        idx, val = lib.topk_e4m3(q, s, h, k)
        for b in range(2):
            order = np.lexsort((np.arange(400), -z[b]))[:k]
            np.testing.assert_array_equal(idx[b], order)
            np.testing.assert_array_equal(val[b], z[b][order])


FP8_PINS = [(f.__name__, f) for f in (
    pin_e4m3_decode_matches_library, pin_e4m3_encode_matches_library, pin_quantisation_error_bound,
    pin_zero_row, pin_logits_match_numpy, pin_topk_is_a_full_sort)]


@pytest.mark.parametrize("name,pin", FP8_PINS, ids=[n for n, _ in FP8_PINS])
def test_fp8_pin(name, pin):
    pin(default_oracle._default())
