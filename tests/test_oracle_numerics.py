"""Pins of the oracle's number handling: bf16 rounding, cosine, rotary embedding, Q_obs.

Each pin checks the oracle against something other than itself: torch's own
bf16 conversion, closed forms (complex rotation, orthogonal vectors), scipy's
cosine distance, or invariants that a dropped term / wrong sign / wrong index
breaks.
"""
import math

import numpy as np
import pytest
import torch
from scipy.spatial.distance import cosine as scipy_cosine_distance

from oracle import oracle as O


def _torch_bf16_bits(x32: np.ndarray) -> np.ndarray:
    t = torch.from_numpy(np.ascontiguousarray(x32, np.float32)).to(torch.bfloat16)
    return t.view(torch.int16).numpy().view(np.uint16)


# ------------------------------------------------------------------ bf16
def test_bf16_known_patterns(olib):
    assert O.f32_to_bf16(1.0, olib) == 0x3F80
    assert O.f32_to_bf16(-2.0, olib) == 0xC000
    # exactly halfway between 1.0 (0x3F80) and 1.0078125 (0x3F81): ties to even -> 0x3F80
    assert O.f32_to_bf16(1.0 + 2.0 ** -8, olib) == 0x3F80
    # halfway between 0x3F81 and 0x3F82: ties to even -> 0x3F82
    assert O.f32_to_bf16(1.0 + 3 * 2.0 ** -8, olib) == 0x3F82
    # just above halfway rounds up
    assert O.f32_to_bf16(1.0 + 2.0 ** -8 + 2.0 ** -20, olib) == 0x3F81
    assert O.f32_to_bf16(float("inf"), olib) == 0x7F80
    nan_bits = O.f32_to_bf16(float("nan"), olib)
    assert (nan_bits & 0x7F80) == 0x7F80 and (nan_bits & 0x7F) != 0


def test_bf16_matches_torch_on_random_floats(olib):
    rng = np.random.default_rng(1)
    x = np.concatenate([
        rng.standard_normal(4000).astype(np.float32) * 10.0 ** rng.integers(-30, 30, 4000),
        rng.standard_normal(4000).astype(np.float32),
    ]).astype(np.float32)
    ours = np.array([O.f32_to_bf16(v, olib) for v in x], np.uint16)
    np.testing.assert_array_equal(ours, _torch_bf16_bits(x))


def test_bf16_widening_is_exact(olib):
    bits = np.arange(0, 65536, 7, dtype=np.uint16)
    bits = bits[(bits & 0x7F80) != 0x7F80]  # finite only
    ref = torch.from_numpy(bits.view(np.int16).copy()).view(torch.bfloat16).to(torch.float64).numpy()
    np.testing.assert_array_equal(O.bf16_to_f64(bits), ref)


def test_scoring_rounding_goes_through_fp32(olib):
    # 1 + 2^-8 + 2^-30: fp32 drops the 2^-30 (below half an fp32 ulp), leaving an
    # exact bf16 tie that goes to even (1.0).  Rounding fp64 straight to bf16
    # would give 1.0078125 instead.
    x = 1.0 + 2.0 ** -8 + 2.0 ** -30
    assert O.round_scoring(x, olib) == 1.0
    rng = np.random.default_rng(2)
    for v in rng.standard_normal(500) * 7.0:
        want = float(torch.tensor(np.float32(v)).to(torch.bfloat16).to(torch.float64))
        assert O.round_scoring(float(v), olib) == want


# ------------------------------------------------------------------ cosine
def test_cosine_closed_forms(olib):
    e1 = np.array([1.0, 0.0, 0.0])
    e2 = np.array([0.0, 1.0, 0.0])
    assert O.cosine(e1, 3 * e1, olib) == pytest.approx(1.0, abs=1e-15)
    assert O.cosine(e1, -2 * e1, olib) == pytest.approx(-1.0, abs=1e-15)
    assert O.cosine(e1, e2, olib) == 0.0
    assert O.cosine(e1, e1 + e2, olib) == pytest.approx(1.0 / math.sqrt(2.0), rel=1e-15)
    assert O.cosine(e1, np.zeros(3), olib) == 0.0


def test_cosine_matches_scipy(olib):
    rng = np.random.default_rng(3)
    for _ in range(200):
        a, b = rng.standard_normal((2, 64)) * rng.uniform(0.01, 100, 2)[:, None]
        assert O.cosine(a, b, olib) == pytest.approx(1.0 - scipy_cosine_distance(a, b), abs=1e-13)


# ------------------------------------------------------------------ rotary embedding
def test_rope_is_complex_rotation_of_rotate_half_pairs(olib):
    """Pair (i, i + d/2) rotates as the complex number x_i + i x_{i+d/2}
    by angle pos * theta^(-2i/d)."""
    rng = np.random.default_rng(4)
    for d, theta, pos in ((2, 10000.0, 3), (4, 10000.0, 7), (8, 500000.0, 123), (128, 1e6, 8319)):
        x = rng.standard_normal(d)
        y = O.rope(x, pos, theta, olib)
        h = d // 2
        z = (x[:h] + 1j * x[h:]) * np.exp(1j * pos * theta ** (-2.0 * np.arange(h) / d))
        np.testing.assert_allclose(y[:h], z.real, rtol=0, atol=1e-12 * max(1.0, pos / 100))
        np.testing.assert_allclose(y[h:], z.imag, rtol=0, atol=1e-12 * max(1.0, pos / 100))


def test_rope_identity_cases(olib):
    rng = np.random.default_rng(5)
    x = rng.standard_normal(16)
    np.testing.assert_array_equal(O.rope(x, 0, 10000.0, olib), x)       # position 0
    np.testing.assert_array_equal(O.rope(x, 999, 0.0, olib), x)         # rotation disabled


def test_rope_preserves_norm_and_relative_position(olib):
    rng = np.random.default_rng(6)
    d, theta = 64, 10000.0
    q, k = rng.standard_normal((2, d))
    for a, b in ((5, 2), (100, 97), (40, 37)):
        qa, kb = O.rope(q, a, theta, olib), O.rope(k, b, theta, olib)
        assert np.linalg.norm(qa) == pytest.approx(np.linalg.norm(q), rel=1e-13)
        # <R(a) q, R(b) k> depends only on a - b (= 3 for all three pairs)
        assert qa @ kb == pytest.approx(O.rope(q, 3, theta, olib) @ k, rel=1e-11, abs=1e-11)


# ------------------------------------------------------------------ Q_obs
def test_qobs_layout_rotation_and_rounding(olib):
    rng = np.random.default_rng(7)
    G, W, nb, d, theta = 2, 3, 2, 8, 10000.0
    q_recent = _torch_bf16_bits(rng.standard_normal((G, W, d)).astype(np.float32))
    cent = rng.standard_normal((nb, d)).astype(np.float32)
    counts = np.array([3, 0], np.int64)
    recent_pos = np.array([17, 18, 19], np.int64)
    t = 25
    qobs, valid = O.build_qobs(cent, counts, q_recent, recent_pos, t, theta, olib)
    assert qobs.shape == (G * W + nb, d)
    np.testing.assert_array_equal(valid, [1] * (G * W) + [1, 0])
    for h in range(G):
        for w in range(W):
            x = O.bf16_to_f64(q_recent[h, w])
            want = [O.round_scoring(v, olib) for v in O.rope(x, recent_pos[w], theta, olib)]
            np.testing.assert_array_equal(qobs[h * W + w], want)
    for b in range(nb):
        want = [O.round_scoring(v, olib) for v in O.rope(cent[b].astype(np.float64), t, theta, olib)]
        np.testing.assert_array_equal(qobs[G * W + b], want)
    # every value is a bf16 number
    as32 = qobs.astype(np.float32)
    np.testing.assert_array_equal(O.bf16_to_f64(_torch_bf16_bits(as32)), qobs)
