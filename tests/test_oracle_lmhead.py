"""Pins of the LM-head oracle (oracle/lmhead.py) against exact arithmetic,
closed forms and independent implementations."""

import numpy as np
import pytest
import scipy.special
import torch

from oracle import lmhead


def test_logits_exact_on_integers():
    """Integer-valued operands: the float64 product is exact; compare with
    Python integer arithmetic."""
    rng = np.random.default_rng(0)
    H = rng.integers(-50, 50, size=(5, 24))
    W = rng.integers(-50, 50, size=(7, 24))
    got = lmhead.logits(H, W)
    for r in range(5):
        for v in range(7):
            assert got[r, v] == sum(int(H[r, k]) * int(W[v, k]) for k in range(24))


def test_bf16_rounding_special_values():
    one = 1.0
    step = 2.0 ** -7                     # bf16 spacing in [1, 2)
    assert lmhead.to_bf16(one) == one
    assert lmhead.to_bf16(one + step / 2) == one                 # tie to even (down)
    assert lmhead.to_bf16(one + 1.5 * step) == one + 2 * step    # tie to even (up)
    assert lmhead.to_bf16(one + 0.6 * step) == one + step
    assert lmhead.to_bf16(-(one + 0.6 * step)) == -(one + step)
    assert lmhead.to_bf16(0.0) == 0.0
    assert lmhead.to_bf16(3.0 * 2.0 ** -130) > 0                 # subnormal range of float32


def test_bf16_rounding_matches_torch_on_float32_values():
    """Values exactly representable in float32: torch's float32 -> bfloat16
    conversion (round to nearest even) is an independent implementation."""
    rng = np.random.default_rng(1)
    x = (rng.standard_normal(20000) * np.exp2(rng.integers(-20, 20, 20000))).astype(np.float32)
    ref = torch.from_numpy(x).to(torch.bfloat16).to(torch.float64).numpy()
    assert np.array_equal(lmhead.to_bf16(x.astype(np.float64)), ref)


def test_boundary_distance():
    step = 2.0 ** -7
    assert lmhead.bf16_boundary_distance(1.0 + step / 2) == 0.0
    assert lmhead.bf16_boundary_distance(1.0) == step / 2
    assert abs(lmhead.bf16_boundary_distance(1.0 + 0.25 * step) - 0.25 * step) < 1e-18
    # rounding a value moved by less than its distance never changes the result
    rng = np.random.default_rng(2)
    x = rng.standard_normal(5000) * 8
    d = lmhead.bf16_boundary_distance(x)
    for t in (0.49, -0.49):
        assert np.array_equal(lmhead.to_bf16(x + t * d), lmhead.to_bf16(x))


@pytest.mark.parametrize("T", [0.5, 1.0, 2.0])
def test_row_stats_closed_forms(T):
    V = 1000
    m, s = lmhead.row_stats(np.zeros((2, V)), T)
    assert np.all(m == 0) and np.allclose(s, V, rtol=0, atol=1e-9)
    c = 3.25
    row = np.zeros(V)
    row[17] = c
    m, s = lmhead.row_stats(row[None], T)
    assert m[0] == c
    assert s[0] == pytest.approx(1.0 + (V - 1) * np.exp(-c / T), rel=1e-13)


def test_row_stats_give_the_softmax():
    rng = np.random.default_rng(3)
    l = rng.standard_normal((4, 3000)) * 3
    T = 0.7
    m, s = lmhead.row_stats(l, T)
    mb = np.exp2((l - m[:, None]) * lmhead.LOG2E / T) / s[:, None]
    assert np.allclose(mb, scipy.special.softmax(l / T, axis=1), rtol=1e-12, atol=0)
