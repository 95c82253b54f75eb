"""Property checks of the oracle's primitives on many random cases (CPU):
round-half-even shifts against exact rationals, the (M, n) rule's bounds and
maximality, the integer transform's linearity and involution, and the affine
quantizer's error bound."""
import math
from fractions import Fraction

import numpy as np
import pytest

from oracle import hatq_oracle as O

hyp = pytest.importorskip("hypothesis")
from hypothesis import given, settings, strategies as st  # noqa: E402


@settings(max_examples=300, deadline=None)
@given(st.integers(min_value=-(2 ** 62) + 1, max_value=2 ** 62 - 1), st.integers(min_value=0, max_value=62))
def test_rshift_rne_is_round_half_even_of_the_exact_quotient(v, n):
    assert int(O.rshift_rne(np.array([v]), n)[0]) == O.round_half_even_fraction(Fraction(v, 2 ** n))


@settings(max_examples=150, deadline=None)
@given(st.lists(st.floats(min_value=1e-6, max_value=4.0), min_size=1, max_size=6),
       st.lists(st.integers(min_value=1, max_value=2 ** 24), min_size=6, max_size=6),
       st.sampled_from([1, 16, 64, 128 * 64]))
def test_fixed_point_bounds_and_maximality(rho, bounds, gain):
    bounds = bounds[:len(rho)]
    try:
        M, n = O.fixed_point(rho, bounds, gain)
    except OverflowError:
        return
    M = [int(m) for m in M]
    assert max(M) < 2 ** 31 and max(m * a for m, a in zip(M, bounds)) * gain < 2 ** 62
    assert max(M) >= 2 ** 15
    if n < 62:                       # the next shift breaks one of the bounds
        M2 = [int(np.rint(math.ldexp(r, n + 1))) for r in rho]
        assert max(M2) >= 2 ** 31 or max(m * a for m, a in zip(M2, bounds)) * gain >= 2 ** 62


@settings(max_examples=100, deadline=None)
@given(st.sampled_from([2, 4, 8, 16, 32, 64]), st.integers(min_value=0, max_value=2 ** 31 - 1))
def test_integer_transform_is_linear_and_an_involution_up_to_hb(hb, seed):
    rng = np.random.default_rng(seed)
    x = rng.integers(-127, 128, size=(3, 2 * hb))
    y = rng.integers(-127, 128, size=(3, 2 * hb))
    a, b = int(rng.integers(-5, 6)), int(rng.integers(-5, 6))
    assert np.array_equal(O.transform_int(a * x + b * y, hb), a * O.transform_int(x, hb) + b * O.transform_int(y, hb))
    assert np.array_equal(O.transform_int(O.transform_int(x, hb), hb), hb * x)


@settings(max_examples=150, deadline=None)
@given(st.lists(st.floats(min_value=-1e3, max_value=1e3, allow_nan=False), min_size=1, max_size=40))
def test_affine_quantizer_error_bound(vals):
    x = np.array(vals)
    s, z = O.affine_params(x)
    q = O.quantize_affine(x, s, z)
    assert 0 <= q.min() and q.max() <= 255
    assert np.all(np.abs(s * (q - z) - x) <= s / 2 * (1 + 1e-9) + 1e-12)
    assert s * (int(O.quantize_affine(np.array([0.0]), s, z)[0]) - z) == 0.0
