"""The rule by which the solver kernels add a CTA's fp32 partial of an Eq. 2 /
Eq. 4 sum into an fp64 accumulator (quantize_partial in the kernels' internal
header): the partial is rounded up to a multiple of 2^-32 first. Pinned here by
arithmetic, on the host: sums of such terms below 2^21 are exact, hence the
same in every order of addition (the order in which CTAs arrive), while plain
fp64 sums of the same fp32 partials are not; a nonzero partial stays nonzero.
"""
from fractions import Fraction

import numpy as np

SCALE = 2.0 ** 32


def quantize_up(v32):
    return np.ceil(v32.astype(np.float64) * SCALE) / SCALE


def _partials(rng, n):
    # magnitudes from converged errors (1e-14) to early-iteration ones (1e3)
    return (10.0 ** rng.uniform(-14, 3, n)).astype(np.float32)


def test_rounding_is_up_by_less_than_one_step_and_keeps_nonzero():
    rng = np.random.default_rng(1)
    v = np.concatenate([_partials(rng, 5000), np.array([0.0, 1e-30, 2.0 ** -33, 2.0 ** -32], np.float32)])
    q = quantize_up(v)
    d = np.array([Fraction(float(a)) - Fraction(float(b)) for a, b in zip(q, v)])
    assert (d >= 0).all() and (d < Fraction(1, 2 ** 32)).all()
    assert ((q > 0) == (v > 0)).all()
    assert q[-1] == 2.0 ** -32 and q[-2] == 2.0 ** -32 and q[-4] == 0.0
    assert np.array_equal(q * SCALE, np.round(q * SCALE))   # multiples of 2^-32


def test_quantized_sums_are_exact_in_every_order():
    rng = np.random.default_rng(2)
    checked = 0
    for _ in range(30):
        n = int(rng.integers(2, 700))
        q = quantize_up(_partials(rng, n))
        exact = sum(Fraction(float(x)) for x in q)
        if exact >= 2 ** 21:
            continue
        for _ in range(20):
            s = 0.0
            for x in q[rng.permutation(n)]:
                s += float(x)
            assert Fraction(s) == exact
        checked += 1
    assert checked >= 20


def test_unquantized_fp64_sums_depend_on_the_order():
    """Why the rule exists: without it, the order of arrival moves the last bits."""
    rng = np.random.default_rng(3)
    differs = 0
    for _ in range(20):
        v = _partials(rng, 300).astype(np.float64)
        sums = set()
        for _ in range(20):
            s = 0.0
            for x in v[rng.permutation(len(v))]:
                s += float(x)
            sums.add(s)
        differs += len(sums) > 1
    assert differs > 0
