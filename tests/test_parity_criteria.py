"""The parity criteria of tests/parity.py on CPU: they accept outputs that
differ from the oracle by fp32-level rounding and reject plausible mistakes."""
import numpy as np
import pytest

import oracle
from parity import check_normalized
from pins import rand_qkv

EPS = 1e-6


def _ref(n=300, d=16, dv=8, seed=3):
    q, k, v = rand_qkv(n, d, dv, seed, BH=2)
    num, den = oracle.hla2_serial(q, k, v, masked=True, normalized=False, return_den=True)
    return num, den


def _fp32_like(x, rng, rel):
    return x * (1 + rel * rng.standard_normal(x.shape))


def test_accepts_rounded_outputs():
    num, den = _ref()
    rng = np.random.default_rng(0)
    scale = np.abs(den).max()
    num_g = _fp32_like(num, rng, 1e-6)
    den_g = den + 1e-7 * scale * rng.standard_normal(den.shape)
    o_g = num_g / (den_g + EPS)[..., None]
    res = check_normalized(o_g, num_g, num, den, EPS, 2e-2)
    assert res["num"] < 1e-5


def test_rejects_wrong_denominator():
    num, den = _ref()
    o_g = num / (den + 1.0 + EPS)[..., None]  # denominator off by one everywhere
    with pytest.raises(AssertionError):
        check_normalized(o_g, num, num, den, EPS, 2e-2)


def test_rejects_wrong_numerator():
    num, den = _ref()
    bad = num.copy()
    bad[:, 100:] *= 1.05
    with pytest.raises(AssertionError):
        check_normalized(bad / (den + EPS)[..., None], bad, num, den, EPS, 2e-2)


def test_rejects_missing_eps():
    num, den = _ref(n=64)
    o_g = num / (den + 0.3)[..., None]  # a visible eps mistake
    with pytest.raises(AssertionError):
        check_normalized(o_g, num, num, den, EPS, 1e-4)
