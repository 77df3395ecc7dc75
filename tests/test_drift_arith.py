"""CPU pins of the arithmetic the drift kernels rely on (Eq. 8), in plain NumPy:

* the combine's expansion of tr(GB GA) over the block structure of the two Grams,
    sum_ij DD_B(i,j) BB_A(i,j) + BB_B(i,j) DD_A(i,j) + 2 DB_B(i,j) DB_A(j,i),
  equals the dense ||B1 A1 - B0 A0||_F^2, and sum_i DD_B(i,i) + DD_A(i,i) equals
  ||B1 - B0||^2 + ||A1 - A0||^2;
* the rank-4 packing: a Gram over rows [row 2j | row 2j + 1] (8 fragment features), folded as
  G(i, j) + G(i + 4, j + 4), is the Gram over the rows;
* Knuth's TwoSum of a and -b in bf16 arithmetic (round to nearest even) gives hi + lo == a - b
  exactly, so the hi/lo pair carries the exact difference of two bf16 factors.
"""
import numpy as np
import pytest

from oracle import drift

RNG = np.random.default_rng(23)


def _bf16(x):
    """Round float64 values to the nearest bf16 (ties to even), returned as float64."""
    f = np.asarray(x, np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


def _blocks(X, base):
    """DD, DB, BB of the feature vectors [d | base] over the rows of X (d = X)."""
    return X.T @ X, X.T @ base, base.T @ base


@pytest.mark.parametrize("r,i,o", [(4, 24, 40), (8, 64, 48), (16, 96, 80)])
def test_combine_expansion_equals_dense(r, i, o):
    A0, B0 = RNG.standard_normal((r, i)), RNG.standard_normal((o, r))
    A1 = A0 + 0.05 * RNG.standard_normal(A0.shape)
    B1 = B0 + 0.05 * RNG.standard_normal(B0.shape)
    # B side over the output rows: d = B1 - B0, base = B0; A side over the input columns: d = A1 - A0, base = A1
    DDb, DBb, BBb = _blocks(B1 - B0, B0)
    DDa, DBa, BBa = _blocks((A1 - A0).T, A1.T)
    t = np.sum(DDb * BBa) + np.sum(BBb * DDa) + 2.0 * np.sum(DBb * DBa.T)
    par = np.trace(DDb) + np.trace(DDa)
    assert t == pytest.approx(drift.dense_sq(A0, B0, A1, B1), rel=1e-11)
    assert par == pytest.approx(drift.param_sq(A0, B0, A1, B1), rel=1e-12)


def test_rank4_packed_rows_fold():
    r, o = 4, 64
    X = RNG.standard_normal((o, r))
    packed = X.reshape(o // 2, 2 * r)  # fragment row j = [row 2j | row 2j + 1]
    G = packed.T @ packed
    folded = G[:r, :r] + G[r:, r:]
    np.testing.assert_allclose(folded, X.T @ X, rtol=1e-13, atol=1e-13)


def _two_sum_bf16(a, b):
    hi = _bf16(a - b)
    bv = _bf16(hi - a)           # the part of -b that hi holds
    av = _bf16(hi - bv)          # the part of a that hi holds
    lo = _bf16(_bf16(a - av) - _bf16(b + bv))
    return hi, lo


@pytest.mark.parametrize("scale", [1e-3, 1.0, 30.0])
def test_two_sum_bf16_is_exact(scale):
    a = _bf16(RNG.standard_normal(20000) * scale)
    # b near a (small drifts) and unrelated to a (large ones)
    b = np.concatenate([_bf16(a[:10000] * (1 + 0.01 * RNG.standard_normal(10000))),
                        _bf16(RNG.standard_normal(10000) * scale)])
    hi, lo = _two_sum_bf16(a, b)
    np.testing.assert_array_equal(hi + lo, a - b)  # exact in float64 for these magnitudes
    assert np.all(hi == _bf16(a - b))
    # lo is representable: the pair is exact, not merely close
    assert np.all(_bf16(lo) == lo)


def test_bf16_rounding_pins():
    # ties to even at the 8-bit mantissa boundary, and exact bf16 values unchanged
    one = 1.0
    ulp = 2.0 ** -7
    assert _bf16(one + ulp / 2) == one                 # tie, even stays
    assert _bf16(one + 3 * ulp / 2) == one + 2 * ulp   # tie, rounds up to even
    assert _bf16(one + ulp / 2 + 2.0 ** -20) == one + ulp
    v = _bf16(RNG.standard_normal(100))
    np.testing.assert_array_equal(_bf16(v), v)
