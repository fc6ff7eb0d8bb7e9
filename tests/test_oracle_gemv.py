"""Pins of the oracle's BCQ product (bcq_dequantize, bcq_gemv): the
inference computation of the exported format.

* exact brute force: pure-Python loops over the bit layout of the planes
  (bit b of word t is column 32 t + b, c = +1 when set) with rational
  arithmetic on dyadic inputs, where fp64 is exact;
* Theorem 1 end to end: the quantizer's own output W^ (quantize_fwd, which
  never sees the bit-planes) times x equals the product computed from the
  exported planes, alpha* and z_B*, within the fp32 rounding of the export;
* a one-hot x reads back one column; the product is linear in x.
"""

from fractions import Fraction

import numpy as np
import pytest

import oracle as O
from tests.test_oracle_bwd import make_problem

F32 = np.float32
F64 = np.float64


def brute_force_product(planes, a_star, z_star, x, g):
    q, out, words = planes.shape
    n_in = words * 32
    y = []
    for b in range(x.shape[0]):
        row = []
        for r in range(out):
            acc = Fraction(0)
            for i in range(n_in):
                k = i // g
                w = Fraction(float(z_star[r, k]))
                for j in range(q):
                    bit = (int(planes[j, r, i // 32]) >> (i % 32)) & 1
                    w += Fraction(float(a_star[r, k, j])) * (1 if bit else -1)
                acc += w * Fraction(float(x[b, i]))
            row.append(acc)
        y.append(row)
    return y


@pytest.mark.parametrize("q,g", [(1, 32), (2, 64), (3, 32), (4, 64)])
def test_gemv_equals_exact_brute_force(q, g):
    rng = np.random.default_rng(10 + q)
    out, n_in, batch = 3, 128, 2
    planes = rng.integers(0, 2 ** 32, (q, out, n_in // 32), dtype=np.uint64).astype(np.uint32)
    # dyadic values with few bits: every product and sum below is exact in fp64
    a_star = (rng.integers(-64, 64, (out, n_in // g, q)) / 64.0).astype(F32)
    z_star = (rng.integers(-64, 64, (out, n_in // g)) / 32.0).astype(F32)
    x = (rng.integers(-16, 16, (batch, n_in)) / 8.0).astype(F32)
    y = O.bcq_gemv(planes, a_star, z_star, x, g)
    exact = brute_force_product(planes, a_star, z_star, x, g)
    for b in range(batch):
        for r in range(out):
            assert Fraction(float(y[b, r])) == exact[b][r]


@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_gemv_of_exported_format_reproduces_the_quantizer_output(q):
    """Theorem 1: R_B(C; Theta_B*) = D_R(R_B(C; Theta_B)) = W^.  The planes,
    alpha* and z_B* come from export_bcq; W^ from quantize_fwd."""
    pb = make_problem(900 + q, q, out=4, n_in=256, g=64)
    what, codes = O.quantize_fwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                                 pb["codes"], pb["g"], O.MAP_LOCAL_PERIODIC, 0, 2)
    planes, a_star, z_star, _ = O.export_bcq(pb["W"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"], codes, pb["g"])
    Wt = O.bcq_dequantize(planes, a_star, z_star, pb["g"])
    # fp32 rounding of alpha* = Delta alpha and z* = Delta (z_B - z_U), and of W^ itself
    bound = 8 * np.finfo(F32).eps * np.repeat(
        np.asarray(pb["delta"], F64) * (np.abs(pb["alpha"]).sum(-1) + np.abs(pb["zb"]) + np.abs(pb["zu"])),
        pb["g"], axis=1)
    assert (np.abs(Wt - what) <= bound).all()
    x = np.random.default_rng(q).standard_normal((3, 256)).astype(F32)
    y = O.bcq_gemv(planes, a_star, z_star, x, pb["g"])
    ref = x.astype(F64) @ what.astype(F64).T
    assert (np.abs(y - ref) <= np.abs(x).astype(F64) @ bound.T + 1e-300).all()


def test_one_hot_reads_columns_and_product_is_linear():
    rng = np.random.default_rng(3)
    q, g, out, n_in = 3, 32, 5, 96
    planes = rng.integers(0, 2 ** 32, (q, out, n_in // 32), dtype=np.uint64).astype(np.uint32)
    a_star = rng.standard_normal((out, n_in // g, q)).astype(F32)
    z_star = rng.standard_normal((out, n_in // g)).astype(F32)
    Wt = O.bcq_dequantize(planes, a_star, z_star, g)
    for i in (0, 31, 32, 63, 95):
        e = np.zeros((1, n_in), F32)
        e[0, i] = 1
        assert np.array_equal(O.bcq_gemv(planes, a_star, z_star, e, g)[0], Wt[:, i])
        # column i decoded by hand from the layout: bit i % 32 of word i // 32
        k = i // g
        hand = [float(z_star[r, k]) + sum(float(a_star[r, k, j]) * (1 if (planes[j, r, i // 32] >> (i % 32)) & 1
                                                                      else -1) for j in range(q))
                for r in range(out)]
        assert np.allclose(Wt[:, i], hand, rtol=0, atol=1e-12)
    x1, x2 = rng.standard_normal((2, 1, n_in))
    y12 = O.bcq_gemv(planes, a_star, z_star, 2 * x1 - 3 * x2, g)
    assert np.allclose(y12, 2 * O.bcq_gemv(planes, a_star, z_star, x1, g) - 3 * O.bcq_gemv(planes, a_star, z_star,
                                                                                          x2, g), atol=1e-12)
    # row blocking of the oracle does not change a bit
    assert np.array_equal(O.bcq_gemv(planes, a_star, z_star, x1, g, row_block=2),
                          O.bcq_gemv(planes, a_star, z_star, x1, g))
