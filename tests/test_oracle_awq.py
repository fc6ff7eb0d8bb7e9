"""Pins of the oracle's AWQ-unified quantizer (App. E, extensibility:
T_A(w) = (w s_A) / Delta_A + z_A, D_A(w~) = Delta_A (w~ - z_A) / s_A, s_A one
scale per column).

* s_A = 1 reduces T_A / D_A to RTN's maps, i.e. to quantize_fwd with
  s = s_r = 1 (bit for bit: every fp32 operation is the same);
* exact column equivariance: halving column j of W and doubling s_A[j]
  leaves x (so the codes) unchanged and halves W^ in that column (dyadic
  scalings are exact in fp32);
* backward: central finite differences (fp64) of a surrogate written from
  the forward definitions, codes and filter frozen, including ds_A summed
  over every row of its column;
* export: (C alpha* + z_B*) / s_A reproduces the quantizer output (Theorem 1
  with the column scale outside the BCQ weights).
"""

import numpy as np
import pytest

import oracle as O

F32 = np.float32
F64 = np.float64


def problem(seed, q, out=4, n_in=128, g=32):
    rng = np.random.default_rng(seed)
    W = (rng.standard_normal((out, n_in)) * 0.02).astype(F32)
    Gr = n_in // g
    sa = rng.uniform(0.5, 2.0, n_in).astype(F32)
    Wg = (W * sa).reshape(out, Gr, g)
    delta = ((Wg.max(-1) - Wg.min(-1)) / ((1 << q) - 1)).astype(F32)
    za = (-Wg.min(-1) / delta).astype(F32)
    alpha = (np.array([2.0 ** (q - 2 - j) for j in range(q)]) * rng.uniform(0.9, 1.1, (out, Gr, q))).astype(F32)
    zb = (((1 << q) - 1) / 2 + rng.normal(0, 0.1, (out, Gr))).astype(F32)
    _, codes = O.quantize_fwd_awq(W, sa, delta, za, alpha, zb, None, g, mode=O.MAP_FULL)
    Gup = (rng.standard_normal((out, n_in)) * 0.01).astype(F32)
    return dict(W=W, sa=sa, delta=delta, za=za, alpha=alpha, zb=zb, codes=codes, Gup=Gup, g=g)


@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_unit_column_scale_is_the_rtn_transform(q):
    pb = problem(10 + q, q)
    ones = np.ones_like(pb["sa"])
    for mode, step in ((O.MAP_FULL, 0), (O.MAP_LOCAL_PERIODIC, 0), (O.MAP_LOCAL_PERIODIC, 1)):
        a = O.quantize_fwd_awq(pb["W"], ones, pb["delta"], pb["za"], pb["alpha"], pb["zb"], pb["codes"], pb["g"],
                               mode, step, 2)
        b = O.quantize_fwd(pb["W"], np.ones_like(pb["W"]), np.ones(pb["W"].shape[0], F32), pb["delta"], pb["za"],
                           pb["alpha"], pb["zb"], pb["codes"], pb["g"], mode, step, 2)
        assert np.array_equal(a[0], b[0]) and np.array_equal(a[1], b[1])


def test_column_rescaling_is_exactly_equivariant():
    q = 3
    pb = problem(20, q)
    W2, s2 = pb["W"].copy(), pb["sa"].copy()
    cols = [0, 5, 77, 127]
    W2[:, cols] *= F32(0.5)
    s2[cols] *= F32(2.0)
    a_w, a_c = O.quantize_fwd_awq(pb["W"], pb["sa"], pb["delta"], pb["za"], pb["alpha"], pb["zb"], None, pb["g"],
                                  O.MAP_FULL)
    b_w, b_c = O.quantize_fwd_awq(W2, s2, pb["delta"], pb["za"], pb["alpha"], pb["zb"], None, pb["g"], O.MAP_FULL)
    assert np.array_equal(a_c, b_c)
    expect = a_w.copy()
    expect[:, cols] *= F32(0.5)
    assert np.array_equal(b_w, expect)


def surrogate(P, pb, frozen_f, x0, q):
    W, g = pb["W"].astype(F64), pb["g"]
    out, n_in = W.shape
    Wg = W.reshape(out, -1, g)
    s = P["sa"].reshape(1, -1, g)
    d, z = P["delta"][..., None], P["za"][..., None]
    x = Wg * s / d + z
    cg = pb["codes"].reshape(out, -1, g).astype(np.int64)
    c = np.where(((cg[..., None] >> np.arange(q)) & 1) == 1, 1.0, -1.0)
    m = (c * P["alpha"][..., None, :]).sum(-1) + P["zb"][..., None]
    what = d * (m - z) / s + frozen_f * d * (x - x0) / s
    return float((pb["Gup"].reshape(out, -1, g).astype(F64) * what).sum())


@pytest.mark.parametrize("q", [1, 2, 3])
def test_backward_matches_finite_differences(q):
    pb = problem(40 + q, q)
    pb["alpha"] = (pb["alpha"] * F32(0.6)).astype(F32)
    out, n_in = pb["W"].shape
    g = pb["g"]
    P = {k: pb[k].astype(F64) for k in ("sa", "delta", "za", "alpha", "zb")}
    Wg = pb["W"].reshape(out, -1, g).astype(F64)
    x0 = Wg * P["sa"].reshape(1, -1, g) / P["delta"][..., None] + P["za"][..., None]
    cg = pb["codes"].reshape(out, -1, g).astype(np.int64)
    c = np.where(((cg[..., None] >> np.arange(q)) & 1) == 1, 1.0, -1.0)
    m0 = (c * P["alpha"][..., None, :]).sum(-1) + P["zb"][..., None]
    tau = np.abs(P["alpha"]).min(-1)[..., None]
    f = (np.abs(x0 - m0) <= tau).astype(F64)
    assert np.abs(np.abs(x0 - m0) - tau).min() > 1e-4 and 0 < f.mean() < 1
    grads = O.quantize_bwd_awq(pb["W"], pb["sa"], pb["delta"], pb["za"], pb["alpha"], pb["zb"], pb["codes"],
                               pb["Gup"], g)
    name = {"sa": "dsa", "delta": "ddelta", "za": "dza", "alpha": "dalpha", "zb": "dzb"}
    rng = np.random.default_rng(11)
    for k in name:
        for _ in range(4):
            idx = tuple(rng.integers(s) for s in P[k].shape)
            h = 1e-6 * max(1.0, abs(P[k][idx]))
            Pp = {kk: vv.copy() for kk, vv in P.items()}
            Pm = {kk: vv.copy() for kk, vv in P.items()}
            Pp[k][idx] += h
            Pm[k][idx] -= h
            fd = (surrogate(Pp, pb, f, x0, q) - surrogate(Pm, pb, f, x0, q)) / (2 * h)
            got = grads[name[k]][idx]
            assert abs(got - fd) <= 1e-5 * max(abs(fd), 1e-6), (k, idx, got, fd)


@pytest.mark.parametrize("q", [2, 3, 4])
def test_export_reproduces_the_quantizer_output(q):
    pb = problem(60 + q, q)
    what, codes = O.quantize_fwd_awq(pb["W"], pb["sa"], pb["delta"], pb["za"], pb["alpha"], pb["zb"], pb["codes"],
                                     pb["g"], O.MAP_LOCAL_PERIODIC, 0, 2)
    planes, a_s, z_s, inv = O.export_bcq_awq(pb["sa"], pb["delta"], pb["za"], pb["alpha"], pb["zb"], codes, pb["g"])
    Wt = O.bcq_dequantize(planes, a_s, z_s, pb["g"]) * inv.astype(F64)[None, :]
    scale = np.repeat(np.abs(pb["delta"].astype(F64)) * (np.abs(pb["alpha"]).sum(-1) + np.abs(pb["zb"])
                                                        + np.abs(pb["za"])), pb["g"], axis=1) / pb["sa"][None, :]
    assert np.all(np.abs(Wt - what) <= 8 * np.finfo(F32).eps * scale)
