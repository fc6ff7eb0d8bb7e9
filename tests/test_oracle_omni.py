"""Pins of the oracle's OmniQuant-unified quantizer (App. E, extensibility:
T_O(w) = w / Delta_O + z_O, D_O(w~) = Delta_O (w~ - z_O), with
Delta_O = (gamma w_M - beta w_m) / (2^q - 1), z_O = -round(beta w_m / Delta_O)).

* closed forms: beta = gamma = 1 gives min-max clipping, T_O(w_m) within
  half a step of 0 and T_O(w_M) within half a step of 2^q - 1;
* reduction to OmniQuant's uniform quantizer: with the uniform BCQ levels
  {0, 1, ..., 2^q - 1} and the full mapping, the output is
  Delta (clamp(round(w / Delta) + z, 0, 2^q - 1) - z) (rounding half down
  at exact ties, the library's tie rule);
* backward: central finite differences (fp64) of a surrogate loss written
  from the forward definitions, with codes and filter frozen and the
  rounding of z_O passed straight through (its offset frozen);
* export: the exported BCQ reproduces the quantizer output (Theorem 1).
"""

import numpy as np
import pytest

import oracle as O

F32 = np.float32
F64 = np.float64


def problem(seed, q, out=3, n_in=128, g=32):
    rng = np.random.default_rng(seed)
    W = (rng.standard_normal((out, n_in)) * 0.02).astype(F32)
    Gr = n_in // g
    beta = rng.uniform(0.8, 1.0, (out, Gr)).astype(F32)
    gamma = rng.uniform(0.8, 1.0, (out, Gr)).astype(F32)
    alpha = (np.array([2.0 ** (q - 2 - j) for j in range(q)]) * rng.uniform(0.9, 1.1, (out, Gr, q))).astype(F32)
    zb = (((1 << q) - 1) / 2 + rng.normal(0, 0.1, (out, Gr))).astype(F32)
    _, codes = O.quantize_fwd_omni(W, beta, gamma, alpha, zb, None, g, mode=O.MAP_FULL)
    Gup = (rng.standard_normal((out, n_in)) * 0.01).astype(F32)
    return dict(W=W, beta=beta, gamma=gamma, alpha=alpha, zb=zb, codes=codes, Gup=Gup, g=g)


@pytest.mark.parametrize("q", [2, 3, 4])
def test_min_max_clipping_at_beta_gamma_one(q):
    rng = np.random.default_rng(q)
    W = (rng.standard_normal((4, 256)) * 0.02).astype(F32)
    g = 64
    ones = np.ones((4, 256 // g), F32)
    delta, zo = O.omni_params(W, ones, ones, q, g)
    Wg = W.reshape(4, -1, g).astype(F64)
    assert np.allclose(delta, (Wg.max(-1) - Wg.min(-1)) / ((1 << q) - 1), rtol=1e-6)
    assert np.array_equal(zo, np.round(zo))                       # an integer zero point
    x_min = Wg.min(-1) / delta + zo
    x_max = Wg.max(-1) / delta + zo
    assert np.all(np.abs(x_min) <= 0.5 + 1e-5)
    assert np.all(np.abs(x_max - ((1 << q) - 1)) <= 0.5 + 1e-5)


@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_uniform_levels_reduce_to_omniquants_uniform_quantizer(q):
    pb = problem(30 + q, q, out=4, n_in=256, g=64)
    L = 1 << q
    alpha = np.broadcast_to(np.array([2.0 ** (q - 2 - j) for j in range(q)], F32), pb["alpha"].shape).copy()
    zb = np.full(pb["zb"].shape, (L - 1) / 2, F32)
    what, codes = O.quantize_fwd_omni(pb["W"], pb["beta"], pb["gamma"], alpha, zb, None, pb["g"], mode=O.MAP_FULL)
    delta, zo = O.omni_params(pb["W"], pb["beta"], pb["gamma"], q, pb["g"])
    out, n_in = pb["W"].shape
    g = pb["g"]
    x = (pb["W"].reshape(out, -1, g) / delta[..., None]).astype(F32) + zo[..., None]
    x = x.astype(F64)
    tie = np.abs(x - np.floor(x) - 0.5) < 1e-12
    k = np.clip(np.where(tie, np.floor(x), np.floor(x + 0.5)), 0, L - 1)   # ties to the lower level
    ref = delta.astype(F64)[..., None] * (k - zo.astype(F64)[..., None])
    assert np.allclose(what.reshape(out, -1, g), ref, rtol=1e-6, atol=1e-9)


def surrogate(P, pb, frozen_f, frozen_off, q):
    """sum G w^ from the forward definitions, in fp64, codes and filter
    frozen; z_O = -(beta w_m / Delta) + offset, the rounding offset frozen."""
    W, g = pb["W"].astype(F64), pb["g"]
    out, n_in = W.shape
    Wg = W.reshape(out, -1, g)
    wm, wM = Wg.min(-1), Wg.max(-1)
    L1 = (1 << q) - 1
    d = (P["gamma"] * wM - P["beta"] * wm) / L1
    z = -(P["beta"] * wm / d) + frozen_off
    x = Wg / d[..., None] + z[..., None]
    cg = pb["codes"].reshape(out, -1, g).astype(np.int64)
    c = np.where(((cg[..., None] >> np.arange(q)) & 1) == 1, 1.0, -1.0)
    m = (c * P["alpha"][..., None, :]).sum(-1) + P["zb"][..., None]
    what = d[..., None] * (m - z[..., None]) + frozen_f * d[..., None] * (x - P["x0"])
    return float((pb["Gup"].reshape(out, -1, g).astype(F64) * what).sum())


@pytest.mark.parametrize("q", [1, 2, 3])
def test_backward_matches_finite_differences(q):
    pb = problem(50 + q, q)
    # move the parameters so that some elements fall outside tau
    pb["alpha"] = (pb["alpha"] * F32(0.6)).astype(F32)
    out, n_in = pb["W"].shape
    g = pb["g"]
    P = {k: pb[k].astype(F64) for k in ("beta", "gamma", "alpha", "zb")}
    Wg = pb["W"].reshape(out, -1, g).astype(F64)
    wm, wM = Wg.min(-1), Wg.max(-1)
    L1 = (1 << q) - 1
    d0 = (P["gamma"] * wM - P["beta"] * wm) / L1
    raw = P["beta"] * wm / d0
    off = raw - np.rint(raw)                       # z_O = -raw + off = -round(raw)
    x0 = Wg / d0[..., None] + (-raw + off)[..., None]
    cg = pb["codes"].reshape(out, -1, g).astype(np.int64)
    c = np.where(((cg[..., None] >> np.arange(q)) & 1) == 1, 1.0, -1.0)
    m0 = (c * P["alpha"][..., None, :]).sum(-1) + P["zb"][..., None]
    tau = np.abs(P["alpha"]).min(-1)[..., None]
    f = (np.abs(x0 - m0) <= tau).astype(F64)
    margin = np.abs(np.abs(x0 - m0) - tau)
    assert margin.min() > 1e-4 and 0 < f.mean() < 1
    P["x0"] = x0
    grads = O.quantize_bwd_omni(pb["W"], pb["beta"], pb["gamma"], pb["alpha"], pb["zb"], pb["codes"], pb["Gup"], g)
    name = {"beta": "dbeta", "gamma": "dgamma", "alpha": "dalpha", "zb": "dzb"}
    rng = np.random.default_rng(9)
    for k in ("beta", "gamma", "alpha", "zb"):
        for _ in range(4):
            idx = tuple(rng.integers(s) for s in P[k].shape)
            h = 1e-6 * max(1.0, abs(P[k][idx]))
            Pp = {kk: vv.copy() for kk, vv in P.items()}
            Pm = {kk: vv.copy() for kk, vv in P.items()}
            Pp[k][idx] += h
            Pm[k][idx] -= h
            fd = (surrogate(Pp, pb, f, off, q) - surrogate(Pm, pb, f, off, q)) / (2 * h)
            got = grads[name[k]][idx]
            assert abs(got - fd) <= 1e-5 * max(abs(fd), 1e-6), (k, idx, got, fd)


@pytest.mark.parametrize("q", [2, 3, 4])
def test_export_reproduces_the_quantizer_output(q):
    pb = problem(70 + q, q)
    what, codes = O.quantize_fwd_omni(pb["W"], pb["beta"], pb["gamma"], pb["alpha"], pb["zb"], pb["codes"], pb["g"],
                                      O.MAP_LOCAL_PERIODIC, 0, 2)
    planes, a_s, z_s = O.export_bcq_omni(pb["W"], pb["beta"], pb["gamma"], pb["alpha"], pb["zb"], codes, pb["g"])
    Wt = O.bcq_dequantize(planes, a_s, z_s, pb["g"])
    delta, zo = O.omni_params(pb["W"], pb["beta"], pb["gamma"], q, pb["g"])
    scale = np.repeat(np.abs(delta.astype(F64)) * (np.abs(pb["alpha"]).sum(-1) + np.abs(pb["zb"]) + np.abs(zo)),
                      pb["g"], axis=1)
    assert np.all(np.abs(Wt - what) <= 8 * np.finfo(F32).eps * scale)


@pytest.mark.parametrize("wm,wM,expect_zo", [(-2.5, 0.5, 2.0), (-1.5, 1.5, 2.0), (-0.5, 2.5, 0.0), (-3.5, -0.5, 4.0)])
def test_zero_point_rounds_half_to_even(wm, wM, expect_zo):
    """Reading of the zero point z_O = -round(beta w_m / Delta_O): exact
    halves go to the even integer.  With q = 2 and beta = gamma = 1,
    Delta_O = (w_M - w_m) / 3 = 1 for these groups, so beta w_m / Delta_O = w_m
    exactly: -2.5 -> -2 (not -3), -1.5 -> -2, -0.5 -> -0, -3.5 -> -4."""
    g = 32
    w = np.linspace(wm, wM, g).astype(F32)
    w[0], w[-1] = wm, wM
    W = w[None, :]
    one = np.ones((1, 1), F32)
    delta, zo = O.omni_params(W, one, one, 2, g)
    assert delta[0, 0] == F32(1.0)
    assert zo[0, 0] == F32(expect_zo)
