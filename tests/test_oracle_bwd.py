"""Pins of the oracle's backward pass (App. C.1 straight-through estimator with
gradient filtering, differentiating Eq. 3).

The gradients are checked against central finite differences and against
torch.autograd, both applied to a surrogate loss written here from the
forward definitions only (no gradient formula is shared with the oracle):

    L(Theta) = sum_i G_i * w^_i(Theta),
    w^_i = Delta * (w~_i - z_U) + f_i * Delta * (x_i(Theta) - x_i(Theta_0)),
    w~_i = c_i . alpha + z_B,   x_i = w_i / (Delta s_i s_r) + z_U,

with the codes c_i and the filter f_i frozen at Theta_0: the mapping has
zero derivative, the straight-through estimator passes dL/dw~ to x where the
element is not filtered.
"""

import numpy as np
import pytest

import oracle as O

F32 = np.float32
F64 = np.float64


def make_problem(seed, q, out=3, n_in=96, g=32, tau_scale=1.0):
    rng = np.random.default_rng(seed)
    W = (rng.standard_normal((out, n_in)) * 0.02).astype(F32)
    Gr = n_in // g
    delta = rng.uniform(0.008, 0.012, (out, Gr)).astype(F32)
    zu = rng.uniform(3, 4, (out, Gr)).astype(F32)
    alpha = (tau_scale * np.array([2.0 ** (q - 1 - j) for j in range(q)]) *
             rng.uniform(0.8, 1.2, (out, Gr, q))).astype(F32)
    zb = (((1 << q) - 1) / 2 + rng.normal(0, 0.2, (out, Gr))).astype(F32)
    s = rng.uniform(0.9, 1.1, (out, n_in)).astype(F32)
    sr = rng.uniform(0.9, 1.1, out).astype(F32)
    _, codes = O.quantize_fwd(W, s, sr, delta, zu, alpha, zb, None, g, mode=O.MAP_FULL)
    # move the parameters so that some elements fall outside tau
    delta = (delta * F32(0.93)).astype(F32)
    Gup = (rng.standard_normal((out, n_in)) * 0.01).astype(F32)
    return dict(W=W, s=s, sr=sr, delta=delta, zu=zu, alpha=alpha, zb=zb, codes=codes, Gup=Gup, g=g)


def surrogate(P, frozen_f, x0, codes, W, Gup, g, q):
    """Surrogate loss in fp64 from the forward definitions (see module doc)."""
    out, n_in = W.shape
    Wg = W.reshape(out, -1, g).astype(F64)
    x = Wg / (P["delta"][..., None] * P["s"].reshape(out, -1, g) * P["sr"][:, None, None]) + P["zu"][..., None]
    cg = codes.reshape(out, -1, g).astype(np.int64)
    c = np.where(((cg[..., None] >> np.arange(q)) & 1) == 1, 1.0, -1.0)
    wt = (c * P["alpha"][..., None, :]).sum(-1) + P["zb"][..., None]
    what = P["delta"][..., None] * (wt - P["zu"][..., None]) + frozen_f * P["delta"][..., None] * (x - x0)
    return float((Gup.reshape(out, -1, g).astype(F64) * what).sum())


def frozen_state(pb, q):
    out, n_in = pb["W"].shape
    g = pb["g"]
    P = {k: pb[k].astype(F64) for k in ("delta", "zu", "alpha", "zb", "s", "sr")}
    Wg = pb["W"].reshape(out, -1, g).astype(F64)
    x0 = Wg / (P["delta"][..., None] * P["s"].reshape(out, -1, g) * P["sr"][:, None, None]) + P["zu"][..., None]
    cg = pb["codes"].reshape(out, -1, g).astype(np.int64)
    c = np.where(((cg[..., None] >> np.arange(q)) & 1) == 1, 1.0, -1.0)
    wt = (c * P["alpha"][..., None, :]).sum(-1) + P["zb"][..., None]
    tau = np.abs(P["alpha"]).min(-1)[..., None]
    margin = np.abs(np.abs(x0 - wt) - tau)
    f = (np.abs(x0 - wt) <= tau).astype(F64)
    return P, x0, f, margin


@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_bwd_matches_finite_differences(q):
    pb = make_problem(100 + q, q)
    P, x0, f, margin = frozen_state(pb, q)
    assert margin.min() > 1e-4          # the fp32 filter decision is unambiguous here
    assert 0 < f.mean() < 1             # both filtered and unfiltered elements occur
    grads = O.quantize_bwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                           pb["codes"], pb["Gup"], pb["g"])
    name_of = {"delta": "ddelta", "zu": "dzu", "zb": "dzb", "alpha": "dalpha", "s": "ds", "sr": "dsr"}
    rng = np.random.default_rng(7)
    for pname, gname in name_of.items():
        flat = P[pname].reshape(-1)
        idx = rng.choice(flat.size, size=min(flat.size, 12), replace=False)
        for k in idx:
            h = 1e-6 * max(1.0, abs(flat[k]))
            Pp = {kk: vv.copy() for kk, vv in P.items()}
            Pm = {kk: vv.copy() for kk, vv in P.items()}
            Pp[pname].reshape(-1)[k] += h
            Pm[pname].reshape(-1)[k] -= h
            fd = (surrogate(Pp, f, x0, pb["codes"], pb["W"], pb["Gup"], pb["g"], q) -
                  surrogate(Pm, f, x0, pb["codes"], pb["W"], pb["Gup"], pb["g"], q)) / (2 * h)
            got = grads[gname].reshape(-1)[k]
            assert abs(got - fd) <= 1e-6 * max(abs(fd), 1e-3), (pname, k, got, fd)


@pytest.mark.parametrize("q", [2, 3])
def test_bwd_matches_torch_autograd(q):
    torch = pytest.importorskip("torch")
    pb = make_problem(200 + q, q, out=4, n_in=256, g=64)
    P, x0, f, _ = frozen_state(pb, q)
    out, n_in = pb["W"].shape
    g = pb["g"]
    T = {k: torch.tensor(v, dtype=torch.float64, requires_grad=True) for k, v in P.items()}
    Wg = torch.tensor(pb["W"].reshape(out, -1, g), dtype=torch.float64)
    x = Wg / (T["delta"][..., None] * T["s"].reshape(out, -1, g) * T["sr"][:, None, None]) + T["zu"][..., None]
    xs = x.detach()                                   # stop-gradient copy of x
    cg = torch.tensor(pb["codes"].reshape(out, -1, g).astype(np.int64))
    c = torch.where(((cg[..., None] >> torch.arange(q)) & 1) == 1, 1.0, -1.0).double()
    wt = (c * T["alpha"][..., None, :]).sum(-1) + T["zb"][..., None]
    ft = torch.tensor(f)
    what = T["delta"][..., None] * (wt + ft * (x - xs) - T["zu"][..., None])
    (torch.tensor(pb["Gup"].reshape(out, -1, g), dtype=torch.float64) * what).sum().backward()
    grads = O.quantize_bwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                           pb["codes"], pb["Gup"], g)
    pairs = {"delta": "ddelta", "zu": "dzu", "zb": "dzb", "alpha": "dalpha", "s": "ds", "sr": "dsr"}
    for pname, gname in pairs.items():
        ref = T[pname].grad.numpy()
        assert np.allclose(grads[gname], ref, rtol=1e-10, atol=1e-14), pname


def test_filter_semantics():
    q = 3
    pb = make_problem(300, q)
    P, x0, f, margin = frozen_state(pb, q)
    gr = O.quantize_bwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                        pb["codes"], pb["Gup"], pb["g"])
    ds = gr["ds"].reshape(f.shape)
    clear = margin > 1e-4
    # filtered elements (|x - w~| > min|alpha|) get no straight-through gradient
    assert np.all(ds[clear & (f == 0)] == 0)
    assert np.all(ds[clear & (f == 1)] != 0)
    assert 0 < (f == 0).mean() < 1
    # tiny tau: almost everything filtered, so dz_U -> -dz_B
    tiny = pb["alpha"].copy()
    tiny[..., -1] = F32(1e-6)
    gr = O.quantize_bwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], tiny, pb["zb"],
                        pb["codes"], pb["Gup"], pb["g"])
    assert (gr["ds"] == 0).mean() > 0.99
    assert np.allclose(gr["dzu"], -gr["dzb"], rtol=0.2)


def test_l1_mass_bounds_sums():
    pb = make_problem(400, 3)
    gr = O.quantize_bwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                        pb["codes"], pb["Gup"], pb["g"])
    ms = O.bwd_l1_mass(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                       pb["codes"], pb["Gup"], pb["g"])
    for k in ("ddelta", "dzu", "dzb", "dalpha", "dsr"):
        assert np.all(np.abs(gr[k]) <= ms[k] * (1 + 1e-12) + 1e-300), k


@pytest.mark.parametrize("q", [1, 2, 3])
def test_element_filter_matches_finite_differences_of_the_masked_surrogate(q):
    """The whole-element filter: a filtered element contributes nothing, i.e.
    the gradient of sum over the UNfiltered elements of G w^ (filtered ones
    frozen)."""
    pb = make_problem(100 + q, q)
    P, x0, f, margin = frozen_state(pb, q)
    assert margin.min() > 1e-4 and 0 < f.mean() < 1
    grads = O.quantize_bwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                           pb["codes"], pb["Gup"], pb["g"], filter_mode=O.FILTER_ELEMENT)
    masked = dict(pb)
    masked["Gup"] = np.where(f.reshape(pb["Gup"].shape) > 0, pb["Gup"], 0).astype(F32)
    name_of = {"delta": "ddelta", "zu": "dzu", "zb": "dzb", "alpha": "dalpha", "s": "ds", "sr": "dsr"}
    rng = np.random.default_rng(17)
    for k in ("delta", "zu", "zb", "alpha", "s", "sr"):
        for _ in range(3):
            idx = tuple(rng.integers(n) for n in P[k].shape)
            h = 1e-6 * max(1.0, abs(P[k][idx]))
            Pp = {kk: vv.copy() for kk, vv in P.items()}
            Pm = {kk: vv.copy() for kk, vv in P.items()}
            Pp[k][idx] += h
            Pm[k][idx] -= h
            args = (x0, pb["codes"], pb["W"], masked["Gup"], pb["g"], q)
            fd = (surrogate(Pp, f, *args) - surrogate(Pm, f, *args)) / (2 * h)
            got = grads[name_of[k]][idx]
            assert abs(got - fd) <= 1e-5 * max(abs(fd), 1e-7), (k, idx, got, fd)
    assert np.all(grads["dzu"] == 0.0)


def test_half_export_rounds_to_nearest_even():
    """The 16-bit export equals IEEE half rounding of the fp32 export, checked
    with Python's own half-precision packing ('e', round half to even)."""
    import struct
    pb = make_problem(600, 3, out=4, n_in=256, g=64)
    planes, a32, z32, _ = O.export_bcq(pb["W"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"], pb["codes"], pb["g"])
    planes_h, a16, z16, _ = O.export_bcq_half(pb["W"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"], pb["codes"],
                                              pb["g"])
    assert np.array_equal(planes, planes_h)
    for v32, v16 in ((a32, a16), (z32, z16)):
        for a, b in zip(v32.ravel(), v16.ravel()):
            assert struct.unpack("<H", struct.pack("<e", float(a)))[0] == int(b)


@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_l1_mass_is_tight_when_every_term_has_one_sign(q):
    """The masses set the gradient tolerances, so they must not be inflated:
    with dL/dW^ >= 0, Delta > 0 and every code bit set (c_j = +1 for all j),
    every term of dz_B = sum Delta G and of dalpha_j = sum Delta G c_j has
    the same sign, and the mass equals the absolute value of the sum."""
    pb = make_problem(500 + q, q)
    codes = np.full_like(pb["codes"], (1 << q) - 1)
    Gup = np.abs(pb["Gup"]).astype(F32)
    args = (pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"], codes, Gup, pb["g"])
    gr, ms = O.quantize_bwd(*args), O.bwd_l1_mass(*args)
    assert np.allclose(ms["dzb"], np.abs(gr["dzb"]), rtol=1e-6, atol=0)
    assert np.allclose(ms["dalpha"], np.abs(gr["dalpha"]), rtol=1e-6, atol=0)


def test_variant_l1_masses_are_tight_when_every_term_has_one_sign():
    """The same for the OmniQuant and AWQ maps: with dL/dW^ >= 0 and every
    code bit set, the masses of dz_B and dalpha equal |dz_B| and |dalpha|."""
    from tests.test_oracle_awq import problem as awq_problem
    from tests.test_oracle_omni import problem as omni_problem
    q = 3
    po = omni_problem(61, q)
    codes = np.full_like(po["codes"], (1 << q) - 1)
    Gup = np.abs(po["Gup"]).astype(F32)
    args = (po["W"], po["beta"], po["gamma"], po["alpha"], po["zb"], codes, Gup, po["g"])
    gr, ms = O.quantize_bwd_omni(*args), O.bwd_l1_mass_omni(*args)
    assert np.allclose(ms["dzb"], np.abs(gr["dzb"]), rtol=1e-6, atol=0)
    assert np.allclose(ms["dalpha"], np.abs(gr["dalpha"]), rtol=1e-6, atol=0)
    pa = awq_problem(62, q)
    codes = np.full_like(pa["codes"], (1 << q) - 1)
    Gup = np.abs(pa["Gup"]).astype(F32)
    args = (pa["W"], pa["sa"], pa["delta"], pa["za"], pa["alpha"], pa["zb"], codes, Gup, pa["g"])
    gr, ms = O.quantize_bwd_awq(*args), O.bwd_l1_mass_awq(*args)
    assert np.allclose(ms["dzb"], np.abs(gr["dzb"]), rtol=1e-6, atol=0)
    assert np.allclose(ms["dalpha"], np.abs(gr["dalpha"]), rtol=1e-6, atol=0)
