"""GPU parity of the OmniQuant-unified quantizer (uq_quantize_fwd_omni,
uq_quantize_bwd_omni, uq_omni_scales + uq_export_bcq) against the oracle.

Forward, scales and export: bit-exact (every decision and value in fp32 with
the oracle's operation order).  Backward: the kernel sums in fp32, the
oracle in fp64; |gpu - oracle| <= 1e-4 x the L1 mass of the reduction
(oracle.bwd_l1_mass_omni), as for the UniQuan_F backward.
"""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_03781_gb300 import api, synth
from tests import gpu_cases as C

pytestmark = pytest.mark.gpu
F32 = np.float32
PN = ("beta", "gamma", "alpha", "zb")


def inputs(out, n_in, q, g, seed, wdtype="bf16"):
    rng = np.random.default_rng(seed)
    W32 = (rng.standard_t(4, (out, n_in)) * 0.02 / np.sqrt(2)).astype(F32)
    raw, W = synth.bf16_round(W32) if wdtype == "bf16" else (W32, W32)
    Gr = n_in // g
    P = dict(beta=rng.uniform(0.8, 1.0, (out, Gr)).astype(F32), gamma=rng.uniform(0.8, 1.0, (out, Gr)).astype(F32),
             alpha=(np.array([2.0 ** (q - 2 - j) for j in range(q)]) * rng.uniform(0.85, 1.15, (out, Gr, q))).astype(F32),
             zb=(((1 << q) - 1) / 2 + rng.normal(0, 0.2, (out, Gr))).astype(F32))
    _, codes = O.quantize_fwd_omni(W, P["beta"], P["gamma"], P["alpha"], P["zb"], None, g, O.MAP_FULL)
    # move alpha a little so that remap steps move some codes
    P["alpha"] = (P["alpha"] * rng.uniform(0.97, 1.03, P["alpha"].shape)).astype(F32)
    Gup = synth.upstream_grad(out, n_in, 1e-4, seed)
    return raw, W, P, codes, Gup


def dev_params(P):
    return {k: torch.from_numpy(np.ascontiguousarray(P[k])).cuda() for k in PN}


SHAPES = [(37, 512, 32), (20, 1024, 64), (33, 1536, 128), (9, 2048, 256), (5, 4096, 512), (64, 4096, 128)]


@pytest.mark.parametrize("out,n_in,g", SHAPES)
@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_omni_forward_all_modes_bit_exact(out, n_in, g, q):
    raw, W, P, codes, _ = inputs(out, n_in, q, g, seed=out + q + g)
    Wd = api.weights_tensor(raw, C.dev())
    pd = dev_params(P)
    for mode, step in ((api.MAP_FULL, 0), (api.MAP_LOCAL_PERIODIC, 0), (api.MAP_LOCAL_PERIODIC, 1)):
        cd = torch.from_numpy(codes.copy()).cuda()
        what = torch.full((out, n_in), float("nan"), device=C.dev())
        api.uq_quantize_fwd_omni(Wd, q, g, pd, cd, what, mode, step, 2)
        r_what, r_codes = O.quantize_fwd_omni(W, P["beta"], P["gamma"], P["alpha"], P["zb"], codes, g, mode, step, 2)
        C.assert_fwd_equal(C.host(what), C.host(cd), r_what, r_codes, f"omni {out}x{n_in} g{g} q{q} m{mode} s{step}")


@pytest.mark.parametrize("wdtype", ["f32", "bf16"])
@pytest.mark.parametrize("g", [32, 128, 512])
def test_omni_scales_and_export_bit_exact(wdtype, g):
    q = 3
    raw, W, P, codes, _ = inputs(24, 2048, q, g, seed=g, wdtype=wdtype)
    Wd = api.weights_tensor(raw, C.dev())
    pd = dev_params(P)
    Gr = 2048 // g
    delta = torch.empty(24, Gr, device=C.dev())
    zo = torch.empty(24, Gr, device=C.dev())
    api.uq_omni_scales(Wd, q, g, pd["beta"], pd["gamma"], delta, zo)
    r_delta, r_zo = O.omni_params(W, P["beta"], P["gamma"], q, g)
    assert np.array_equal(C.host(delta), r_delta) and np.array_equal(C.host(zo), r_zo)
    # export = uq_export_bcq with (delta, zu) = (Delta_O, z_O)
    planes = torch.empty(q, 24, 2048 // 32, dtype=torch.int32, device=C.dev())
    a_s = torch.empty(24, Gr, q, device=C.dev())
    z_s = torch.empty(24, Gr, device=C.dev())
    params = {"delta": delta, "zu": zo, "alpha": pd["alpha"], "zb": pd["zb"]}
    api.uq_export_bcq(None, q, g, params, torch.from_numpy(codes).cuda(), planes, a_s, z_s, shape=(24, 2048))
    r_planes, r_as, r_zs = O.export_bcq_omni(W, P["beta"], P["gamma"], P["alpha"], P["zb"], codes, g)
    assert np.array_equal(C.host(planes).view(np.uint32), r_planes)
    assert np.array_equal(C.host(a_s), r_as) and np.array_equal(C.host(z_s), r_zs)


@pytest.mark.parametrize("out,n_in,g", SHAPES)
@pytest.mark.parametrize("q", [1, 3, 4])
def test_omni_backward_within_l1_mass_tolerance(out, n_in, g, q):
    raw, W, P, codes, Gup = inputs(out, n_in, q, g, seed=100 + out + q)
    Wd = api.weights_tensor(raw, C.dev())
    pd = dev_params(P)
    Gr = n_in // g
    gr = {"dbeta": torch.full((out, Gr), float("nan"), device=C.dev()),
          "dgamma": torch.full((out, Gr), float("nan"), device=C.dev()),
          "dalpha": torch.full((out, Gr, q), float("nan"), device=C.dev()),
          "dzb": torch.full((out, Gr), float("nan"), device=C.dev())}
    api.uq_quantize_bwd_omni(Wd, q, g, pd, torch.from_numpy(codes).cuda(), torch.from_numpy(Gup).cuda(), gr)
    args = (W, P["beta"], P["gamma"], P["alpha"], P["zb"], codes, Gup, g)
    ref, mass = O.quantize_bwd_omni(*args), O.bwd_l1_mass_omni(*args)
    for k in ("dbeta", "dgamma", "dalpha", "dzb"):
        got = C.host(gr[k]).astype(np.float64)
        err = np.abs(got - ref[k])
        bad = err > 1e-4 * mass[k] + 1e-30
        assert not bad.any(), f"{k}: {int(bad.sum())} outside; worst {(err / (mass[k] + 1e-30)).max():.3g}"


@pytest.mark.parametrize("q,g", [(1, 32), (2, 64), (3, 128), (4, 128), (3, 256)])
def test_omni_backward_filter_boundary_within_ulps(q, g):
    """Weights placed within 4 ulps of the filter boundary |x - w~| = tau
    (x = w / Delta_O + z_O), the group's smallest and largest weight kept so
    that Delta_O and z_O do not move: the decisions must be those of the IEEE
    quotient however the kernel forms x (a flipped decision moves dz-terms by
    a whole G, far outside the tolerance)."""
    out, n_in = 24, 1024
    raw, W, P, codes, Gup = inputs(out, n_in, q, g, seed=600 + q + g, wdtype="f32")
    Gr = n_in // g
    delta, zo = O.omni_params(W, P["beta"], P["gamma"], q, g)
    m = O.reconstruct(codes.reshape(out, Gr, g).astype(np.int64), O.levels(P["alpha"], P["zb"])).astype(np.float64)
    tau = np.abs(P["alpha"].astype(np.float64)).min(-1)[..., None]
    rng = np.random.default_rng(q + g)
    xt = m + rng.choice([-1.0, 1.0], m.shape) * tau * (1.0 + rng.integers(-4, 5, m.shape) * 2.0 ** -23)
    Wg = W.reshape(out, Gr, g).astype(np.float64)
    wn = (xt - zo.astype(np.float64)[..., None]) * delta.astype(np.float64)[..., None]
    lo, hi = Wg.min(-1, keepdims=True), Wg.max(-1, keepdims=True)
    inside = (wn > lo) & (wn < hi) & (Wg > lo) & (Wg < hi)        # the extremes themselves stay
    W2 = np.where(inside, wn, Wg).astype(F32).reshape(out, n_in)
    assert np.array_equal(O.omni_params(W2, P["beta"], P["gamma"], q, g)[0], delta) and inside.mean() > 0.5
    Wd = api.weights_tensor(W2, C.dev())
    gr = {"dbeta": torch.full((out, Gr), float("nan"), device=C.dev()),
          "dgamma": torch.full((out, Gr), float("nan"), device=C.dev()),
          "dalpha": torch.full((out, Gr, q), float("nan"), device=C.dev()),
          "dzb": torch.full((out, Gr), float("nan"), device=C.dev())}
    api.uq_quantize_bwd_omni(Wd, q, g, dev_params(P), torch.from_numpy(codes).cuda(), torch.from_numpy(Gup).cuda(), gr)
    args = (W2, P["beta"], P["gamma"], P["alpha"], P["zb"], codes, Gup, g)
    ref, mass = O.quantize_bwd_omni(*args), O.bwd_l1_mass_omni(*args)
    for k in ("dbeta", "dgamma", "dalpha", "dzb"):
        err = np.abs(C.host(gr[k]).astype(np.float64) - ref[k])
        bad = err > 1e-4 * mass[k] + 1e-30
        assert not bad.any(), f"{k}: {int(bad.sum())} outside; worst {(err / (mass[k] + 1e-30)).max():.3g}"


def test_omni_unsupported_group_size_raises():
    raw, W, P, codes, _ = inputs(4, 2048, 2, 1024, seed=1)
    Wd = api.weights_tensor(raw, C.dev())
    with pytest.raises(api.UQError) as e:
        api.uq_quantize_fwd_omni(Wd, 2, 1024, dev_params(P), torch.from_numpy(codes).cuda(),
                                 torch.empty(4, 2048, device=C.dev()))
    assert e.value.status == api.UQ_ERR_UNSUPPORTED


@pytest.mark.parametrize("q,g,n_in", [(1, 32, 1024), (2, 64, 1024), (3, 128, 2048), (4, 128, 1024)])
def test_omni_remap_near_level_midpoints_is_bit_exact(q, g, n_in):
    """Weights aimed within 4 ulps of the midpoints between each element's
    level and a rank neighbour (the group's extremes kept, so Delta_O and z_O
    do not move): the remap step's codes and W^ are the oracle's bit for bit
    (the pipelined forward decides from the reciprocal of Delta_O only inside
    a proven interval)."""
    out = 24
    _, W0, P, codes, _ = inputs(out, n_in, q, g, seed=500 + q + g, wdtype="f32")
    W, moved_share = C.omni_midpoint_weights(W0, P, codes, g, seed=q + g)
    assert moved_share > 0.5
    Wd = api.weights_tensor(W, C.dev())
    cd = torch.from_numpy(codes.copy()).cuda()
    what = torch.full((out, n_in), float("nan"), device=C.dev())
    api.uq_quantize_fwd_omni(Wd, q, g, dev_params(P), cd, what, api.MAP_LOCAL_PERIODIC, 0, 2)
    r_what, r_codes = O.quantize_fwd_omni(W, P["beta"], P["gamma"], P["alpha"], P["zb"], codes, g,
                                          O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(C.host(what), C.host(cd), r_what, r_codes, f"omni midpoints q={q} g={g}")
    assert (r_codes != codes).mean() > 0.05
