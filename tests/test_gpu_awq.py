"""GPU parity of the AWQ-unified quantizer (uq_quantize_fwd_awq,
uq_quantize_bwd_awq; export through uq_export_bcq with (delta, zu) =
(Delta_A, z_A)) against the oracle.

Forward and export: bit-exact (fp32, the oracle's operation order).
Backward: the kernel sums in fp32 (ds_A in two stages: per row range, then
over the ranges), the oracle in fp64; |gpu - oracle| <= 1e-4 x the L1 mass
of each reduction (oracle.bwd_l1_mass_awq).
"""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_03781_gb300 import api, synth
from tests import gpu_cases as C

pytestmark = pytest.mark.gpu
F32 = np.float32
PN = ("sa", "delta", "za", "alpha", "zb")


def inputs(out, n_in, q, g, seed, wdtype="bf16"):
    rng = np.random.default_rng(seed)
    W32 = (rng.standard_t(4, (out, n_in)) * 0.02 / np.sqrt(2)).astype(F32)
    raw, W = synth.bf16_round(W32) if wdtype == "bf16" else (W32, W32)
    Gr = n_in // g
    sa = rng.uniform(0.5, 2.0, n_in).astype(F32)
    Wg = (W * sa).reshape(out, Gr, g)
    delta = ((Wg.max(-1) - Wg.min(-1)) / ((1 << q) - 1) * rng.uniform(0.9, 1.0, (out, Gr))).astype(F32)
    za = (-Wg.min(-1) / delta).astype(F32)
    alpha = (np.array([2.0 ** (q - 2 - j) for j in range(q)]) * rng.uniform(0.85, 1.15, (out, Gr, q))).astype(F32)
    zb = (((1 << q) - 1) / 2 + rng.normal(0, 0.2, (out, Gr))).astype(F32)
    P = dict(sa=sa, delta=delta, za=za, alpha=alpha, zb=zb)
    _, codes = O.quantize_fwd_awq(W, sa, delta, za, alpha, zb, None, g, O.MAP_FULL)
    P["alpha"] = (alpha * rng.uniform(0.97, 1.03, alpha.shape)).astype(F32)
    Gup = synth.upstream_grad(out, n_in, 1e-4, seed)
    return raw, W, P, codes, Gup


def dev_params(P):
    return {k: torch.from_numpy(np.ascontiguousarray(P[k])).cuda() for k in PN}


SHAPES = [(37, 512, 32), (20, 1024, 64), (33, 1536, 128), (9, 2048, 256), (5, 4096, 512), (300, 4096, 128)]


@pytest.mark.parametrize("out,n_in,g", SHAPES)
@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_awq_forward_all_modes_bit_exact(out, n_in, g, q):
    raw, W, P, codes, _ = inputs(out, n_in, q, g, seed=out + q + g)
    Wd = api.weights_tensor(raw, C.dev())
    pd = dev_params(P)
    for mode, step in ((api.MAP_FULL, 0), (api.MAP_LOCAL_PERIODIC, 0), (api.MAP_LOCAL_PERIODIC, 1)):
        cd = torch.from_numpy(codes.copy()).cuda()
        what = torch.full((out, n_in), float("nan"), device=C.dev())
        api.uq_quantize_fwd_awq(Wd, q, g, pd, cd, what, mode, step, 2)
        r_what, r_codes = O.quantize_fwd_awq(W, P["sa"], P["delta"], P["za"], P["alpha"], P["zb"], codes, g, mode,
                                             step, 2)
        C.assert_fwd_equal(C.host(what), C.host(cd), r_what, r_codes, f"awq {out}x{n_in} g{g} q{q} m{mode} s{step}")


@pytest.mark.parametrize("out,n_in,g", SHAPES)
@pytest.mark.parametrize("q", [1, 3, 4])
def test_awq_backward_within_l1_mass_tolerance(out, n_in, g, q):
    raw, W, P, codes, Gup = inputs(out, n_in, q, g, seed=200 + out + q)
    Wd = api.weights_tensor(raw, C.dev())
    pd = dev_params(P)
    Gr = n_in // g
    nan = lambda *s: torch.full(s, float("nan"), device=C.dev())
    gr = {"dsa": nan(n_in), "ddelta": nan(out, Gr), "dza": nan(out, Gr), "dalpha": nan(out, Gr, q),
          "dzb": nan(out, Gr)}
    ws = torch.full((api.uq_awq_bwd_workspace_bytes(out, n_in, q, g) // 4,), float("nan"), device=C.dev())
    api.uq_quantize_bwd_awq(Wd, q, g, pd, torch.from_numpy(codes).cuda(), torch.from_numpy(Gup).cuda(), gr,
                            workspace=ws)
    args = (W, P["sa"], P["delta"], P["za"], P["alpha"], P["zb"], codes, Gup, g)
    ref, mass = O.quantize_bwd_awq(*args), O.bwd_l1_mass_awq(*args)
    for k in ("dsa", "ddelta", "dza", "dalpha", "dzb"):
        got = C.host(gr[k]).astype(np.float64)
        err = np.abs(got - ref[k])
        bad = err > 1e-4 * mass[k] + 1e-30
        assert not bad.any(), f"{k}: {int(bad.sum())} outside; worst {(err / (mass[k] + 1e-30)).max():.3g}"


@pytest.mark.parametrize("q,g", [(1, 32), (2, 64), (3, 128), (4, 128), (3, 512)])
def test_awq_backward_filter_boundary_within_ulps(q, g):
    """Weights placed within 4 ulps of the filter boundary |x - w~| = tau
    (x = (w s_A) / Delta_A + z_A): the decisions must be those of the IEEE
    quotient however the kernel forms x."""
    out, n_in = 24, 1024
    raw, W, P, codes, Gup = inputs(out, n_in, q, g, seed=650 + q + g, wdtype="f32")
    Gr = n_in // g
    m = O.reconstruct(codes.reshape(out, Gr, g).astype(np.int64), O.levels(P["alpha"], P["zb"])).astype(np.float64)
    tau = np.abs(P["alpha"].astype(np.float64)).min(-1)[..., None]
    rng = np.random.default_rng(q + g)
    xt = m + rng.choice([-1.0, 1.0], m.shape) * tau * (1.0 + rng.integers(-4, 5, m.shape) * 2.0 ** -23)
    wn = ((xt - P["za"].astype(np.float64)[..., None]) * P["delta"].astype(np.float64)[..., None]
          / P["sa"].astype(np.float64).reshape(1, Gr, g))
    W2 = wn.astype(F32).reshape(out, n_in)
    Wd = api.weights_tensor(W2, C.dev())
    nan = lambda *s: torch.full(s, float("nan"), device=C.dev())
    gr = {"dsa": nan(n_in), "ddelta": nan(out, Gr), "dza": nan(out, Gr), "dalpha": nan(out, Gr, q),
          "dzb": nan(out, Gr)}
    api.uq_quantize_bwd_awq(Wd, q, g, dev_params(P), torch.from_numpy(codes).cuda(), torch.from_numpy(Gup).cuda(), gr)
    args = (W2, P["sa"], P["delta"], P["za"], P["alpha"], P["zb"], codes, Gup, g)
    ref, mass = O.quantize_bwd_awq(*args), O.bwd_l1_mass_awq(*args)
    for k in ("dsa", "ddelta", "dza", "dalpha", "dzb"):
        err = np.abs(C.host(gr[k]).astype(np.float64) - ref[k])
        bad = err > 1e-4 * mass[k] + 1e-30
        assert not bad.any(), f"{k}: {int(bad.sum())} outside; worst {(err / (mass[k] + 1e-30)).max():.3g}"


@pytest.mark.parametrize("g", [32, 128, 512])
def test_awq_export_through_uq_export_bcq_bit_exact(g):
    q = 3
    raw, W, P, codes, _ = inputs(24, 2048, q, g, seed=g)
    pd = dev_params(P)
    Gr = 2048 // g
    planes = torch.empty(q, 24, 64, dtype=torch.int32, device=C.dev())
    a_s = torch.empty(24, Gr, q, device=C.dev())
    z_s = torch.empty(24, Gr, device=C.dev())
    params = {"delta": pd["delta"], "zu": pd["za"], "alpha": pd["alpha"], "zb": pd["zb"]}
    api.uq_export_bcq(None, q, g, params, torch.from_numpy(codes).cuda(), planes, a_s, z_s, shape=(24, 2048))
    r_planes, r_as, r_zs, _ = O.export_bcq_awq(P["sa"], P["delta"], P["za"], P["alpha"], P["zb"], codes, g)
    assert np.array_equal(C.host(planes).view(np.uint32), r_planes)
    assert np.array_equal(C.host(a_s), r_as) and np.array_equal(C.host(z_s), r_zs)


def test_awq_backward_rejects_a_small_workspace():
    raw, W, P, codes, Gup = inputs(16, 1024, 2, 64, seed=3)
    Wd = api.weights_tensor(raw, C.dev())
    gr = {"dsa": torch.empty(1024, device=C.dev()), "ddelta": torch.empty(16, 16, device=C.dev()),
          "dza": torch.empty(16, 16, device=C.dev()), "dalpha": torch.empty(16, 16, 2, device=C.dev()),
          "dzb": torch.empty(16, 16, device=C.dev())}
    with pytest.raises(api.UQError) as e:
        api.uq_quantize_bwd_awq(Wd, 2, 64, dev_params(P), torch.from_numpy(codes).cuda(), torch.from_numpy(Gup).cuda(),
                                gr, workspace=torch.empty(4, device=C.dev()))
    assert e.value.status == api.UQ_ERR_ARG


@pytest.mark.parametrize("q,g,n_in", [(1, 32, 1024), (2, 64, 1024), (3, 128, 2048), (4, 128, 1024)])
def test_awq_remap_near_level_midpoints_is_bit_exact(q, g, n_in):
    """Weights aimed within 4 ulps of the midpoints between each element's
    level and a rank neighbour: the remap step's codes and W^ are the
    oracle's bit for bit (the pipelined forward decides from the reciprocal
    of Delta_A only inside a proven interval)."""
    out = 24
    _, _, P, codes, _ = inputs(out, n_in, q, g, seed=600 + q + g, wdtype="f32")
    W = C.awq_midpoint_weights(P, codes, g, seed=q + g)
    Wd = api.weights_tensor(W, C.dev())
    cd = torch.from_numpy(codes.copy()).cuda()
    what = torch.full((out, n_in), float("nan"), device=C.dev())
    api.uq_quantize_fwd_awq(Wd, q, g, dev_params(P), cd, what, api.MAP_LOCAL_PERIODIC, 0, 2)
    r_what, r_codes = O.quantize_fwd_awq(W, P["sa"], P["delta"], P["za"], P["alpha"], P["zb"], codes, g,
                                         O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(C.host(what), C.host(cd), r_what, r_codes, f"awq midpoints q={q} g={g}")
    assert (r_codes != codes).mean() > 0.05
