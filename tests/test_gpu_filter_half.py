"""GPU parity of the whole-element gradient filter (uq_quantize_bwd_ex with
UQ_FILTER_ELEMENT) and of the 16-bit export (uq_export_bcq_half).

* element filter: against oracle.quantize_bwd(filter_mode=FILTER_ELEMENT),
  within 1e-4 x the L1 mass of each reduction, on the pipelined shapes and
  the general-path shapes; dz_U is exactly zero; UQ_FILTER_STE through the
  same entry point is bit-identical to uq_quantize_bwd;
* half export: bit-exact against oracle.export_bcq_half (IEEE half of the
  fp32 export, nearest even), both code modes.
"""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_03781_gb300 import api
from tests import gpu_cases as C

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("out,n_in,g", [(37, 4096, 128), (19, 1024, 64), (11, 768, 32), (9, 1536, 384)])
@pytest.mark.parametrize("q", [2, 3])
def test_element_filter_backward(out, n_in, g, q):
    raw, W, P, codes, Gup = C.make_inputs(out, n_in, q, g, seed=out + q)
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    pd = C.to_dev(P)
    cd = torch.from_numpy(codes).to(d)
    Gd = torch.from_numpy(Gup).to(d)
    gr = api.empty_grads(out, n_in, q, g, d)
    api.uq_quantize_bwd_ex(Wd, q, g, pd, cd, Gd, gr, api.FILTER_ELEMENT)
    args = (W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, Gup, g)
    ref = O.quantize_bwd(*args, filter_mode=O.FILTER_ELEMENT)
    mass = O.bwd_l1_mass(*args, filter_mode=O.FILTER_ELEMENT)
    C.assert_grads_close({k: C.host(v) for k, v in gr.items()}, ref, mass, f"element {out}x{n_in} g{g} q{q}")
    assert np.all(C.host(gr["dzu"]) == 0.0)
    # the STE filter through the same entry point is uq_quantize_bwd, bit for bit
    g1 = api.empty_grads(out, n_in, q, g, d)
    g2 = api.empty_grads(out, n_in, q, g, d)
    api.uq_quantize_bwd_ex(Wd, q, g, pd, cd, Gd, g1, api.FILTER_STE)
    api.uq_quantize_bwd(Wd, q, g, pd, cd, Gd, g2)
    for k in g1:
        assert torch.equal(g1[k], g2[k]), k


@pytest.mark.parametrize("mode", [api.EXPORT_REUSE_CODES, api.EXPORT_REMAP_EQ4])
@pytest.mark.parametrize("q,g", [(2, 64), (3, 128), (4, 32)])
def test_half_export_bit_exact(mode, q, g):
    out, n_in = 21, 1024
    raw, W, P, codes, _ = C.make_inputs(out, n_in, q, g, seed=q + g)
    d = C.dev()
    planes = torch.empty(q, out, n_in // 32, dtype=torch.int32, device=d)
    a16 = torch.empty(out, n_in // g, q, dtype=torch.float16, device=d)
    z16 = torch.empty(out, n_in // g, dtype=torch.float16, device=d)
    api.uq_export_bcq_half(api.weights_tensor(raw, d), q, g, C.to_dev(P), torch.from_numpy(codes).to(d), planes, a16,
                           z16, mode)
    r_planes, r_a, r_z, _ = O.export_bcq_half(W, P["delta"], P["zu"], P["alpha"], P["zb"], codes, g, mode)
    assert np.array_equal(C.host(planes).view(np.uint32), r_planes)
    assert np.array_equal(C.host(a16).view(np.uint16), r_a) and np.array_equal(C.host(z16).view(np.uint16), r_z)
