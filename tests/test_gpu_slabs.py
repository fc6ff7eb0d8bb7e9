"""Grouped quantization (api.RowSlabs): matrices of one input width stored as
row ranges of one slab and quantized by one call per width.  Rows are
independent (groups lie inside rows, s_r is per row), so every output --
codes, W^, every gradient, the fused step's updated parameters and the export
-- must equal that of one call per matrix bit for bit.  A Llama-style block:
two widths, seven matrices of different row counts."""

import numpy as np
import pytest
import torch

from paper_2506_03781_gb300 import api
from tests import gpu_cases as C

pytestmark = pytest.mark.gpu

SHAPES = {"q": (64, 1024), "k": (16, 1024), "v": (16, 1024), "o": (64, 1024), "gate": (88, 1024),
          "up": (88, 1024), "down": (64, 2048)}


def _fill(slabs, seed, q, g):
    d = C.dev()
    gen = torch.Generator(device=d)
    gen.manual_seed(seed)
    for n, (out, n_in) in SHAPES.items():
        v = slabs.view(n)
        v["W"].copy_((torch.randn(out, n_in, generator=gen, device=d) * 0.02).to(v["W"].dtype))
    slabs.init_params(G=4, T=2)
    # one initialization call per matrix gives the same parameters and codes
    for n, (out, n_in) in SHAPES.items():
        v = slabs.view(n)
        p = api.empty_params(out, n_in, q, g, d)
        cd = torch.empty(out, n_in, dtype=torch.uint8, device=d)
        api.uq_init_params(v["W"].contiguous(), q, g, p, cd, G=4, T=2)
        for k in p:
            assert torch.equal(p[k], v["params"][k]), (n, k)
        assert torch.equal(cd, v["codes"]), n
    for sl in slabs.slabs.values():
        for k in ("delta", "s", "sr", "alpha"):
            sl["params"][k].mul_(1.0 + 0.01 * torch.randn(sl["params"][k].shape, generator=gen, device=d))
        sl["dL_dWhat"].copy_(torch.randn(sl["dL_dWhat"].shape, generator=gen, device=d) * 0.01)


def _per_matrix(v, q, g):
    """A per-matrix Quantizer on copies of the matrix's (pre-step) tensors."""
    c = {k: v[k].clone() for k in ("W", "codes", "W_hat", "dL_dWhat")}
    c["params"] = {k: t.clone() for k, t in v["params"].items()}
    c["grads"] = {k: torch.empty_like(t) for k, t in v["grads"].items()}
    c["export"] = tuple(torch.empty_like(t) for t in v["export"])
    c["qz"] = api.Quantizer(c["W"], q, g, c["params"], c["codes"], c["W_hat"], c["dL_dWhat"], c["grads"])
    return c


@pytest.mark.parametrize("q,g", [(2, 64), (3, 128)])
def test_slab_calls_equal_per_matrix_calls(q, g):
    slabs = api.RowSlabs(SHAPES, q, g, torch.bfloat16, C.dev(), with_export=True)
    assert len(slabs.slabs) == 2
    _fill(slabs, 3 + q, q, g)
    refs = {n: _per_matrix(slabs.view(n), q, g) for n in SHAPES}
    for t in (0, 1):                                          # a remap step, then a keep step
        slabs.fwd(t, 2)
        slabs.bwd()
        for c in refs.values():
            c["qz"].fwd(t, 2)
            c["qz"].bwd()
    slabs.export()
    for c in refs.values():
        c["qz"].export(*c["export"])
    slabs.train_step(2)
    for c in refs.values():
        c["qz"].train_step(2)
    torch.cuda.synchronize()
    api.uq_check_device()
    for n in SHAPES:
        v, c = slabs.view(n), refs[n]
        for k in ("codes", "W_hat"):
            assert torch.equal(v[k], c[k]), (n, k)
        for k in v["params"]:
            assert torch.equal(v["params"][k], c["params"][k]), (n, k)
        for k in v["grads"]:
            assert torch.equal(v["grads"][k], c["grads"][k]), (n, k)
        for a, b in zip(v["export"], c["export"]):
            assert torch.equal(a, b), n
