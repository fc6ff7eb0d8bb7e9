"""GPU parity of the BCQ product from the exported format (uq_bcq_gemv)
against the oracle's fp64 product (oracle.bcq_gemv).

Tolerance: the kernel accumulates in fp32 in its own fixed order (per-8-
column partial sums of x, per-lane terms z* S + sum_j alpha*_j (2 P_j - S),
a warp reduction, then the tiles).  Every rounding error is bounded by a
small multiple of the unit roundoff times the L1 mass of the expanded terms,
sum_i (sum_j |alpha*_j| + |z*|) |x_i| (computed in fp64 here); the tests
allow 1e-5 of that mass (about 170 unit roundoffs).
"""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_03781_gb300 import api, synth
from tests import gpu_cases as C

pytestmark = pytest.mark.gpu
F32 = np.float32
F64 = np.float64
TOL = 1e-5


def mass(a_star, z_star, x, g):
    per_col = np.repeat(np.abs(np.asarray(a_star, F64)).sum(-1) + np.abs(np.asarray(z_star, F64)), g, axis=1)
    return np.abs(np.asarray(x, F64)) @ per_col.T             # [batch, out]


def random_export(out, n_in, q, g, seed):
    rng = np.random.default_rng(seed)
    planes = rng.integers(0, 2 ** 32, (q, out, n_in // 32), dtype=np.uint64).astype(np.uint32)
    a_star = (rng.standard_normal((out, n_in // g, q)) * 0.01).astype(F32)
    z_star = (rng.standard_normal((out, n_in // g)) * 0.003).astype(F32)
    return planes, a_star, z_star


def gpu_gemv(planes, a_star, z_star, x, g, xdtype="f32"):
    d = C.dev()
    pd = torch.from_numpy(planes.view(np.int32)).to(d)
    ad = torch.from_numpy(a_star).to(d)
    zd = torch.from_numpy(z_star).to(d)
    if xdtype == "bf16":
        raw, _ = synth.bf16_round(x)
        xd = api.weights_tensor(raw, d)
    else:
        xd = torch.from_numpy(np.ascontiguousarray(x, F32)).to(d)
    y = torch.full((x.shape[0], planes.shape[1]), float("nan"), device=d)
    # the workspace starts as NaN: every word the product reads must have been written by it
    ws = torch.full((api.uq_bcq_gemv_workspace_bytes(planes.shape[1], x.shape[1], x.shape[0]) // 4,), float("nan"),
                    device=d)
    api.uq_bcq_gemv(pd, ad, zd, xd, y, g, workspace=ws)
    api.uq_check_device()                         # no pipeline wait ran out, no layout refused
    return C.host(y)


def check(planes, a_star, z_star, x, g, xdtype="f32", label=""):
    if xdtype == "bf16":
        _, x = synth.bf16_round(x)               # the oracle sees the values the kernel reads
    y = gpu_gemv(planes, a_star, z_star, x, g, xdtype)
    ref = O.bcq_gemv(planes, a_star, z_star, x, g)
    err = np.abs(y.astype(F64) - ref)
    bound = TOL * mass(a_star, z_star, x, g) + 1e-30
    assert np.isfinite(y).all(), label
    assert (err <= bound).all(), f"{label}: worst {(err / bound).max():.3g} x tolerance"
    return y


# in: one ragged tile, several tiles, a non-multiple of 512.  In a multiple of 1024 with
# g <= 256 takes the wide-lane kernel (1024-column tiles, 4 to 32 groups per tile); other
# whole 512-column tiles with 4, 8 and 16 groups per tile the tensor-copy staging, the
# rest the per-lane copies
@pytest.mark.parametrize("out,n_in,g", [(40, 256, 32), (33, 512, 64), (17, 1536, 128), (64, 4096, 128),
                                        (9, 4096 + 32 * 3, 32), (5, 8192, 256), (3, 28672, 128), (300, 1024, 512),
                                        (24, 1024, 32), (13, 2560, 64), (11, 3072, 1024), (6, 4096, 2048)])
@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_gemv_matches_oracle(out, n_in, g, q):
    if n_in % g:
        pytest.skip("in must be a multiple of g")
    planes, a_star, z_star = random_export(out, n_in, q, g, seed=out + q)
    x = np.random.default_rng(q).standard_normal((1, n_in)).astype(F32)
    check(planes, a_star, z_star, x, g, label=f"{out}x{n_in} g{g} q{q}")


@pytest.mark.parametrize("batch", [2, 5])
@pytest.mark.parametrize("xdtype", ["f32", "bf16"])
def test_gemv_batches_and_bf16_activations(batch, xdtype):
    planes, a_star, z_star = random_export(48, 2048, 3, 128, seed=7)
    x = np.random.default_rng(batch).standard_normal((batch, 2048)).astype(F32)
    check(planes, a_star, z_star, x, 128, xdtype, label=f"batch {batch} {xdtype}")


@pytest.mark.parametrize("out,n_in,g,q", [(9000, 512, 64, 2), (9001, 2048, 64, 2), (2053, 3072, 32, 4),
                                          (1, 1024, 256, 1), (7, 1024, 128, 3)])
def test_gemv_many_rows(out, n_in, g, q):
    """Many more rows than one wave of row blocks, a ragged last batch of
    rows, and single-row and single-tile products, on both kernels."""
    planes, a_star, z_star = random_export(out, n_in, q, g, seed=9 + out)
    x = np.random.default_rng(0).standard_normal((2, n_in)).astype(F32)
    check(planes, a_star, z_star, x, g, label=f"{out} rows {n_in} g{g} q{q}")


def test_gemv_deterministic():
    planes, a_star, z_star = random_export(100, 8192, 3, 128, seed=11)
    x = np.random.default_rng(1).standard_normal((2, 8192)).astype(F32)
    a = gpu_gemv(planes, a_star, z_star, x, 128)
    b = gpu_gemv(planes, a_star, z_star, x, 128)
    assert np.array_equal(a, b)


def test_gemv_of_the_quantizer_export_reproduces_w_hat():
    """End to end on the GPU: forward (W^), export (bit-planes, alpha*, z*),
    then the product from the export alone against the oracle's product of
    the oracle's own export, and against x W^T (Theorem 1)."""
    q, g = 3, 128
    raw, W, P, codes, _ = C.make_inputs(64, 2048, q, g, seed=4)
    what, codes1 = C.gpu_fwd(raw, P, codes, q, g, api.MAP_LOCAL_PERIODIC, 0, 2)
    planes, a_s, z_s = C.gpu_export(raw, P, codes1, q, g, api.EXPORT_REUSE_CODES)
    r_planes, r_as, r_zs, _ = O.export_bcq(W, P["delta"], P["zu"], P["alpha"], P["zb"], codes1, g)
    x = np.random.default_rng(5).standard_normal((3, 2048)).astype(F32)
    y = gpu_gemv(planes, a_s, z_s, x, g)
    ref = O.bcq_gemv(r_planes, r_as, r_zs, x, g)
    assert (np.abs(y - ref) <= TOL * mass(r_as, r_zs, x, g)).all()
    # Theorem 1: the same numbers as the quantizer's own output times x
    thm = x.astype(F64) @ what.astype(F64).T
    assert (np.abs(y - thm) <= 2 * TOL * mass(r_as, r_zs, x, g)).all()


def test_gemv_full_size_headline_matrix():
    """14336 x 4096, q = 3, g = 128 (the benchmark's export), every row."""
    q, g, out, n_in = 3, 128, 14336, 4096
    planes, a_star, z_star = random_export(out, n_in, q, g, seed=21)
    x = np.random.default_rng(2).standard_normal((1, n_in)).astype(F32)
    check(planes, a_star, z_star, x, g, label="14336x4096")


def test_gemv_full_size_70b_down_projection_sampled():
    """8192 x 28672: the oracle recomputes a sample of rows (rows are
    independent: each output is one row of the product)."""
    q, g, out, n_in = 3, 128, 8192, 28672
    planes, a_star, z_star = random_export(out, n_in, q, g, seed=22)
    x = np.random.default_rng(3).standard_normal((1, n_in)).astype(F32)
    y = gpu_gemv(planes, a_star, z_star, x, g)
    rows = np.array(sorted(set([0, 1, 4095, 4096, out - 1]) | set(np.random.default_rng(0).choice(out, 40).tolist())))
    ref = O.bcq_gemv(np.ascontiguousarray(planes[:, rows]), a_star[rows], z_star[rows], x, g)
    assert (np.abs(y[:, rows] - ref) <= TOL * mass(a_star[rows], z_star[rows], x, g)).all()


def test_gemv_rejects_a_small_workspace():
    d = C.dev()
    planes, a_star, z_star = random_export(16, 1024, 2, 64, seed=1)
    need = api.uq_bcq_gemv_workspace_bytes(16, 1024, 1)
    assert need == 2 * 16 * 4
    ws = torch.empty(need // 4 - 1, device=d)
    y = torch.empty(1, 16, device=d)
    with pytest.raises(api.UQError) as e:
        api.uq_bcq_gemv(torch.from_numpy(planes.view(np.int32)).to(d), torch.from_numpy(a_star).to(d),
                        torch.from_numpy(z_star).to(d), torch.zeros(1, 1024, device=d), y, 64, workspace=ws)
    assert e.value.status == api.UQ_ERR_ARG
