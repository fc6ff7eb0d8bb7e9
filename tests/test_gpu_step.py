"""GPU parity of the fused optimisation step (uq_train_step): backward of
step t, SGD update of Theta_IF, forward of step t + 1.

Three checks:

* against the oracle (oracle.train_step) on the same seeded inputs.  The
  updated parameters agree within lr x the gradient tolerance (the kernel
  reduces in fp32, the oracle in fp64) plus two fp32 ulps.  The codes of
  step t + 1 agree bit for bit, except where the oracle's own decision is a
  near-tie within the perturbation those parameter tolerances allow (derived
  per element below, and counted).  W^ of step t + 1 agrees within
  1e-6 relative to max(|ref|, Delta max|alpha|);
* against the separate entry points on the GPU (uq_quantize_bwd, the SGD
  update in torch fp32 as fl(theta - fl(lr g)), uq_quantize_fwd at t + 1):
  bit-identical parameters, codes and W^ where both reduce ds_r in the same
  order (rows of at most 8 work units);
* determinism, the thread-block-cluster path (rows of more than 8 units),
  ragged row counts and the full-size workloads on sampled rows.
"""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_03781_gb300 import api, synth
from tests import gpu_cases as C
from tests.test_gpu_workloads import sample_rows, setup_matrix

pytestmark = pytest.mark.gpu
PK = C.PKEYS
F64 = np.float64
LR_F, LR_B = api.LR_THETA_F, api.LR_THETA_B
GRAD = {"delta": "ddelta", "zu": "dzu", "s": "ds", "sr": "dsr", "alpha": "dalpha", "zb": "dzb"}


def gpu_step(raw, P, codes, Gup, q, g, t, mode, p, lr_F=LR_F, lr_B=LR_B):
    out, n_in = raw.shape
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    pd = C.to_dev(P)
    cd = torch.from_numpy(np.ascontiguousarray(codes)).to(d)
    Gd = torch.from_numpy(np.ascontiguousarray(Gup, np.float32)).to(d)
    what = torch.full((out, n_in), float("nan"), dtype=torch.float32, device=d)
    api.uq_train_step(Wd, q, g, pd, cd, Gd, what, t, lr_F, lr_B, mode, p)
    api.uq_check_device(None)
    return {k: C.host(v) for k, v in pd.items()}, C.host(cd), C.host(what)


def param_tolerances(W, P, codes, Gup, g, lr_F, lr_B):
    """Bound on |theta'_gpu - theta'_oracle| per parameter entry (fp64)."""
    grads, mass = C.oracle_bwd(W, P, codes, Gup, g)
    ref = O.sgd_update(P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], grads, lr_F, lr_B)
    tol = {}
    for k in PK:
        lr = lr_F if k in ("delta", "zu", "s", "sr") else lr_B
        if k == "s":
            ds = grads["ds"]
            gm = np.maximum(np.abs(ds), 1e-6 * np.abs(ds).max())
        else:
            gm = mass[GRAD[k]]
        ulp = np.spacing(np.abs(ref[k]).astype(np.float32)).astype(F64)
        prod_ulp = np.spacing(np.abs(lr * grads[GRAD[k]]).astype(np.float32)).astype(F64)
        tol[k] = lr * C.GTOL * gm + 2 * ulp + prod_ulp
    return ref, tol


# Code mismatches allowed per case: every one must also be a near-tie (assert_near_ties).
# Measured over the 109 cases of this file: 1 mismatch in 7,088,640 codes (1.4e-7); the worst
# single case had 1 of 86,016 (1.16e-5).  The cap is four times that worst case.
MAX_TIE_FRAC = 5e-5


def check_against_oracle(raw, W, P, codes, Gup, q, g, t, mode, p, lr_F=LR_F, lr_B=LR_B, label="",
                         max_tie_frac=MAX_TIE_FRAC):
    newP, c1, w1 = gpu_step(raw, P, codes, Gup, q, g, t, mode, p, lr_F, lr_B)
    ref, tol = param_tolerances(W, P, codes, Gup, g, lr_F, lr_B)
    for k in PK:
        err = np.abs(newP[k].astype(F64) - ref[k].astype(F64))
        bad = err > tol[k]
        assert not bad.any(), f"{label}: {k}: {int(bad.sum())} outside tol, worst {(err / tol[k]).max():.3g}x"
    r_what, r_codes = O.quantize_fwd(W, ref["s"], ref["sr"], ref["delta"], ref["zu"], ref["alpha"], ref["zb"],
                                     codes, g, mode, t + 1, p)
    mism = c1 != r_codes
    n_mis = int(mism.sum())
    print(f"step parity {label}: {n_mis} of {c1.size} codes differ from the oracle ({n_mis / c1.size:.2e})")
    if n_mis:
        assert n_mis <= max_tie_frac * c1.size, f"{label}: {n_mis} code mismatches"
        assert_near_ties(W, ref, tol, c1, r_codes, mism, g, label)
    err = np.abs(w1.astype(F64) - r_what.astype(F64))
    bad = ~mism & (err > what_bound(ref, tol, r_codes, r_what, g))
    assert not bad.any(), f"{label}: W^ {int(bad.sum())} outside its bound"
    return newP, c1, w1, n_mis


def what_bound(ref, tol, codes, r_what, g):
    """Bound on |W^_gpu - W^_oracle| where the codes agree: the 1e-6
    relative bound of the forward (max(|ref|, Delta max|alpha|)) plus the
    first-order effect of the parameter tolerances on Delta (l(c) - z_U)."""
    out, n_in = codes.shape
    q = ref["alpha"].shape[-1]
    rep = lambda a: np.repeat(np.asarray(a, F64), g, axis=1).reshape(out, n_in)
    d = rep(ref["delta"])
    amax = rep(np.abs(ref["alpha"]).max(-1))
    cg = codes.reshape(out, -1, g).astype(np.int64)
    lv = ((O.signs(q, F64)[cg] * ref["alpha"][..., None, :].astype(F64)).sum(-1)
          + ref["zb"][..., None].astype(F64)).reshape(out, n_in)
    dlv = rep(tol["alpha"].sum(-1) + tol["zb"])
    prop = rep(tol["delta"]) * np.abs(lv - rep(ref["zu"])) + np.abs(d) * (dlv + rep(tol["zu"]))
    return 1e-6 * np.maximum(np.abs(r_what.astype(F64)), np.abs(d) * amax) + 1.01 * prop


def assert_near_ties(W, ref, tol, c_gpu, c_ora, mism, g, label):
    """Every code mismatch must be a decision the oracle takes by a margin
    smaller than the parameter tolerances can move it (fp64 evaluation)."""
    out, n_in = W.shape
    q = ref["alpha"].shape[-1]
    rows, cols = np.nonzero(mism)
    grp = cols // g
    d = ref["delta"][rows, grp].astype(F64)
    zu = ref["zu"][rows, grp].astype(F64)
    s = ref["s"][rows, cols].astype(F64)
    sr = ref["sr"][rows].astype(F64)
    u = W[rows, cols].astype(F64) / (d * s * sr)
    x = u + zu
    dx = np.abs(u) * (tol["delta"][rows, grp] / np.abs(d) + tol["s"][rows, cols] / np.abs(s)
                      + tol["sr"][rows] / np.abs(sr)) + tol["zu"][rows, grp]
    dl = tol["alpha"][rows, grp].sum(-1) + tol["zb"][rows, grp]
    sg = O.signs(q, F64)
    lv = lambda c: (sg[c.astype(np.int64)] * ref["alpha"][rows, grp].astype(F64)).sum(-1) + \
        ref["zb"][rows, grp].astype(F64)
    gap = np.abs(np.abs(x - lv(c_gpu[rows, cols])) - np.abs(x - lv(c_ora[rows, cols])))
    margin = 2 * (dx + dl) + 8 * np.spacing(np.abs(x).astype(np.float32)).astype(F64)
    assert (gap <= margin).all(), f"{label}: a code mismatch is not a near-tie (gap/margin {(gap / margin).max()})"


def separate_path(raw, P, codes, Gup, q, g, t, mode, p, lr_F=LR_F, lr_B=LR_B):
    """bwd kernel, torch fp32 SGD fl(theta - fl(lr g)), fwd kernel at t + 1."""
    out, n_in = raw.shape
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    pd = C.to_dev(P)
    cd = torch.from_numpy(np.ascontiguousarray(codes)).to(d)
    Gd = torch.from_numpy(np.ascontiguousarray(Gup, np.float32)).to(d)
    gr = api.empty_grads(out, n_in, q, g, d)
    api.uq_quantize_bwd(Wd, q, g, pd, cd, Gd, gr)
    for k in PK:
        lr = lr_F if k in ("delta", "zu", "s", "sr") else lr_B
        step = gr[GRAD[k]] * np.float32(lr)
        pd[k].copy_(pd[k] - step)
    what = torch.empty(out, n_in, dtype=torch.float32, device=d)
    api.uq_quantize_fwd(Wd, q, g, pd, cd, what, mode, t + 1, p)
    return {k: C.host(v) for k, v in pd.items()}, C.host(cd), C.host(what)


# ---------------------------------------------------------------------------
# small shapes: every template path
# ---------------------------------------------------------------------------

# (out, in, g): rows of 1, 2, 3, 8 work units (R = 8, 4, 2, 1 rows per block),
# and 16, 28, 56, 64 units (clusters of 2, 4, 7, 8 blocks)
SHAPES = [(64, 512, 128), (40, 1024, 64), (21, 768, 32), (37, 4096, 128),
          (10, 8192, 128), (6, 14336, 128), (3, 28672, 128), (2, 16384, 32)]


@pytest.mark.parametrize("out,n_in,g", SHAPES)
@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_step_matches_oracle_all_modes(out, n_in, g, q):
    raw, W, P, codes, Gup = C.make_inputs(out, n_in, q, g, seed=out + n_in + q)
    for t, mode in ((0, O.MAP_LOCAL_PERIODIC), (1, O.MAP_LOCAL_PERIODIC), (0, O.MAP_FULL)):
        check_against_oracle(raw, W, P, codes, Gup, q, g, t, mode, 2, label=f"{out}x{n_in} g{g} q{q} t{t} m{mode}")


@pytest.mark.parametrize("wd", ["f32", "bf16"])
def test_step_fp32_and_bf16_weights(wd):
    raw, W, P, codes, Gup = C.make_inputs(24, 2048, 3, 128, seed=11, wdtype=wd)
    check_against_oracle(raw, W, P, codes, Gup, 3, 128, 1, O.MAP_LOCAL_PERIODIC, 2, label=wd)


def test_large_learning_rates_move_codes():
    """Learning rates x200: the step moves many codes; the remap of step
    t + 1 still matches the oracle up to counted near-ties."""
    q, g = 3, 128
    raw, W, P, codes, Gup = C.make_inputs(32, 2048, q, g, seed=12)
    newP, c1, _, n_mis = check_against_oracle(raw, W, P, codes, Gup, q, g, 1, O.MAP_LOCAL_PERIODIC, 2,
                                              lr_F=LR_F * 200, lr_B=LR_B * 200, label="lr x200")
    assert (c1 != codes).mean() > 1e-3


@pytest.mark.parametrize("out,n_in,g", [s for s in SHAPES if s[1] // (256 if s[2] == 32 else 512) <= 8])
def test_step_equals_separate_entry_points(out, n_in, g):
    q = 3
    raw, W, P, codes, Gup = C.make_inputs(out, n_in, q, g, seed=5 + out)
    for t, mode in ((0, O.MAP_LOCAL_PERIODIC), (1, O.MAP_LOCAL_PERIODIC), (0, O.MAP_FULL)):
        a = gpu_step(raw, P, codes, Gup, q, g, t, mode, 2)
        b = separate_path(raw, P, codes, Gup, q, g, t, mode, 2)
        for k in PK:
            assert np.array_equal(a[0][k], b[0][k]), (k, t, mode)
        assert np.array_equal(a[1], b[1]) and np.array_equal(a[2], b[2]), (t, mode)


@pytest.mark.parametrize("q,g", [(2, 64), (3, 128)])
def test_step_filter_boundary_within_ulps(q, g):
    """Weights within 4 ulps of the filter boundary (every vector of the
    backward phase takes the IEEE fallback): the fused step still equals the
    separate entry points bit for bit, and the oracle (the forward of t + 1 is
    a keep step, so no mapping near-ties enter)."""
    out, n_in = 16, 1024
    _, W0, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=40 + q, wdtype="f32")
    _, codes = O.quantize_fwd(W0, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                              O.MAP_LOCAL_PERIODIC, 0, 2)
    W, gap = C.boundary_weights(P, codes, g, seed=q)
    assert 0.3 < (gap > 0).mean() < 0.7
    a = gpu_step(W, P, codes, Gup, q, g, 0, O.MAP_LOCAL_PERIODIC, 2)
    b = separate_path(W, P, codes, Gup, q, g, 0, O.MAP_LOCAL_PERIODIC, 2)
    for k in PK:
        assert np.array_equal(a[0][k], b[0][k]), k
    assert np.array_equal(a[1], b[1]) and np.array_equal(a[2], b[2])
    check_against_oracle(W, W, P, codes, Gup, q, g, 0, O.MAP_LOCAL_PERIODIC, 2, label=f"boundary q{q} g{g}")


def test_multistep_chain_equals_separate_entry_points():
    """Eight consecutive steps (remap and keep alternating) on each path,
    each from its own state: still bit-identical."""
    q, g = 3, 128
    raw, W, P, codes, Gup0 = C.make_inputs(48, 4096, q, g, seed=21)
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    pa, pb = C.to_dev(P), C.to_dev(P)
    ca = torch.from_numpy(codes.copy()).to(d)
    cb = ca.clone()
    wa = torch.empty(48, 4096, dtype=torch.float32, device=d)
    wb = torch.empty_like(wa)
    gr = api.empty_grads(48, 4096, q, g, d)
    for t in range(8):
        Gd = torch.from_numpy(synth.upstream_grad(48, 4096, 1e-4, (21, t))).to(d)
        api.uq_train_step(Wd, q, g, pa, ca, Gd, wa, t)
        api.uq_quantize_bwd(Wd, q, g, pb, cb, Gd, gr)
        for k in PK:
            lr = LR_F if k in ("delta", "zu", "s", "sr") else LR_B
            pb[k].copy_(pb[k] - gr[GRAD[k]] * np.float32(lr))
        api.uq_quantize_fwd(Wd, q, g, pb, cb, wb, api.MAP_LOCAL_PERIODIC, t + 1, 2)
        torch.cuda.synchronize()
        for k in PK:
            assert torch.equal(pa[k], pb[k]), (t, k)
        assert torch.equal(ca, cb) and torch.equal(wa, wb), t


@pytest.mark.parametrize("out,n_in,g", [(64, 512, 128), (5, 28672, 128), (3, 16384, 32)])
def test_step_is_deterministic(out, n_in, g):
    raw, W, P, codes, Gup = C.make_inputs(out, n_in, 2, g, seed=3)
    a = gpu_step(raw, P, codes, Gup, 2, g, 1, O.MAP_LOCAL_PERIODIC, 2)
    b = gpu_step(raw, P, codes, Gup, 2, g, 1, O.MAP_LOCAL_PERIODIC, 2)
    for k in PK:
        assert np.array_equal(a[0][k], b[0][k]), k
    assert np.array_equal(a[1], b[1]) and np.array_equal(a[2], b[2])


@pytest.mark.parametrize("out", [1, 2, 7, 9])
def test_step_ragged_row_counts(out):
    """Fewer rows than one block's rows (R = 8), or than clusters."""
    for n_in, g in ((512, 128), (28672, 128)):
        raw, W, P, codes, Gup = C.make_inputs(out, n_in, 2, g, seed=out)
        check_against_oracle(raw, W, P, codes, Gup, 2, g, 1, O.MAP_LOCAL_PERIODIC, 2, label=f"{out}x{n_in}")


def test_step_zero_gradient_is_the_next_forward():
    q, g = 3, 128
    raw, W, P, codes, _ = C.make_inputs(16, 4096, q, g, seed=8)
    zero = np.zeros((16, 4096), np.float32)
    newP, c1, w1 = gpu_step(raw, P, codes, zero, q, g, 1, O.MAP_LOCAL_PERIODIC, 2)
    for k in PK:
        assert np.array_equal(newP[k], P[k]), k
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, g,
                                     O.MAP_LOCAL_PERIODIC, 2, 2)
    C.assert_fwd_equal(w1, c1, r_what, r_codes, "zero gradient")


def test_step_on_side_stream_and_check_device():
    q, g = 2, 64
    raw, W, P, codes, Gup = C.make_inputs(8, 1024, q, g, seed=9)
    d = C.dev()
    s = torch.cuda.Stream(d)
    Wd = api.weights_tensor(raw, d)
    pd = C.to_dev(P)
    cd = torch.from_numpy(codes.copy()).to(d)
    Gd = torch.from_numpy(Gup).to(d)
    what = torch.empty(8, 1024, dtype=torch.float32, device=d)
    torch.cuda.synchronize()
    with torch.cuda.stream(s):
        api.uq_train_step(Wd, q, g, pd, cd, Gd, what, 0, stream=s)
    api.uq_check_device(s)
    ref = gpu_step(raw, P, codes, Gup, q, g, 0, O.MAP_LOCAL_PERIODIC, 2)
    assert np.array_equal(C.host(what), ref[2]) and np.array_equal(C.host(cd), ref[1])


def test_unsupported_shape_raises_before_launch():
    d = C.dev()
    W = torch.zeros(4, 768, dtype=torch.bfloat16, device=d)          # 1.5 units of 512
    p = api.empty_params(4, 768, 3, 128, d)
    with pytest.raises(api.UQError) as e:
        api.uq_train_step(W, 3, 128, p, torch.zeros(4, 768, dtype=torch.uint8, device=d),
                          torch.zeros(4, 768, device=d), torch.zeros(4, 768, device=d), 0)
    assert e.value.status == api.UQ_ERR_UNSUPPORTED


def test_quantizer_train_step_in_a_cuda_graph():
    q, g = 3, 128
    raw, W, P, codes, Gup = C.make_inputs(32, 4096, q, g, seed=13)
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    pd = C.to_dev(P)
    cd = torch.from_numpy(codes.copy()).to(d)
    Gd = torch.from_numpy(Gup).to(d)
    what = torch.empty(32, 4096, dtype=torch.float32, device=d)
    Qz = api.Quantizer(Wd, q, g, pd, cd, what, Gd, api.empty_grads(32, 4096, q, g, d))
    s = torch.cuda.Stream(d)
    s.wait_stream(torch.cuda.current_stream(d))
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=s):
        Qz.train_step(1)
    # capture does not run the kernel: restore nothing, replay once
    graph.replay()
    torch.cuda.synchronize()
    ref = gpu_step(raw, P, codes, Gup, q, g, 1, O.MAP_LOCAL_PERIODIC, 2)
    for k in PK:
        assert np.array_equal(C.host(pd[k]), ref[0][k]), k
    assert np.array_equal(C.host(cd), ref[1]) and np.array_equal(C.host(what), ref[2])


# ---------------------------------------------------------------------------
# full-size workloads, sampled rows (the launch configuration of the benchmark)
# ---------------------------------------------------------------------------

def full_size_step(wl, idx, rows, t, label):
    s = setup_matrix(wl, idx, rows)
    q, g, d = s["q"], s["g"], C.dev()
    pd = C.to_dev(s["P"])
    cd = torch.from_numpy(s["codes"]).to(d)
    Gup = synth.upstream_grad(s["out"], s["n_in"], 1e-4, (wl.seed, idx, t))
    Gd = torch.from_numpy(Gup).to(d)
    what = torch.empty(s["out"], s["n_in"], dtype=torch.float32, device=d)
    api.uq_train_step(s["Wd"], q, g, pd, cd, Gd, what, t)
    newP = {k: C.host(v)[rows] for k, v in pd.items()}
    c1, w1 = C.host(cd)[rows], C.host(what)[rows]
    Pr = C.slice_rows(s["P"], rows)
    Wr, cr, Gr = s["W"][rows], s["codes"][rows], Gup[rows]
    ref, tol = param_tolerances(Wr, Pr, cr, Gr, g, LR_F, LR_B)
    for k in PK:
        err = np.abs(newP[k].astype(F64) - ref[k].astype(F64))
        assert (err <= tol[k]).all(), f"{label}: {k}"
    r_what, r_codes = O.quantize_fwd(Wr, ref["s"], ref["sr"], ref["delta"], ref["zu"], ref["alpha"], ref["zb"],
                                     cr, g, O.MAP_LOCAL_PERIODIC, t + 1, 2)
    mism = c1 != r_codes
    assert mism.sum() <= 1e-4 * c1.size, label
    if mism.any():
        assert_near_ties(Wr, ref, tol, c1, r_codes, mism, g, label)
    err = np.abs(w1.astype(F64) - r_what.astype(F64))
    assert ((err <= what_bound(ref, tol, r_codes, r_what, g)) | mism).all(), label


@pytest.mark.parametrize("t", [0, 1])
def test_mlp14336x4096_step_sampled_rows(t):
    wl = synth.WORKLOADS["mlp14336x4096_bf16"]
    full_size_step(wl, 0, sample_rows(14336, 40, 7 + t), t, f"mlp t{t}")


def test_llama2_70b_down_proj_step_sampled_rows():
    """8192 x 28672: 56 work units per row, a cluster of 7 blocks per row."""
    wl = synth.WORKLOADS["llama2_70b_mlp_bf16"]
    idx = [i for i, m in enumerate(wl.matrices) if m.n_in == 28672][0]
    full_size_step(wl, idx, sample_rows(wl.matrices[idx].out, 12, 17), 1, "70b down")


@pytest.mark.parametrize("out,n_in,g", [(64, 512, 128), (21, 768, 32), (37, 4096, 128), (6, 14336, 128)])
@pytest.mark.parametrize("q", [2, 3])
def test_step_bf16_io_equals_the_fp32_step(out, n_in, g, q):
    """uq_train_step_bf16 reads dL/dW^ as bf16 and writes W^ as bf16: given
    dL/dW^ values that bf16 represents exactly, its parameters and codes
    equal uq_train_step's bit for bit, and its W^ is the fp32 step's W^
    rounded to nearest even (torch's fp32 -> bf16 conversion), for a
    remapping and a keeping forward of t + 1 and rows split over a cluster."""
    raw, W, P, codes, Gup = C.make_inputs(out, n_in, q, g, seed=60 + out + q)
    _, Gb = synth.bf16_round(Gup)                 # values exact in bf16
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    for t in (0, 1):
        pa, pb = C.to_dev(P), C.to_dev(P)
        ca = torch.from_numpy(np.ascontiguousarray(codes)).to(d)
        cb = ca.clone()
        Ga = torch.from_numpy(np.ascontiguousarray(Gb)).to(d)
        wa = torch.full((out, n_in), float("nan"), device=d)
        wb = torch.full((out, n_in), float("nan"), device=d).to(torch.bfloat16)
        api.uq_train_step(Wd, q, g, pa, ca, Ga, wa, t)
        api.uq_train_step_bf16(Wd, q, g, pb, cb, Ga.to(torch.bfloat16), wb, t)
        api.uq_check_device(None)
        for k in PK:
            assert torch.equal(pa[k], pb[k]), (k, t)
        assert torch.equal(ca, cb), t
        assert torch.equal(wa.to(torch.bfloat16), wb), (t, int((wa.to(torch.bfloat16) != wb).sum()))


@pytest.mark.parametrize("out,n_in,g,q", [(24, 1024, 128, 3), (16, 768, 32, 2), (6, 14336, 128, 4)])
def test_step_remap_near_level_midpoints_is_bit_exact(out, n_in, g, q):
    """With zero learning rates the update leaves every parameter unchanged,
    so the forward of t + 1 remaps with the levels the weights were aimed at:
    every element within 4 ulps of a midpoint between its level and a rank
    neighbour.  Codes and W^ must be the oracle's bit for bit (phase B takes
    the reciprocal only inside a proven interval, else the IEEE path)."""
    _, W0, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=900 + out + q, wdtype="f32")
    W = C.midpoint_weights(P, codes0, g, seed=out + q)
    newP, c1, w1 = gpu_step(W, P, codes0, Gup, q, g, 1, O.MAP_LOCAL_PERIODIC, 2, lr_F=0.0, lr_B=0.0)
    for k in PK:
        assert np.array_equal(newP[k], P[k]), k
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 2, 2)
    C.assert_fwd_equal(w1, c1, r_what, r_codes, f"step midpoints q={q} g={g}")
    assert (r_codes != codes0).mean() > 0.05
