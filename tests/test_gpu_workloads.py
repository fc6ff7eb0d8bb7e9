"""Parity at the full workload sizes, in the launch configuration the
benchmark times (one call per matrix over the whole matrix).

The oracle cannot run a whole 14336x4096 (or larger) matrix through the
unified initialization in test time, so for every workload but the 1k one
the GPU processes the full matrix and the oracle recomputes a sample of rows:
rows are independent (groups lie inside rows, s_r is per row), so a row's
outputs depend only on that row's inputs.  The sampled rows' parameters come
from the oracle's own initialization (jittered by the seeded generator); the
other rows' from the GPU initialization.  Every oracle input is therefore the
oracle's or the generator's, never the CUDA path's.
"""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_03781_gb300 import api, synth
from tests import gpu_cases as C

pytestmark = pytest.mark.gpu
PK = C.PKEYS


def sample_rows(out, n, seed):
    rng = np.random.default_rng(seed)
    rows = set([0, 1, out // 2, out - 1]) | set(rng.choice(out, size=min(out, n), replace=False).tolist())
    return np.array(sorted(rows))


def setup_matrix(wl, idx, rows, q=None):
    """Full-size device inputs + host copies of the sampled rows (see module doc)."""
    m = wl.matrices[idx]
    q = q or wl.q
    g = wl.g
    raw, W = synth.workload_weights(wl, idx)
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    p = api.empty_params(m.out, m.n_in, q, g, d)
    codes = torch.empty(m.out, m.n_in, dtype=torch.uint8, device=d)
    api.uq_init_params(Wd, q, g, p, codes, G=wl.G, T=wl.T)
    init_rows, errs, chosen = O.unified_init(W[rows], q, g, G=wl.G, T=wl.T, return_errors=True)
    full = {k: C.host(v).copy() for k, v in p.items()}
    gpu_init_rows = {k: full[k][rows].copy() for k in PK}
    gpu_codes_rows = C.host(codes)[rows].copy()
    for k in PK:
        full[k][rows] = init_rows[k]
    c_full = C.host(codes).copy()
    c_full[rows] = init_rows["codes"]
    fac = synth.perturb_factors(synth.param_shapes(m.out, m.n_in, g, q), wl.init_eps, (wl.seed, idx, q))
    P = synth.jitter(full, fac)
    return dict(raw=raw, W=W, Wd=Wd, P=P, codes=c_full, init_rows=init_rows, gpu_init_rows=gpu_init_rows,
                gpu_codes_rows=gpu_codes_rows, q=q, g=g, out=m.out, n_in=m.n_in, rows=rows, errs=errs,
                chosen=chosen, G=wl.G, label=m.name)


def init_agreement(s):
    """Every sampled group checked against the oracle (C.check_init); returns
    the fraction of groups with bit-identical parameters."""
    return C.check_init(s["W"][s["rows"]], s["q"], s["g"], s["G"], api.CLIP_FIXED_MIN, s["gpu_init_rows"],
                        s["gpu_codes_rows"], s["init_rows"], s["errs"], s["chosen"], f"{s['label']} q={s['q']}")


def run_and_compare(s, rows, steps=(0,), step_eps=0.0, seed=0, export=True, label=""):
    q, g, d = s["q"], s["g"], C.dev()
    P = {k: v.copy() for k, v in s["P"].items()}
    pd = C.to_dev(P)
    cd = torch.from_numpy(s["codes"]).to(d)
    what = torch.empty(s["out"], s["n_in"], dtype=torch.float32, device=d)
    gr = api.empty_grads(s["out"], s["n_in"], q, g, d)
    Gup = synth.upstream_grad(s["out"], s["n_in"], 1e-4, seed)
    Gd = torch.from_numpy(Gup).to(d)
    r_codes = s["codes"][rows].copy()
    Wr = s["W"][rows]
    for t in steps:
        if step_eps > 0:
            fac = synth.perturb_factors(synth.param_shapes(s["out"], s["n_in"], g, q), step_eps, (seed, 1000 + t))
            P = synth.jitter(P, fac)
            for k in PK:
                pd[k].copy_(torch.from_numpy(P[k]))
        api.uq_quantize_fwd(s["Wd"], q, g, pd, cd, what, api.MAP_LOCAL_PERIODIC, t, 2)
        api.uq_quantize_bwd(s["Wd"], q, g, pd, cd, Gd, gr)
        Pr = C.slice_rows(P, rows)
        r_what, r_codes = O.quantize_fwd(Wr, Pr["s"], Pr["sr"], Pr["delta"], Pr["zu"], Pr["alpha"], Pr["zb"],
                                         r_codes, g, O.MAP_LOCAL_PERIODIC, t, 2)
        C.assert_fwd_equal(C.host(what)[rows], C.host(cd)[rows], r_what, r_codes, f"{label} step {t}")
        ref, mass = C.oracle_bwd(Wr, Pr, r_codes, Gup[rows], g)
        C.assert_grads_close({k: C.host(v)[rows] for k, v in gr.items()}, ref, mass, f"{label} step {t}")
    if export:
        planes = torch.empty(q, s["out"], s["n_in"] // 32, dtype=torch.int32, device=d)
        a_s = torch.empty(s["out"], s["n_in"] // g, q, dtype=torch.float32, device=d)
        z_s = torch.empty(s["out"], s["n_in"] // g, dtype=torch.float32, device=d)
        api.uq_export_bcq(s["Wd"], q, g, pd, cd, planes, a_s, z_s, api.EXPORT_REUSE_CODES)
        Pr = C.slice_rows(P, rows)
        r_planes, r_as, r_zs, _ = O.export_bcq(Wr, Pr["delta"], Pr["zu"], Pr["alpha"], Pr["zb"], r_codes, g)
        assert np.array_equal(C.host(planes).view(np.uint32)[:, rows], r_planes), label
        assert np.array_equal(C.host(a_s)[rows], r_as) and np.array_equal(C.host(z_s)[rows], r_zs), label


@pytest.fixture(scope="module")
def mat1k():
    """1024x1024 fp32 N(0, 0.02^2): small enough for the oracle to do everything."""
    wl = synth.WORKLOADS["mat1k_f32"]
    rows = np.arange(1024)
    return wl, rows, setup_matrix(wl, 0, rows)


def test_mat1k_init_full_matrix(mat1k):
    wl, rows, s = mat1k
    assert init_agreement(s) == 1.0
    assert np.array_equal(s["gpu_codes_rows"], s["init_rows"]["codes"])


def test_mat1k_fwd_bwd_export_full_matrix(mat1k):
    wl, rows, s = mat1k
    run_and_compare(s, rows, steps=(0,), seed=0, label="mat1k")
    # the full mapping (Eq. 2) and the Eq. 4 export on the same inputs
    what, codes = C.gpu_fwd(s["raw"], s["P"], None, wl.q, wl.g, api.MAP_FULL, 0, 2)
    P = s["P"]
    r_what, r_codes = O.quantize_fwd(s["W"], P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], None,
                                     wl.g, O.MAP_FULL)
    C.assert_fwd_equal(what, codes, r_what, r_codes, "mat1k full")
    planes, a_s, z_s = C.gpu_export(s["raw"], P, None, wl.q, wl.g, api.EXPORT_REMAP_EQ4)
    r_planes, r_as, r_zs, _ = O.export_bcq(s["W"], P["delta"], P["zu"], P["alpha"], P["zb"], None, wl.g,
                                           O.EXPORT_REMAP_EQ4)
    assert np.array_equal(planes, r_planes)


def test_attn4k_sampled_rows():
    wl = synth.WORKLOADS["attn4k_bf16"]
    rows = sample_rows(4096, 40, 1)
    s = setup_matrix(wl, 0, rows)
    assert init_agreement(s) == 1.0
    run_and_compare(s, rows, steps=(0, 1), seed=1, label="attn4k")


@pytest.mark.parametrize("q", [2, 3, 4])
def test_mlp14336x4096_multistep_sampled_rows(q):
    """The benchmark workload: local mapping with p = 2 over 4 steps (2 remap,
    2 keep) with the per-step parameter jitter between steps."""
    wl = synth.WORKLOADS["mlp14336x4096_bf16"]
    rows = sample_rows(14336, 28, 2 + q)
    s = setup_matrix(wl, 0, rows, q=q)
    assert init_agreement(s) == 1.0
    run_and_compare(s, rows, steps=(0, 1, 2, 3), step_eps=wl.step_eps, seed=wl.seed, label=f"mlp q={q}")


def test_llama3_8b_block_sampled_rows():
    wl = synth.WORKLOADS["llama3_8b_block_bf16"]
    for idx, m in enumerate(wl.matrices):
        rows = sample_rows(m.out, 12, 30 + idx)
        s = setup_matrix(wl, idx, rows)
        assert init_agreement(s) == 1.0, m.name
        run_and_compare(s, rows, steps=(0,), seed=3 + idx, label=m.name)
        del s
        torch.cuda.empty_cache()


def test_llama2_70b_mlp_sampled_rows():
    wl = synth.WORKLOADS["llama2_70b_mlp_bf16"]
    for idx, m in enumerate(wl.matrices):
        rows = sample_rows(m.out, 6, 40 + idx)
        s = setup_matrix(wl, idx, rows)
        assert init_agreement(s) == 1.0, m.name
        run_and_compare(s, rows, steps=(0,), seed=4 + idx, label=m.name)
        del s
        torch.cuda.empty_cache()
