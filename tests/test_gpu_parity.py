"""GPU parity of the CUDA library (through the C ABI) against the CPU oracle
on small and ragged shapes, every bit-width, group-size class, weight dtype
and mode, plus edge cases, determinism, buffer bounds and streams."""

import numpy as np
import pytest
import torch

import oracle as O
from paper_2506_03781_gb300 import api, synth
from tests import gpu_cases as C

pytestmark = pytest.mark.gpu

QS = [1, 2, 3, 4]
GS = [32, 64, 128, 256]


def shape_for(g):
    # several warp-steps, a partial last warp-step for g < 128, several
    # batches per warp for the larger rows
    return {32: (37, 32 * 45), 64: (29, 64 * 9), 128: (23, 128 * 72), 256: (11, 256 * 6)}[g]


@pytest.mark.parametrize("wd", ["bf16", "f32"])
@pytest.mark.parametrize("g", GS)
@pytest.mark.parametrize("q", QS)
def test_fwd_all_modes(q, g, wd):
    out, n_in = shape_for(g)
    raw, W, P, codes0, _ = C.make_inputs(out, n_in, q, g, seed=100 * q + g, wdtype=wd)
    # full mapping (Eq. 2)
    what, codes = C.gpu_fwd(raw, P, None, q, g, api.MAP_FULL, 0, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], None, g,
                                     O.MAP_FULL)
    C.assert_fwd_equal(what, codes, r_what, r_codes, "full")
    # local remap step (Algorithm 4) from the initial codes
    what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 4, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 4, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, "remap")
    assert (r_codes != codes0).any()
    # keep step: codes untouched, w~ recomputed with the current levels
    what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 3, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 3, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, "keep")
    assert np.array_equal(codes, codes0)


@pytest.mark.parametrize("wd", ["bf16", "f32"])
@pytest.mark.parametrize("g", GS + [384])
@pytest.mark.parametrize("q", QS)
def test_bwd(q, g, wd):
    out, n_in = shape_for(g) if g != 384 else (7, 384 * 5)
    raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=300 * q + g, wdtype=wd)
    _, codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                              O.MAP_LOCAL_PERIODIC, 0, 2)
    gr = C.gpu_bwd(raw, P, codes, Gup, q, g)
    ref, mass = C.oracle_bwd(W, P, codes, Gup, g)
    C.assert_grads_close(gr, ref, mass, f"q={q} g={g} {wd}")
    # the filter is exercised: some elements are filtered, most are not
    assert 0 < (gr["ds"] == 0).mean() < 0.5


@pytest.mark.parametrize("mode", [api.EXPORT_REUSE_CODES, api.EXPORT_REMAP_EQ4])
@pytest.mark.parametrize("g", GS)
@pytest.mark.parametrize("q", QS)
def test_export(q, g, mode):
    out, n_in = shape_for(g)
    raw, W, P, codes0, _ = C.make_inputs(out, n_in, q, g, seed=500 * q + g, wdtype="bf16")
    planes, a_s, z_s = C.gpu_export(raw, P, codes0, q, g, mode)
    r_planes, r_as, r_zs, r_codes = O.export_bcq(W, P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                                 O.EXPORT_REMAP_EQ4 if mode else O.EXPORT_REUSE_CODES)
    assert np.array_equal(a_s, r_as) and np.array_equal(z_s, r_zs)
    assert np.array_equal(planes, r_planes), int((planes != r_planes).sum())


@pytest.mark.parametrize("clip", [api.CLIP_FIXED_MIN, api.CLIP_FIXED_MAX, api.CLIP_BALANCED])
@pytest.mark.parametrize("G,T", [(1, 15), (7, 5)])
@pytest.mark.parametrize("g", [32, 64, 128, 256])
@pytest.mark.parametrize("q", QS)
def test_init(q, g, G, T, clip):
    out, n_in = 9, g * 6
    rng = np.random.default_rng(q * 1000 + g)
    raw, W = synth.bf16_round((rng.standard_t(4, (out, n_in)) * 0.014).astype(np.float32))
    Wd = api.weights_tensor(raw, C.dev())
    p = api.empty_params(out, n_in, q, g, C.dev())
    codes = torch.empty(out, n_in, dtype=torch.uint8, device=C.dev())
    api.uq_init_params(Wd, q, g, p, codes, G=G, T=T, clip=clip)
    ref, errs, chosen = O.unified_init(W, q, g, G=G, T=T, clip=clip, return_errors=True)
    got = {k: C.host(v) for k, v in p.items()}
    # every group: candidate, error, gamma index and codes (see check_init)
    same = C.check_init(W, q, g, G, clip, got, C.host(codes), ref, errs, chosen, f"q={q} g={g} G={G} clip={clip}")
    # measured: every group bit-identical in every case (fp64 sums are exact here)
    assert same == 1.0, same
    assert np.all(got["s"] == 1) and np.all(got["sr"] == 1)


def test_edge_tiny_and_degenerate():
    # one row, one group of 32, one bit; and a constant row for init
    q, g = 1, 32
    raw, W = synth.bf16_round(np.linspace(-0.05, 0.05, 32, dtype=np.float32)[None, :])
    Wd = api.weights_tensor(raw, C.dev())
    p = api.empty_params(1, 32, q, g, C.dev())
    codes = torch.empty(1, 32, dtype=torch.uint8, device=C.dev())
    api.uq_init_params(Wd, q, g, p, codes, G=30, T=15)
    ref = O.unified_init(W, q, g, G=30, T=15)
    assert np.array_equal(C.host(codes), ref["codes"])
    Wc = np.full((2, 128), 0.0123, np.float32)
    raw, W = synth.bf16_round(Wc)
    Wd = api.weights_tensor(raw, C.dev())
    p = api.empty_params(2, 128, 3, 128, C.dev())
    codes = torch.empty(2, 128, dtype=torch.uint8, device=C.dev())
    api.uq_init_params(Wd, 3, 128, p, codes, G=30, T=15)
    for k, v in p.items():
        assert torch.isfinite(v).all(), k


@pytest.mark.parametrize("clip", [api.CLIP_FIXED_MIN, api.CLIP_FIXED_MAX, api.CLIP_BALANCED])
@pytest.mark.parametrize("q,g", [(2, 64), (3, 128), (4, 32), (3, 256)])
def test_init_singular_gram_groups_match_the_oracle_bit_for_bit(q, g, clip):
    """Constant weight groups make C^T C exactly singular in every round of
    Algorithm 3 (the greedy start leaves a zero residual, so every bit after
    the first is +1); alpha must then keep its value (reading R11), which the
    oracle pins.  Such groups sit between ordinary groups of the same rows,
    and every group is compared with the oracle: the constant ones bit for
    bit in every parameter and code, the rest through check_init."""
    out, n_in = 6, g * 5
    rng = np.random.default_rng(7 * q + g + clip)
    W32 = (rng.standard_t(4, (out, n_in)) * 0.014).astype(np.float32)
    W32.reshape(out, -1, g)[1::2, 1::2] = np.float32(0.0123)
    W32.reshape(out, -1, g)[0, 2] = np.float32(-0.04)
    raw, W = synth.bf16_round(W32)
    Wd = api.weights_tensor(raw, C.dev())
    p = api.empty_params(out, n_in, q, g, C.dev())
    codes = torch.empty(out, n_in, dtype=torch.uint8, device=C.dev())
    api.uq_init_params(Wd, q, g, p, codes, G=7, T=5, clip=clip)
    ref, errs, chosen = O.unified_init(W, q, g, G=7, T=5, clip=clip, return_errors=True)
    got = {k: C.host(v) for k, v in p.items()}
    gc = C.host(codes)
    const = (W.reshape(out, -1, g) == W.reshape(out, -1, g)[..., :1]).all(-1)
    assert const.sum() >= 7
    for k in ("delta", "zu", "zb", "alpha"):
        assert np.array_equal(got[k][const], ref[k][const]), k
    assert np.all(ref["alpha"][const][:, 1:] == 0)
    assert np.array_equal(gc.reshape(out, -1, g)[const], ref["codes"].reshape(out, -1, g)[const])
    C.check_init(W, q, g, 7, clip, got, gc, ref, errs, chosen, f"singular q={q} g={g} clip={clip}")


def test_edge_level_ties_negative_alpha_and_high_code_bits():
    """alpha_1 == alpha_2 makes two code words share a level (ties in the sort
    and in the mapping); a negative alpha reverses part of the order; code
    bytes with bits above q set must be treated as their low q bits."""
    q, g, out, n_in = 3, 64, 6, 640
    raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=77)
    P["alpha"][..., 1] = P["alpha"][..., 0]
    P["alpha"][::2, :, 2] *= -1
    dirty = (codes0 | np.uint8(0xF0)).astype(np.uint8)
    what, codes = C.gpu_fwd(raw, P, dirty, q, g, api.MAP_LOCAL_PERIODIC, 0, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, "ties")
    what, codes = C.gpu_fwd(raw, P, None, q, g, api.MAP_FULL, 0, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], None, g,
                                     O.MAP_FULL)
    C.assert_fwd_equal(what, codes, r_what, r_codes, "ties-full")
    gr = C.gpu_bwd(raw, P, dirty, Gup, q, g)
    ref, mass = C.oracle_bwd(W, P, codes0, Gup, g)
    C.assert_grads_close(gr, ref, mass, "ties-bwd")


@pytest.mark.parametrize("q,g", [(1, 32), (2, 64), (3, 128), (4, 128), (3, 256)])
def test_bwd_filter_boundary_within_ulps(q, g):
    """Every element within 4 ulps of the filter boundary |x - w~| = tau, some
    exactly on it: the filter decisions must be those of the IEEE quotient
    (a flipped decision moves ds of that element from 0 to -G Delta u / s or
    back, far outside the tolerance), whichever way the kernel forms x."""
    out, n_in = 24, 1024
    _, W0, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=700 + 10 * q + g, wdtype="f32")
    _, codes = O.quantize_fwd(W0, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                              O.MAP_LOCAL_PERIODIC, 0, 2)
    W, gap = C.boundary_weights(P, codes, g, seed=q + g)
    assert 0.3 < (gap > 0).mean() < 0.7 and (gap == 0).mean() > 0.02
    gr = C.gpu_bwd(W, P, codes, Gup, q, g)
    ref, mass = C.oracle_bwd(W, P, codes, Gup, g)
    C.assert_grads_close(gr, ref, mass, f"boundary q={q} g={g}")
    assert np.array_equal(gr["ds"] == 0, ref["ds"] == 0)          # the same elements filtered


def test_exact_decision_ties_are_bit_exact():
    """Dyadic weights and parameters put many elements exactly half-way
    between two levels; both sides must take the same (documented) choice."""
    q, g, out, n_in = 2, 32, 4, 128
    rng = np.random.default_rng(5)
    W = (rng.integers(-64, 65, (out, n_in)) / 256).astype(np.float32)
    Gr = n_in // g
    P = {"delta": np.full((out, Gr), 0.0625, np.float32), "zu": np.full((out, Gr), 1.5, np.float32),
         "s": np.ones((out, n_in), np.float32), "sr": np.ones(out, np.float32),
         "alpha": np.tile(np.array([1.0, 0.5], np.float32), (out, Gr, 1)), "zb": np.full((out, Gr), 1.5, np.float32)}
    what, codes = C.gpu_fwd(W, P, None, q, g, api.MAP_FULL, 0, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], None, g,
                                     O.MAP_FULL)
    x = W / 0.0625 + 1.5
    assert (np.abs(x - np.round(x)) == 0.5).sum() > 10        # genuine ties present
    C.assert_fwd_equal(what, codes, r_what, r_codes, "exact ties")


@pytest.mark.parametrize("q,g,n_in", [(1, 32, 1024), (2, 64, 1024), (3, 128, 2048), (4, 128, 1024), (3, 256, 1024)])
def test_remap_near_level_midpoints_is_bit_exact(q, g, n_in):
    """Every element within 4 ulps of the midpoint between its level and a
    rank neighbour (some exactly on it): the remap step's codes and W^ must
    be the oracle's bit for bit, whichever way the kernel forms x (the
    pipelined kernels decide from the reciprocal only inside a proven
    interval and fall back to the IEEE quotient and the three distances)."""
    out = 24
    _, W0, P, codes0, _ = C.make_inputs(out, n_in, q, g, seed=800 + 10 * q + g, wdtype="f32")
    W = C.midpoint_weights(P, codes0, g, seed=q + g)
    what, codes = C.gpu_fwd(W, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 0, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, f"midpoints q={q} g={g}")
    assert (r_codes != codes0).mean() > 0.05         # many decisions go to the neighbour


def test_deterministic_and_in_bounds():
    """Two identical calls give identical bits; outputs written into the middle
    of larger buffers leave the sentinel margins untouched."""
    q, g, out, n_in = 3, 128, 17, 1024
    raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=9)
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    pd = C.to_dev(P)
    pad = 64                                        # floats; keeps 16-byte alignment
    res = []
    for _ in range(2):
        big = torch.full((out * n_in + 2 * pad,), 12345.0, device=d)
        what = big[pad:pad + out * n_in].view(out, n_in)
        codes = torch.from_numpy(codes0).to(d)
        api.uq_quantize_fwd(Wd, q, g, pd, codes, what, api.MAP_LOCAL_PERIODIC, 0, 2)
        gbig = {k: torch.full((v.numel() + 2 * pad,), 777.0, device=d) for k, v in
                api.empty_grads(out, n_in, q, g, d).items()}
        gr = {k: gbig[k][pad:pad + v.numel()].view(v.shape) for k, v in api.empty_grads(out, n_in, q, g, d).items()}
        api.uq_quantize_bwd(Wd, q, g, pd, codes, torch.from_numpy(Gup).to(d), gr)
        torch.cuda.synchronize()
        assert torch.all(big[:pad] == 12345.0) and torch.all(big[-pad:] == 12345.0)
        for k in gbig:
            assert torch.all(gbig[k][:pad] == 777.0) and torch.all(gbig[k][-pad:] == 777.0), k
        res.append((C.host(what).copy(), C.host(codes).copy(), {k: C.host(v).copy() for k, v in gr.items()}))
    assert np.array_equal(res[0][0], res[1][0]) and np.array_equal(res[0][1], res[1][1])
    for k in res[0][2]:
        assert np.array_equal(res[0][2][k], res[1][2][k]), k


def test_side_stream_and_error_leaves_outputs_untouched():
    q, g, out, n_in = 3, 128, 8, 512
    raw, W, P, codes0, _ = C.make_inputs(out, n_in, q, g, seed=11)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 0, 2, stream=s)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, "stream")
    # a rejected call (q = 5) writes nothing
    d = C.dev()
    Wd = api.weights_tensor(raw, d)
    pd = C.to_dev(P)
    what = torch.full((out, n_in), 3.0, device=d)
    cd = torch.from_numpy(codes0).to(d)
    with pytest.raises(api.UQError) as ei:
        api.lib()  # loaded
        st = api.lib().uq_quantize_fwd(Wd.data_ptr(), api.W_BF16, out, n_in, 5, g,
                                       api._params(pd, out, n_in, 3, g, d), cd.data_ptr(), 1, 0, 2,
                                       what.data_ptr(), None)
        api._raise(st)
    assert ei.value.status == api.UQ_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert torch.all(what == 3.0) and torch.equal(cd.cpu(), torch.from_numpy(codes0))


def test_device_check_reports_no_timeouts_after_normal_work():
    """The pipelined kernels bound every wait; after ordinary calls no wait ran
    out and uq_check_device reports OK (and synchronises the stream)."""
    q, g, out, n_in = 3, 128, 64, 2048
    raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=21)
    what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 0, 2)
    gr = C.gpu_bwd(raw, P, codes, Gup, q, g)
    api.uq_check_device()
    assert api.uq_last_error() == ""


@pytest.mark.parametrize("n_in,g", [(512, 128), (2048, 64), (768, 32), (1536, 128), (384, 128)])
def test_pipelined_and_plain_paths_agree_across_shapes(n_in, g):
    """Rows that split into whole 512-element units (256 for g = 32) take the
    pipelined kernels, others the per-row kernels; both match the oracle,
    including short rows packed several to a block and a ragged last block."""
    q, out = 3, 21
    raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=n_in + g)
    what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 0, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, f"n_in={n_in} g={g}")
    gr = C.gpu_bwd(raw, P, codes, Gup, q, g)
    ref, mass = C.oracle_bwd(W, P, r_codes, Gup, g)
    C.assert_grads_close(gr, ref, mass, f"n_in={n_in} g={g}")


@pytest.mark.parametrize("n_in,g,q", [(4096, 128, 3), (2048, 128, 1), (3072, 128, 4), (1536, 128, 2),
                                      (1024, 32, 4), (768, 32, 3), (2048, 64, 2), (1536, 64, 3)])
def test_keep_step_items_of_several_units(n_in, g, q):
    """The keep step's work items are 4, 2 or 1 adjacent units of a row (by
    what divides the row's units): W^ = Delta (l(code) - z_U) bit-exact with
    the oracle for each item width, with rows packed several to a block and a
    ragged last block; the codes are untouched."""
    out = 37
    raw, W, P, codes0, _ = C.make_inputs(out, n_in, q, g, seed=7 * n_in + g + q)
    what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 1, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 1, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, f"keep n_in={n_in} g={g} q={q}")
    assert np.array_equal(codes, codes0)
    api.uq_check_device()
    assert api.uq_last_error() == ""


@pytest.mark.parametrize("n_in,g,q", [(512 * 36, 128, 3), (256 * 40, 32, 2), (512 * 33, 64, 4)])
def test_backward_of_long_rows(n_in, g, q):
    """Rows of 32 or more work units take the backward's branch-per-array
    gradient stores (the launcher's choice by row length); their gradients
    match the oracle like those of shorter rows, on a ragged row count."""
    out = 13
    raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=n_in + q)
    what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 0, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, f"n_in={n_in} g={g}")
    gr = C.gpu_bwd(raw, P, codes, Gup, q, g)
    ref, mass = C.oracle_bwd(W, P, r_codes, Gup, g)
    C.assert_grads_close(gr, ref, mass, f"n_in={n_in} g={g}")
    api.uq_check_device()
    assert api.uq_last_error() == ""


def test_host_buffer_apis_match_the_oracle():
    """HostStep and HostPipeline (pinned host buffers in, results back on the
    host) give the oracle's results; two independent problems are submitted
    alternately through the overlapped pipeline."""
    q, g, out, n_in = 3, 128, 48, 1024
    probs = []
    for seed in (31, 32):
        raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=seed)
        r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                         O.MAP_LOCAL_PERIODIC, 0, 2)
        ref, mass = C.oracle_bwd(W, P, r_codes, Gup, g)
        probs.append((raw, P, codes0, Gup, r_what, r_codes, ref, mass))
    hp = api.HostPipeline(out, n_in, q, g, torch.bfloat16, C.dev(), depth=2)
    bufs = []
    for raw, P, codes0, Gup, *_ in probs:
        hin, hout = hp.empty_host(pinned=True)
        hin["W"].copy_(torch.from_numpy(raw.view(np.int16)).view(torch.bfloat16))
        for k in api.PARAM_NAMES:
            hin[k].copy_(torch.from_numpy(P[k]))
        hin["codes"].copy_(torch.from_numpy(codes0))
        hin["dL_dWhat"].copy_(torch.from_numpy(Gup))
        bufs.append((hin, hout))
    for rep in range(3):
        for (hin, hout) in bufs:
            hp.submit(hin, hout, 0, 2)
    hp.synchronize()
    for (hin, hout), (raw, P, codes0, Gup, r_what, r_codes, ref, mass) in zip(bufs, probs):
        C.assert_fwd_equal(hout["W_hat"].numpy(), hout["codes"].numpy(), r_what, r_codes, "pipeline")
        C.assert_grads_close({k: hout[k].numpy() for k in api.GRAD_NAMES}, ref, mass, "pipeline")
    hs = api.HostStep(out, n_in, q, g, torch.bfloat16, C.dev())
    hin, hout = bufs[0][0], hs.empty_host(pinned=True)[1]
    hs.run(hin, hout, 0, 2)
    hs.stream.synchronize()
    raw, P, codes0, Gup, r_what, r_codes, ref, mass = probs[0]
    C.assert_fwd_equal(hout["W_hat"].numpy(), hout["codes"].numpy(), r_what, r_codes, "hoststep")


def test_quantizer_object_and_cuda_graph_capture():
    """The pre-validated Quantizer gives the same bits as the function API, and
    a step captured in a CUDA graph and replayed gives the same bits as eager
    calls (the launch path makes no call that breaks stream capture)."""
    q, g, out, n_in = 3, 128, 32, 1024
    raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=41)
    d = C.dev()

    def make():
        Wd = api.weights_tensor(raw, d)
        pd = C.to_dev(P)
        cd = torch.from_numpy(codes0).to(d)
        qz = api.Quantizer(Wd, q, g, pd, cd, torch.empty(out, n_in, device=d), torch.from_numpy(Gup).to(d),
                           api.empty_grads(out, n_in, q, g, d))
        return qz, cd

    qz, cd = make()
    qz.fwd(0, 2)
    qz.bwd()
    eager = (C.host(qz.keep[2]).copy(), C.host(cd).copy(), {k: C.host(v).copy() for k, v in qz.keep[4].items()})
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(eager[0], eager[1], r_what, r_codes, "quantizer")
    qz2, cd2 = make()
    qz2.fwd(1, 2)                                   # warm the launch path before capture
    torch.cuda.synchronize()
    cd2.copy_(torch.from_numpy(codes0))
    side = torch.cuda.Stream(d)
    cg = torch.cuda.CUDAGraph()
    with torch.cuda.graph(cg, stream=side):
        qz2.fwd(0, 2)
        qz2.bwd()
    cd2.copy_(torch.from_numpy(codes0))
    torch.cuda.synchronize()
    cg.replay()
    torch.cuda.synchronize()
    assert np.array_equal(C.host(qz2.keep[2]), eager[0]) and np.array_equal(C.host(cd2), eager[1])
    for k in eager[2]:
        assert np.array_equal(C.host(qz2.keep[4][k]), eager[2][k]), k


def test_bounded_wait_runs_out_reports_and_context_survives():
    """Failure path of the pipelined kernels without any fault: a wait on an
    mbarrier nothing arrives at gives up (bounded), the host reads the status
    through uq_check_device, the indicator is cleared, and normal work on the
    same context still matches the oracle."""
    api.uq_check_device()                               # start clean
    api.uq_selftest_wait_timeout()
    with pytest.raises(api.UQError) as ei:
        api.uq_check_device()
    assert ei.value.status == api.UQ_ERR_CUDA and "bounded wait" in str(ei.value)
    api.uq_check_device()                               # cleared
    q, g, out, n_in = 3, 128, 16, 1024
    raw, W, P, codes0, _ = C.make_inputs(out, n_in, q, g, seed=51)
    what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 0, 2)
    r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                     O.MAP_LOCAL_PERIODIC, 0, 2)
    C.assert_fwd_equal(what, codes, r_what, r_codes, "after timeout")


@pytest.mark.parametrize("g,n_in", [(512, 2048), (1024, 3072), (2048, 2048), (640, 1280)])
def test_large_groups_all_entry_points(g, n_in):
    """Groups of more than 128 elements, including one group per row
    (channel-wise, g = in): forward (all modes), backward, export and
    initialization on the general path."""
    q, out = 3, 9
    raw, W, P, codes0, Gup = C.make_inputs(out, n_in, q, g, seed=g + n_in, init_G=4, init_T=2)
    for mode, step in ((api.MAP_FULL, 0), (api.MAP_LOCAL_PERIODIC, 0), (api.MAP_LOCAL_PERIODIC, 1)):
        what, codes = C.gpu_fwd(raw, P, codes0 if mode else None, q, g, mode, step, 2)
        r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"],
                                         codes0 if mode else None, g, mode, step, 2)
        C.assert_fwd_equal(what, codes, r_what, r_codes, f"g={g} mode={mode} step={step}")
    gr = C.gpu_bwd(raw, P, codes0, Gup, q, g)
    ref, mass = C.oracle_bwd(W, P, codes0, Gup, g)
    C.assert_grads_close(gr, ref, mass, f"g={g}")
    planes, a_s, z_s = C.gpu_export(raw, P, codes0, q, g, api.EXPORT_REUSE_CODES)
    r_planes, r_as, r_zs, _ = O.export_bcq(W, P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g)
    assert np.array_equal(planes, r_planes) and np.array_equal(a_s, r_as) and np.array_equal(z_s, r_zs)
    Wd = api.weights_tensor(raw, C.dev())
    p = api.empty_params(out, n_in, q, g, C.dev())
    codes = torch.empty(out, n_in, dtype=torch.uint8, device=C.dev())
    api.uq_init_params(Wd, q, g, p, codes, G=4, T=2)
    ref_i, errs, chosen = O.unified_init(W, q, g, G=4, T=2, return_errors=True)
    got = {k: C.host(v) for k, v in p.items()}
    same = C.check_init(W, q, g, 4, api.CLIP_FIXED_MIN, got, C.host(codes), ref_i, errs, chosen, f"g={g}")
    assert same == 1.0, same


def test_maximum_row_length():
    """The longest supported row (in = 2^24) on both paths: g = 128 takes the
    pipelined kernels, g = 256 the general ones.  Parameters are a jittered
    uniform level grid (no initialization needed at this size)."""
    q, out, n_in = 2, 1, 1 << 24
    rng = np.random.default_rng(8)
    W32 = (rng.standard_normal((out, n_in)) * 0.02).astype(np.float32)
    raw, W = synth.bf16_round(W32)
    Gup = synth.upstream_grad(out, n_in, 1e-4, 8)
    for g in (128, 256):
        Gr = n_in // g
        P = {"delta": rng.uniform(0.008, 0.012, (out, Gr)).astype(np.float32),
             "zu": rng.uniform(1.3, 1.7, (out, Gr)).astype(np.float32),
             "s": rng.uniform(0.95, 1.05, (out, n_in)).astype(np.float32),
             "sr": np.ones(out, np.float32),
             "alpha": (np.array([1.0, 0.5]) * rng.uniform(0.9, 1.1, (out, Gr, q))).astype(np.float32),
             "zb": np.full((out, Gr), 1.5, np.float32)}
        _, codes0 = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], None, g, O.MAP_FULL)
        P["delta"] = (P["delta"] * np.float32(1.01)).astype(np.float32)
        what, codes = C.gpu_fwd(raw, P, codes0, q, g, api.MAP_LOCAL_PERIODIC, 0, 2)
        r_what, r_codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes0, g,
                                         O.MAP_LOCAL_PERIODIC, 0, 2)
        C.assert_fwd_equal(what, codes, r_what, r_codes, f"max row g={g}")
        gr = C.gpu_bwd(raw, P, r_codes, Gup, q, g)
        ref, mass = C.oracle_bwd(W, P, r_codes, Gup, g)
        C.assert_grads_close(gr, ref, mass, f"max row g={g}")
