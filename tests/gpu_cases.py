"""Helpers for the GPU parity tests: run the CUDA library through the C ABI
and the CPU oracle on identical seeded inputs, and compare.

Comparison rules (derived from the arithmetic; see the design notes):
* codes and bit-planes: bit-exact (both sides take every decision in fp32
  with the same operations and the same tie rules);
* w^ and alpha*, z_B*: bit-exact where the codes agree (same fp32 ops);
  the stated bound is 1e-6 relative to max(|ref|, Delta max|alpha|);
* gradient sums: |gpu - oracle| <= 1e-4 * (sum of |terms|), the L1 mass of
  the reduction (fp32 accumulation error is at most ~n u times that mass);
* ds: |gpu - oracle| <= 1e-4 * max(|oracle|, 1e-6 max|ds|).
"""

from __future__ import annotations

import numpy as np
import torch

import oracle as O
from paper_2506_03781_gb300 import api, synth

F32 = np.float32
PKEYS = ("delta", "zu", "s", "sr", "alpha", "zb")
GTOL = 1e-4


def dev():
    return torch.device("cuda:0")


def to_dev(P, d=None):
    d = d or dev()
    return {k: torch.from_numpy(np.ascontiguousarray(P[k], F32)).to(d) for k in PKEYS}


def host(t):
    torch.cuda.synchronize()
    return t.cpu().numpy()


def make_inputs(out, n_in, q, g, seed, wdtype="bf16", std=0.02, init_G=6, init_T=3, eps=0.01):
    """Weights, oracle-initialised (then jittered) parameters, codes and dL/dW^."""
    rng = np.random.default_rng(seed)
    W32 = (rng.standard_t(4, (out, n_in)) * std / np.sqrt(2)).astype(F32)
    if wdtype == "bf16":
        raw, W = synth.bf16_round(W32)
    else:
        raw, W = W32, W32
    init = O.unified_init(W, q, g, G=init_G, T=init_T)
    fac = synth.perturb_factors(synth.param_shapes(out, n_in, g, q), eps, seed)
    P = synth.jitter({k: init[k] for k in PKEYS}, fac)
    Gup = synth.upstream_grad(out, n_in, 1e-4, seed)
    return raw, W, P, init["codes"], Gup


def gpu_fwd(raw, P, codes, q, g, mode, step, p, stream=None):
    out, n_in = raw.shape
    Wd = api.weights_tensor(raw, dev())
    pd = to_dev(P)
    cd = torch.from_numpy(np.ascontiguousarray(codes)).to(dev()) if codes is not None else \
        torch.zeros(out, n_in, dtype=torch.uint8, device=dev())
    what = torch.empty(out, n_in, dtype=torch.float32, device=dev())
    api.uq_quantize_fwd(Wd, q, g, pd, cd, what, mode, step, p, stream=stream)
    return host(what), host(cd)


def gpu_bwd(raw, P, codes, Gup, q, g):
    out, n_in = raw.shape
    Wd = api.weights_tensor(raw, dev())
    gr = api.empty_grads(out, n_in, q, g, dev())
    api.uq_quantize_bwd(Wd, q, g, to_dev(P), torch.from_numpy(np.ascontiguousarray(codes)).to(dev()),
                        torch.from_numpy(np.ascontiguousarray(Gup, F32)).to(dev()), gr)
    return {k: host(v) for k, v in gr.items()}


def gpu_export(raw, P, codes, q, g, mode):
    out, n_in = raw.shape
    Wd = api.weights_tensor(raw, dev())
    planes = torch.full((q, out, n_in // 32), -1, dtype=torch.int32, device=dev())
    a_s = torch.empty(out, n_in // g, q, dtype=torch.float32, device=dev())
    z_s = torch.empty(out, n_in // g, dtype=torch.float32, device=dev())
    cd = torch.from_numpy(np.ascontiguousarray(codes)).to(dev()) if codes is not None else None
    api.uq_export_bcq(Wd, q, g, to_dev(P), cd, planes, a_s, z_s, mode)
    return host(planes).view(np.uint32), host(a_s), host(z_s)


def assert_fwd_equal(what, codes, r_what, r_codes, label=""):
    n_code = int((codes != r_codes).sum())
    assert n_code == 0, f"{label}: {n_code} code mismatches of {codes.size}"
    n_w = int((what != r_what).sum())
    assert n_w == 0, f"{label}: {n_w} w_hat mismatches (max abs {np.abs(what - r_what).max()})"


def assert_grads_close(gr, ref, mass, label=""):
    for k in ("ddelta", "dzu", "dzb", "dalpha", "dsr"):
        err = np.abs(gr[k].astype(np.float64) - ref[k])
        bad = err > GTOL * mass[k] + 1e-30
        assert not bad.any(), (f"{label}: {k}: {int(bad.sum())} outside tol; worst ratio "
                               f"{(err / (mass[k] + 1e-30)).max():.3e}")
    ds_ref = ref["ds"]
    floor = 1e-6 * np.abs(ds_ref).max()
    err = np.abs(gr["ds"].astype(np.float64) - ds_ref)
    bad = err > GTOL * np.maximum(np.abs(ds_ref), floor)
    assert not bad.any(), f"{label}: ds: {int(bad.sum())} outside tol"


def oracle_bwd(W, P, codes, Gup, g):
    args = (W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, Gup, g)
    return O.quantize_bwd(*args), O.bwd_l1_mass(*args)


def boundary_weights(P, codes, g, seed, ulps=4):
    """fp32 weights that put every element within `ulps` ulps of the filter
    boundary |x - w~| = tau (App. C.1): x is aimed at w~ +- tau (1 + k 2^-23),
    k uniform in [-ulps, ulps], and w = (x - z_U) Delta s s_r in fp64, so
    roughly half the elements are filtered and some sit exactly on the
    boundary.  Built from the oracle's levels; the codes are the given ones."""
    out, n_in = P["s"].shape
    Gr = n_in // g
    lv = O.levels(P["alpha"], P["zb"])
    m = O.reconstruct(np.asarray(codes).reshape(out, Gr, g).astype(np.int64), lv).astype(np.float64)
    tau = np.abs(np.asarray(P["alpha"], np.float64)).min(-1)[..., None]
    rng = np.random.default_rng(seed)
    x = m + rng.choice([-1.0, 1.0], m.shape) * tau * (1.0 + rng.integers(-ulps, ulps + 1, m.shape) * 2.0 ** -23)
    den = (np.asarray(P["delta"], np.float64)[..., None] * np.asarray(P["s"], np.float64).reshape(out, Gr, g)
           * np.asarray(P["sr"], np.float64)[:, None, None])
    W = ((x - np.asarray(P["zu"], np.float64)[..., None]) * den).astype(F32).reshape(out, n_in)
    x32, _ = O.transform_F(W.reshape(out, Gr, g), P["s"].reshape(out, Gr, g), P["delta"], P["zu"], P["sr"][:, None])
    gap = np.abs(x32 - O.reconstruct(np.asarray(codes).reshape(out, Gr, g).astype(np.int64), lv)) - tau
    return W, gap.reshape(out, n_in)


def slice_rows(P, rows):
    return {k: np.ascontiguousarray(np.asarray(v)[rows]) for k, v in P.items()}


def check_init(W, q, g, G, clip, got, got_codes, ref, errs, chosen, label=""):
    """Unified initialization (Algorithm 2 / Algorithm 3) on the GPU against
    the oracle, with every group checked (reading R10/R11 criteria):

    * the GPU's (Delta, z_U) must be one of the oracle's clipping candidates
      (App. E.2) for gamma_i = i/G, which identifies the GPU's gamma index;
    * the GPU's error e' -- recomputed by the oracle's own formula
      (oracle.init_error) from the GPU's parameters -- must be within 1e-5
      relative of the oracle's kept error;
    * the gamma index must be the oracle's, except where the oracle's own
      error for the GPU's candidate is within 1e-6 relative of its best (a
      near-tie between candidates; counted and printed);
    * the GPU's codes must be, bit for bit, the full mapping of T_F(w)
      (s = s_r = 1) under the GPU's own parameters, in every group, so groups
      with identical parameters have identical codes.

    got: dict of the GPU's per-group parameters shaped like ref's; errs
    [G, NG] and chosen [out, Gr] from oracle.unified_init(return_errors).
    Returns the fraction of groups whose parameters are bit-identical."""
    W = np.asarray(W, F32)
    out, n_in = W.shape
    NG = out * (n_in // g)
    w = W.reshape(NG, g)
    d_gpu, z_gpu = got["delta"].reshape(NG), got["zu"].reshape(NG)
    a_gpu, zb_gpu = got["alpha"].reshape(NG, q), got["zb"].reshape(NG)
    same = (d_gpu == ref["delta"].reshape(NG)) & (z_gpu == ref["zu"].reshape(NG)) & \
        (zb_gpu == ref["zb"].reshape(NG)) & (a_gpu == ref["alpha"].reshape(NG, q)).all(-1)
    wm, wM = w.min(-1), w.max(-1)
    match = np.zeros((G, NG), bool)
    for i in range(1, G + 1):
        d_c, z_c = O.clip_params(wm, wM, F32(i) / F32(G), q, clip)
        match[i - 1] = (d_c == d_gpu) & (z_c == z_gpu)
    assert match.any(0).all(), f"{label}: {int((~match.any(0)).sum())} groups whose Delta, z_U is no candidate"
    gi = match.argmax(0)
    ch = np.asarray(chosen).reshape(NG)
    cols = np.arange(NG)
    e_best = errs[ch, cols]
    e_gpu = O.init_error(w, d_gpu, z_gpu, a_gpu, zb_gpu)
    rel = np.abs(e_gpu - e_best) / np.maximum(e_best, 1e-300)
    assert (rel <= 1e-5).all(), f"{label}: {int((rel > 1e-5).sum())} groups with e' off by more than 1e-5 " \
                                f"(worst {rel.max():.3e})"
    moved = gi != ch
    near = np.abs(errs[gi, cols] - e_best) <= 1e-6 * e_best
    assert (near | ~moved).all(), f"{label}: {int((moved & ~near).sum())} groups took another gamma without a near-tie"
    x, _ = O.transform_F(w, np.ones((NG, g), F32), d_gpu, z_gpu, np.ones(NG, F32))
    srt, cor, _ = O.sorted_levels(O.levels(a_gpu, zb_gpu))
    want = O.map_full(x, srt, cor)
    bad = np.asarray(got_codes).reshape(NG, g).astype(np.int64) != want
    assert not bad.any(), f"{label}: {int(bad.sum())} init codes are not the full mapping of the GPU's parameters"
    print(f"init {label}: {same.mean():.6f} of {NG} groups bit-identical, {int(moved.sum())} near-tie gamma "
          f"choices, worst e' rel diff {rel.max():.2e}")
    return same.mean()


def midpoint_targets(alpha, zb, codes, g, seed, ulps=4):
    """fp64 targets x [out, in/g, g]: for each element, the midpoint between its
    level and one of its two rank neighbours (Algorithm 4's d - 1, d + 1),
    moved by up to `ulps` relative ulps (a tenth exactly on it)."""
    q = np.asarray(alpha).shape[-1]
    L = 1 << q
    out, Gr = np.asarray(zb).shape
    lv = O.levels(alpha, zb)
    srt, _, rank_of_code = O.sorted_levels(lv)
    c = (np.asarray(codes).reshape(out, Gr, g).astype(np.int64)) & (L - 1)
    r = np.take_along_axis(rank_of_code, c, axis=-1)
    rng = np.random.default_rng(seed)
    rn = np.clip(r + rng.choice([-1, 1], r.shape), 0, L - 1)
    l_c = np.take_along_axis(lv, c, axis=-1).astype(np.float64)
    l_n = np.take_along_axis(srt, rn, axis=-1).astype(np.float64)
    mid = 0.5 * (l_c + l_n)
    k = rng.integers(-ulps, ulps + 1, mid.shape)
    k[rng.random(mid.shape) < 0.1] = 0
    return mid + k * 2.0 ** -23 * np.abs(mid)


def midpoint_weights(P, codes, g, seed, ulps=4):
    """fp32 weights whose x = T_F(w) lies within `ulps` relative ulps of the
    midpoint between each element's level and one of its two rank neighbours
    (Algorithm 4's candidates d - 1, d + 1), about a tenth of them exactly on
    it, so every local remap decision is taken by a hair or by the tie rule.
    Built from the oracle's levels and sorted order; codes are the given ones."""
    out, n_in = P["s"].shape
    Gr = n_in // g
    q = P["alpha"].shape[-1]
    L = 1 << q
    lv = O.levels(P["alpha"], P["zb"])
    srt, _, rank_of_code = O.sorted_levels(lv)
    c = (np.asarray(codes).reshape(out, Gr, g).astype(np.int64)) & (L - 1)
    r = np.take_along_axis(rank_of_code, c, axis=-1)
    rng = np.random.default_rng(seed)
    rn = np.clip(r + rng.choice([-1, 1], r.shape), 0, L - 1)
    l_c = np.take_along_axis(lv, c, axis=-1).astype(np.float64)
    l_n = np.take_along_axis(srt, rn, axis=-1).astype(np.float64)
    mid = 0.5 * (l_c + l_n)
    k = rng.integers(-ulps, ulps + 1, mid.shape)
    k[rng.random(mid.shape) < 0.1] = 0
    x = mid + k * 2.0 ** -23 * np.abs(mid)
    den = (np.asarray(P["delta"], np.float64)[..., None] * np.asarray(P["s"], np.float64).reshape(out, Gr, g)
           * np.asarray(P["sr"], np.float64)[:, None, None])
    return ((x - np.asarray(P["zu"], np.float64)[..., None]) * den).astype(F32).reshape(out, n_in)


def omni_midpoint_weights(W, P, codes, g, seed, ulps=4):
    """OmniQuant's maps: weights whose x = w / Delta_O + z_O lies at level
    midpoints (midpoint_targets).  Every group keeps its smallest and largest
    weight, so Delta_O and z_O (functions of w_m, w_M) are unchanged; the
    other weights move to a target when it lies strictly inside (w_m, w_M)."""
    W = np.asarray(W, F32)
    out, n_in = W.shape
    Gr = n_in // g
    d, zo = O.omni_params(W, P["beta"], P["gamma"], P["alpha"].shape[-1], g)
    x = midpoint_targets(P["alpha"], P["zb"], codes, g, seed, ulps)
    Wg = W.reshape(out, Gr, g).copy()
    cand = ((x - np.asarray(zo, np.float64)[..., None]) * np.asarray(d, np.float64)[..., None]).astype(F32)
    lo, hi = Wg.min(-1, keepdims=True), Wg.max(-1, keepdims=True)
    ok = (cand > lo) & (cand < hi) & (Wg != lo) & (Wg != hi)    # the extremes stay
    Wn = np.where(ok, cand, Wg).reshape(out, n_in)
    d2, z2 = O.omni_params(Wn, P["beta"], P["gamma"], P["alpha"].shape[-1], g)
    assert np.array_equal(d2, d) and np.array_equal(z2, zo)
    return Wn, ok.mean()


def awq_midpoint_weights(P, codes, g, seed, ulps=4):
    """AWQ's maps: weights whose x = (w s_A) / Delta_A + z_A lies at level
    midpoints (midpoint_targets)."""
    out, Gr = np.asarray(P["zb"]).shape
    n_in = Gr * g
    x = midpoint_targets(P["alpha"], P["zb"], codes, g, seed, ulps)
    w = ((x - np.asarray(P["za"], np.float64)[..., None]) * np.asarray(P["delta"], np.float64)[..., None]
         / np.asarray(P["sa"], np.float64).reshape(1, Gr, g))
    return w.astype(F32).reshape(out, n_in)
