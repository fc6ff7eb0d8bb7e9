"""Pins of the oracle's unified initialization (Algorithm 2), its clipping
strategies (App. E.2), the greedy start and the general alternating update
(Algorithm 3)."""

import json
import os

import numpy as np
import pytest

import oracle as O

F32 = np.float32
F64 = np.float64
GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_constants.json")))


def groups(seed, n=64, g=128, std=0.02):
    rng = np.random.default_rng(seed)
    return (rng.standard_t(4, (n, g)) * std / np.sqrt(2)).astype(F32)


@pytest.mark.parametrize("strategy", [O.CLIP_FIXED_MIN, O.CLIP_FIXED_MAX, O.CLIP_BALANCED])
@pytest.mark.parametrize("q", [2, 3, 4])
def test_clipping_closed_forms(strategy, q):
    w = groups(1)
    wm, wM = w.min(-1), w.max(-1)
    top = (1 << q) - 1
    for gamma in (F32(1) / F32(30), F32(17) / F32(30), F32(1)):
        d, zu = O.clip_params(wm, wM, gamma, q, strategy)
        assert np.allclose(d, gamma * (wM.astype(F64) - wm) / top, rtol=1e-6)
        if strategy == O.CLIP_FIXED_MIN:
            anchor, target = wm.astype(F64), 0.0             # T_F(w_m) = 0
        elif strategy == O.CLIP_FIXED_MAX:
            anchor, target = wM.astype(F64), float(top)      # T_F(w_M) = 2^q - 1
        else:
            anchor, target = gamma * wm.astype(F64), 0.0     # T_F(gamma w_m) = 0
        x = anchor / d + zu
        assert np.allclose(x, target, atol=1e-5 * top / gamma)


def test_greedy_single_bit_closed_form():
    """q = 1: the greedy code is sign(x - z_B) and alpha the mean |x - z_B|,
    which is also the least-squares alpha for that code."""
    x = groups(2) * F32(100)
    zb = np.full(x.shape[0], F32(0.5))
    alpha, codes = O.greedy_init(x, zb, 1)
    y = x.astype(F64) - 0.5
    assert np.array_equal(codes, (y >= 0).astype(np.int64))
    assert np.allclose(alpha[:, 0], np.abs(y).mean(-1), rtol=1e-7)


def test_greedy_residual_is_reduced():
    x = groups(3) * F32(100)
    zb = np.full(x.shape[0], F32(3.5))
    for q in (2, 3, 4):
        alpha, codes = O.greedy_init(x, zb, q)
        C = O.signs(q, F64)[codes]
        rec = (C * alpha.astype(F64)[:, None, :]).sum(-1) + 3.5
        y = x.astype(F64) - 3.5
        # every greedy bit removes energy: the residual norm is below |y|
        assert np.all(((x - rec) ** 2).sum(-1) < (y ** 2).sum(-1))
        # alphas are non-negative and non-increasing (each bit fits a smaller residual)
        assert np.all(alpha >= 0) and np.all(np.diff(alpha, axis=-1) <= 1e-7)


@pytest.mark.parametrize("q", [2, 3, 4])
def test_alpha_step_is_least_squares(q):
    """One alternating round: alpha = argmin ||x - z_B - C alpha|| for the greedy
    C, checked with numpy's SVD least-squares solver."""
    x = groups(4 + q) * F32(150) + F32(3.5)
    zb = np.full(x.shape[0], F32(3.5))
    _, codes0 = O.greedy_init(x, zb, q)
    alpha1, _, _ = O.general_alternating(x, zb, G=30, T=1, q=q)
    C = O.signs(q, F64)[codes0]
    for n in range(x.shape[0]):
        sol, *_ = np.linalg.lstsq(C[n], x[n].astype(F64) - 3.5, rcond=None)
        assert np.allclose(alpha1[n], sol, rtol=2e-6, atol=1e-6)


@pytest.mark.parametrize("G", [1, 30])
@pytest.mark.parametrize("q", [2, 3])
def test_alternating_error_non_increasing(G, q):
    """Each sub-step of Algorithm 3 minimises the error over its own variable,
    so the error after each round never grows (up to fp32 storage of alpha)."""
    x = groups(10 + q) * F32(150) + F32(3.5)
    zb = np.full(x.shape[0], F32(3.5))
    _, _, _, errs = O.general_alternating(x, zb, G=G, T=15, q=q, trace=True)
    errs = np.stack(errs)
    assert np.all(errs[1:] <= errs[:-1] * (1 + 1e-6) + 1e-9)


def test_zb_update_is_mean_residual():
    q = 3
    x = groups(20) * F32(150) + F32(3.0)
    zb = np.full(x.shape[0], F32(3.5))
    alpha, zb1, codes = O.general_alternating(x, zb, G=1, T=1, q=q)
    C = O.signs(q, F64)[codes]
    ref = (x.astype(F64) - (C * alpha.astype(F64)[:, None, :]).sum(-1)).mean(-1)
    assert np.allclose(zb1, ref, rtol=1e-6)
    # with G > 1, z_B is never moved
    _, zb30, _ = O.general_alternating(x, zb, G=30, T=5, q=q)
    assert np.array_equal(zb30, zb)


def _brute_quant_error(w, delta, zu, alpha, zb, q):
    """||w - D_R(M_B(T_F(w)))||^2 with s = s_r = 1 and a brute-force nearest
    over all sign vectors (fp64 levels)."""
    x = w.astype(F64) / delta[:, None] + zu[:, None]
    lv = alpha.astype(F64) @ O.signs(q, F64).T + zb.astype(F64)[:, None]
    idx = np.abs(x[:, :, None] - lv[:, None, :]).argmin(-1)
    what = delta[:, None].astype(F64) * (np.take_along_axis(lv, idx, -1) - zu[:, None])
    return ((w.astype(F64) - what) ** 2).sum(-1)


@pytest.mark.parametrize("clip", [O.CLIP_FIXED_MIN, O.CLIP_BALANCED])
def test_unified_init_keeps_the_best_candidate(clip):
    q, g, G = 3, 128, 8
    W = groups(30, n=24, g=g).reshape(6, 4 * g)
    res, errs, chosen = O.unified_init(W, q, g, G=G, T=6, clip=clip, return_errors=True)
    errs = errs.reshape(G, 6, 4)
    # Alg. 2 keeps the first strictly smallest error over the gamma grid
    assert np.array_equal(chosen, errs.argmin(0))
    # its stored error equals an independent brute-force re-evaluation
    w = W.reshape(-1, g)
    e_bf = _brute_quant_error(w, res["delta"].reshape(-1), res["zu"].reshape(-1),
                              res["alpha"].reshape(-1, q), res["zb"].reshape(-1), q)
    e_kept = np.take_along_axis(errs.reshape(G, -1), chosen.reshape(1, -1), 0)[0]
    assert np.allclose(e_bf, e_kept, rtol=1e-4)
    # every candidate's Delta follows the clipping rule for gamma_i = i / G
    i = chosen.reshape(-1) + 1
    gamma = i.astype(F32) / F32(G)
    d_ref = gamma * (w.max(-1) - w.min(-1)) / F32((1 << q) - 1)
    assert np.allclose(res["delta"].reshape(-1), d_ref, rtol=1e-6)
    # s = 1, s_r = 1, z_B untouched for G > 1 (Algorithm 2 sets s and s_r to 1; Algorithm 3 moves z_B only when G = 1)
    assert np.all(res["s"] == 1) and np.all(res["sr"] == 1)
    assert np.all(res["zb"] == GOLD["z_B_initial"]["k3"])
    # initial codes are the full mapping under the kept parameters
    _, codes = O.quantize_fwd(W, res["s"], res["sr"], res["delta"], res["zu"], res["alpha"], res["zb"],
                              None, g, mode=O.MAP_FULL)
    assert np.array_equal(codes, res["codes"])


def test_unified_init_beats_plain_grid_and_handles_constant_group():
    q, g = 3, 128
    W = groups(40, n=8, g=g).reshape(8, g)
    W[3] = F32(0.0123)                        # a constant group (w_M = w_m)
    res = O.unified_init(W, q, g, G=30, T=15)
    for k in ("delta", "zu", "alpha", "zb"):
        assert np.all(np.isfinite(res[k])), k
    what, _ = O.quantize_fwd(W, res["s"], res["sr"], res["delta"], res["zu"], res["alpha"], res["zb"],
                             res["codes"], g, mode=O.MAP_LOCAL_PERIODIC, step=1)
    assert np.all(np.isfinite(what))
    # on the uniform grid (alpha = 2^(q-1-j), same Delta, z_U) the learned BCQ
    # levels cannot be worse than RTN: the grid is one of the candidates the
    # least-squares alpha step improves on
    rtn_err = ((W.astype(F64) - O.rtn(W, res["delta"][:, 0], res["zu"][:, 0], q)) ** 2).sum(-1)
    bcq_err = ((W.astype(F64) - what) ** 2).sum(-1)
    ok = np.arange(8) != 3
    assert np.all(bcq_err[ok] <= rtn_err[ok] * 1.05)


def test_hyperparameter_defaults_follow_paper():
    hp = GOLD["hyperparameters"]
    from paper_2506_03781_gb300 import synth
    wl = synth.WORKLOADS["mlp14336x4096_bf16"]
    assert wl.T == hp["alternating_iterations_T"]
    assert wl.p == hp["remapping_period_p"]
    assert wl.G in hp["grid_search_iterations_G"]
    assert hp["clipping_strategy"] == "Fixed-minimum" and O.CLIP_FIXED_MIN == 0


@pytest.mark.parametrize("q", [2, 3, 4])
def test_singular_gram_matrix_leaves_alpha_unchanged(q):
    """Reading R11 for the alpha step of Algorithm 3: when C^T C is exactly
    singular, alpha keeps its value from before the round.  A group whose
    transformed weights all equal z_B - a makes the greedy start pick
    c_1 = -1 everywhere with alpha_1 = a, after which the residual is exactly
    zero and every further bit is +1 with alpha_j = 0: the columns of C are
    +-1 multiples of each other, so C^T C is singular.  Its neighbour in the
    same batch (ordinary weights) is regular and must move.  A pseudo-inverse
    solve, a reset of alpha or an inverted test would each change the
    singular group's alpha and fail here (checked below for the
    pseudo-inverse)."""
    g, a = 64, F32(0.75)
    zb = np.full(2, F32(((1 << q) - 1) / 2), F32)
    x = np.empty((2, g), F32)
    x[0] = zb[0] - a
    x[1] = groups(90, n=1, g=g)[0] * F32(100) + zb[1]
    a0, c0 = O.greedy_init(x, zb, q)
    assert np.array_equal(a0[0], np.array([a] + [0.0] * (q - 1), F32))
    C = O.signs(q, F64)[c0[0]]
    assert np.linalg.matrix_rank(C.T @ C) < q                      # singular (integer Gram matrix)
    a1, zb1, c1 = O.general_alternating(x, zb, 2, 1, q)
    assert np.array_equal(a1[0], a0[0])                           # bit-identical: left unchanged
    assert not np.array_equal(a1[1], a0[1])                       # the regular neighbour moved
    # the minimum-norm least-squares alpha differs from the kept one
    pinv = np.linalg.pinv(C) @ (x[0].astype(F64) - zb[0])
    assert not np.allclose(pinv, a0[0].astype(F64))
    # later rounds stay singular and keep alpha: T = 15 ends where the greedy start did
    a15, _, c15 = O.general_alternating(x, zb, 2, 15, q)
    assert np.array_equal(a15[0], a0[0])


@pytest.mark.parametrize("clip", [O.CLIP_FIXED_MIN, O.CLIP_FIXED_MAX, O.CLIP_BALANCED])
def test_constant_group_initializes_to_the_kept_greedy_alpha(clip):
    """A constant weight group (w_M = w_m): T_F maps every weight to the same
    x, so the greedy start takes alpha_1 = |x - z_B| with one sign for every
    weight, leaves an exactly zero residual, and sets every further bit to +1
    with alpha_j = 0.  The Gram matrix is singular in every round, so the kept
    alpha is the greedy one, bit for bit, and every weight takes one code
    word.  Under Fixed-minimum, x is exactly 0 (u and -z_U are the same
    quotient), so alpha = (z_B, 0, ..., 0) = (3.5, 0, 0) and the code word is
    0 (c_1 = -1; ties between equal levels go to the smaller code word)."""
    q, g = 3, 128
    W = groups(41, n=4, g=g).reshape(4, g)
    W[1] = F32(0.0123)
    W[2] = F32(-0.5)
    res = O.unified_init(W, q, g, G=5, T=4, clip=clip)
    for r in (1, 2):
        x, _ = O.transform_F(W[r][None], np.ones((1, g), F32), res["delta"][r], res["zu"][r], np.ones(1, F32))
        assert np.all(x == x[0, 0])
        r0 = np.abs(x[0, 0] - F32(3.5))
        assert np.array_equal(res["alpha"][r, 0], np.array([r0, 0.0, 0.0], F32)), res["alpha"][r]
        assert np.all(res["codes"][r] == res["codes"][r, 0])
        assert res["zb"][r, 0] == F32(3.5)
        if clip == O.CLIP_FIXED_MIN:
            assert x[0, 0] == 0 and r0 == F32(3.5) and np.all(res["codes"][r] == 0)


def test_init_error_is_the_quantizer_error_under_full_mapping():
    """init_error equals ||w - w^||^2 with w^ from quantize_fwd (full mapping,
    s = s_r = 1) -- a different code path through the same definitions --
    and is the error unified_init keeps for its chosen candidate."""
    q, g = 3, 64
    W = groups(42, n=6, g=g * 4).reshape(6, g * 4)
    res, errs, chosen = O.unified_init(W, q, g, G=6, T=3, return_errors=True)
    NG = W.size // g
    e = O.init_error(W.reshape(NG, g), res["delta"].reshape(-1), res["zu"].reshape(-1),
                     res["alpha"].reshape(NG, q), res["zb"].reshape(-1))
    what, _ = O.quantize_fwd(W, res["s"], res["sr"], res["delta"], res["zu"], res["alpha"], res["zb"], None, g,
                             mode=O.MAP_FULL)
    direct = ((W.astype(F64) - what.astype(F64)) ** 2).reshape(NG, g).sum(-1)
    assert np.array_equal(e, direct)
    assert np.array_equal(e, errs[chosen.reshape(-1), np.arange(NG)])
    # the kept candidate is the first strictly smallest error
    assert np.all(errs[chosen.reshape(-1), np.arange(NG)] == errs.min(0))
    first = np.argmax(errs == errs.min(0)[None], axis=0)
    assert np.array_equal(first, chosen.reshape(-1))
