"""Pins of the oracle's optimisation step (SGD on Theta_IF, then the forward
of the next step; the inner loop of Algorithm 1).

The update is pinned by what gradient descent must do to the surrogate loss
of the backward pins (written from the forward definitions only):

    S(Theta) = sum_i G_i * w^_i(Theta)   (codes and filter frozen at Theta_0)

One step with learning rate eta on one parameter set moves S by
-eta * ||dS/dtheta||^2 to first order, so the measured change, divided by
that prediction, must be 1 up to O(eta) -- a wrong sign, a wrong learning
rate for the set, or a parameter left out fails it.  The learning rates and
the split Theta_F = {Delta, z_U, s, s_r}, Theta_B = {alpha, z_B} come from
the paper's hyperparameter table (tests/golden/paper_constants.json).
"""

import json
import os

import numpy as np
import pytest

import oracle as O
from tests.test_oracle_bwd import frozen_state, make_problem, surrogate

F32 = np.float32
F64 = np.float64

HERE = os.path.dirname(__file__)
with open(os.path.join(HERE, "golden", "paper_constants.json")) as fh:
    HYP = json.load(fh)["hyperparameters"]

THETA_F = ("delta", "zu", "s", "sr")
THETA_B = ("alpha", "zb")
GRAD = {"delta": "ddelta", "zu": "dzu", "s": "ds", "sr": "dsr", "alpha": "dalpha", "zb": "dzb"}
PARAMS = ("s", "sr", "delta", "zu", "alpha", "zb")


def test_learning_rates_are_the_papers():
    assert O.LR_F == HYP["lr_theta_F"] == 0.005
    assert O.LR_B == HYP["lr_theta_B"] == 0.0005


def _only(grads, name):
    return {k: (v if k == GRAD[name] else np.zeros_like(v)) for k, v in grads.items()}


@pytest.mark.parametrize("q", [1, 2, 3, 4])
@pytest.mark.parametrize("name", THETA_F + THETA_B)
def test_sgd_step_descends_the_surrogate_per_parameter(q, name):
    pb = make_problem(300 + q, q)
    P0, x0, f, margin = frozen_state(pb, q)
    assert margin.min() > 1e-4
    grads = O.quantize_bwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                           pb["codes"], pb["Gup"], pb["g"])
    # Table-8 learning rates scaled down together (their ratio kept) so the
    # first-order prediction holds; still far above the fp32 storage step.
    scale = 1e-3
    lr = (HYP["lr_theta_F"] if name in THETA_F else HYP["lr_theta_B"]) * scale
    new = O.sgd_update(pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"], _only(grads, name),
                       lr_F=HYP["lr_theta_F"] * scale, lr_B=HYP["lr_theta_B"] * scale)
    for other in PARAMS:
        if other != name:
            assert np.array_equal(new[other], pb[other]), other
    P1 = dict(P0)
    P1[name] = new[name].astype(F64)
    args = (x0, pb["codes"], pb["W"], pb["Gup"], pb["g"], q)
    dS = surrogate(P1, f, *args) - surrogate(P0, f, *args)
    predicted = -lr * float((grads[GRAD[name]] ** 2).sum())
    assert predicted < 0
    # fp32 storage of the moved parameter: at most half an ulp per entry
    ulp_err = 0.5 * np.spacing(np.abs(new[name]).astype(F32)).astype(F64)
    slack = float((np.abs(grads[GRAD[name]]) * ulp_err).sum())
    assert abs(dS - predicted) <= 0.02 * abs(predicted) + 2 * slack, (dS, predicted, slack)


@pytest.mark.parametrize("q", [2, 3])
def test_full_step_descends_with_the_papers_split(q):
    """All six parameters at once: the decrease is the sum of the per-set
    predictions with Theta_F at lr_F and Theta_B at lr_B (swapping the two
    rates changes the prediction by far more than the tolerance)."""
    pb = make_problem(400 + q, q)
    P0, x0, f, _ = frozen_state(pb, q)
    grads = O.quantize_bwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                           pb["codes"], pb["Gup"], pb["g"])
    scale = 1e-3
    lrF, lrB = HYP["lr_theta_F"] * scale, HYP["lr_theta_B"] * scale
    new = O.sgd_update(pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"], grads, lrF, lrB)
    P1 = {k: new[k].astype(F64) for k in PARAMS}
    args = (x0, pb["codes"], pb["W"], pb["Gup"], pb["g"], q)
    dS = surrogate(P1, f, *args) - surrogate(P0, f, *args)
    nF = sum(float((grads[GRAD[k]] ** 2).sum()) for k in THETA_F)
    nB = sum(float((grads[GRAD[k]] ** 2).sum()) for k in THETA_B)
    predicted = -(lrF * nF + lrB * nB)
    swapped = -(lrB * nF + lrF * nB)
    assert abs(dS - predicted) <= 0.02 * abs(predicted)
    assert abs(swapped - predicted) > 0.1 * abs(predicted)


def _step_inputs(seed, q, g=32, out=3, n_in=96):
    pb = make_problem(seed, q, out=out, n_in=n_in, g=g)
    return pb


@pytest.mark.parametrize("q", [1, 3])
def test_zero_gradient_step_is_the_next_forward(q):
    pb = _step_inputs(500 + q, q)
    zero = np.zeros_like(pb["Gup"])
    for mode in (O.MAP_FULL, O.MAP_LOCAL_PERIODIC):
        for t in (0, 1, 2):
            new, c1, w1 = O.train_step(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                                       pb["codes"], zero, pb["g"], t, mode=mode, p=2)
            for k in PARAMS:
                assert np.array_equal(new[k], pb[k]), k
            w_ref, c_ref = O.quantize_fwd(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"],
                                          pb["zb"], pb["codes"], pb["g"], mode, t + 1, 2)
            assert np.array_equal(c1, c_ref) and np.array_equal(w1, w_ref)


def test_keep_step_keeps_codes_and_uses_updated_levels():
    """Under M*_B with p = 2 the forward after step 0 (step 1) keeps every
    code word; W^ is D_R(l(code)) with the UPDATED alpha, z_B, Delta, z_U."""
    q = 3
    pb = _step_inputs(600, q)
    new, c1, w1 = O.train_step(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                               pb["codes"], pb["Gup"], pb["g"], 0, mode=O.MAP_LOCAL_PERIODIC, p=2)
    assert np.array_equal(c1, pb["codes"])
    out, n_in = pb["W"].shape
    g = pb["g"]
    cg = c1.reshape(out, -1, g).astype(np.int64)
    sg = np.where(((cg[..., None] >> np.arange(q)) & 1) == 1, F32(1), F32(-1))
    lv = np.zeros(cg.shape, F32)
    for j in range(q):                      # fp32, summed j = 1..q, then z_B
        lv = (lv + sg[..., j] * new["alpha"][..., None, j]).astype(F32)
    lv = (lv + new["zb"][..., None]).astype(F32)
    expect = (new["delta"][..., None] * (lv - new["zu"][..., None])).astype(F32)
    assert np.array_equal(w1, expect.reshape(out, n_in))
    # and the parameters did move
    assert not np.array_equal(new["alpha"], pb["alpha"])


def test_remap_step_moves_codes_by_at_most_one_rank():
    """Step 1 -> 2 remaps locally: every code moves to a level-order
    neighbour at most (the locality of Algorithm 4)."""
    q = 3
    pb = _step_inputs(700, q, g=32, out=4, n_in=128)
    big = (pb["Gup"] * 50).astype(F32)        # a large step, so that codes move
    new, c1, _ = O.train_step(pb["W"], pb["s"], pb["sr"], pb["delta"], pb["zu"], pb["alpha"], pb["zb"],
                              pb["codes"], big, pb["g"], 1, mode=O.MAP_LOCAL_PERIODIC, p=2)
    out, n_in = pb["W"].shape
    _, _, roc = O.sorted_levels(O.levels(new["alpha"], new["zb"]))
    g = pb["g"]
    r0 = np.take_along_axis(roc, pb["codes"].reshape(out, -1, g).astype(np.int64), -1)
    r1 = np.take_along_axis(roc, c1.reshape(out, -1, g).astype(np.int64), -1)
    assert np.abs(r1 - r0).max() <= 1
    assert (r1 != r0).any()
