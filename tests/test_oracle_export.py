"""Pins of the oracle's export: Theorem 1, Eq. 4 and the bit-plane layout."""

import json
import os
from fractions import Fraction

import numpy as np
import pytest

import oracle as O

F32 = np.float32
F64 = np.float64
GOLD = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "paper_constants.json")))


def unpack_bitplanes(planes, n_in):
    q, out, words = planes.shape
    bits = (planes[..., None] >> np.arange(32, dtype=np.uint32)) & 1      # [q, out, words, 32]
    bits = bits.reshape(q, out, words * 32)[..., :n_in]
    return (bits.astype(np.uint32) << np.arange(q, dtype=np.uint32)[:, None, None]).sum(0).astype(np.uint8)


def random_params(seed, q, out=6, n_in=256, g=64):
    rng = np.random.default_rng(seed)
    Gr = n_in // g
    return dict(
        W=(rng.standard_normal((out, n_in)) * 0.02).astype(F32),
        s=rng.uniform(0.9, 1.1, (out, n_in)).astype(F32),
        sr=rng.uniform(0.9, 1.1, out).astype(F32),
        delta=rng.uniform(0.004, 0.012, (out, Gr)).astype(F32),
        zu=rng.uniform(2, 5, (out, Gr)).astype(F32),
        alpha=(rng.uniform(0.2, 2.0, (out, Gr, q)) * rng.choice([-1, 1], (out, Gr, q))).astype(F32),
        zb=rng.uniform(1, 6, (out, Gr)).astype(F32),
        g=g,
    )


@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_unify_closed_form_and_identity_exact(q):
    """Theorem 1 (proof, App. E.5): D_R(R_B(C; Theta_B); Theta_R) = R_B(C; Theta_B*)
    with alpha* = Delta alpha, z_B* = Delta (z_B - z_U), for every code C.
    Checked in exact rational arithmetic on the oracle's fp32 outputs: the
    only difference allowed is the fp32 rounding of alpha* and z_B*."""
    P = random_params(500 + q, q, out=2, n_in=128, g=64)
    a_star, z_star = O.unify(P["delta"], P["zu"], P["alpha"], P["zb"])
    assert np.array_equal(a_star, P["delta"][..., None] * P["alpha"])
    assert np.array_equal(z_star, P["delta"] * (P["zb"] - P["zu"]))
    for r in range(2):
        for j in range(2):
            D = Fraction(float(P["delta"][r, j]))
            for word in range(1 << q):
                c = [1 if (word >> b) & 1 else -1 for b in range(q)]
                lhs = D * (sum(Fraction(float(a)) * cb for a, cb in zip(P["alpha"][r, j], c))
                           + Fraction(float(P["zb"][r, j])) - Fraction(float(P["zu"][r, j])))
                rhs = sum(Fraction(float(a)) * cb for a, cb in zip(a_star[r, j], c)) + Fraction(float(z_star[r, j]))
                scale = abs(D) * (sum(abs(Fraction(float(a))) for a in P["alpha"][r, j])
                                  + abs(Fraction(float(P["zb"][r, j]))) + abs(Fraction(float(P["zu"][r, j]))))
                assert abs(lhs - rhs) <= Fraction(q + 2, 2 ** 24) * scale


@pytest.mark.parametrize("q", [2, 3, 4])
def test_exported_bcq_reconstructs_quantizer_output(q):
    """With the codes of the last quantizer step (REUSE), R_B(C; Theta_B*) equals
    the quantizer output w^ up to fp32 rounding of both sides."""
    P = random_params(600 + q, q)
    _, codes = O.quantize_fwd(P["W"], P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], None,
                              P["g"], mode=O.MAP_FULL)
    what, _ = O.quantize_fwd(P["W"], P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes,
                             P["g"], mode=O.MAP_LOCAL_PERIODIC, step=1)
    planes, a_star, z_star, used = O.export_bcq(P["W"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, P["g"])
    assert np.array_equal(used, codes)
    out, n_in = P["W"].shape
    rec = O.levels(a_star, z_star)
    rec = np.take_along_axis(rec, unpack_bitplanes(planes, n_in).reshape(out, -1, P["g"]).astype(np.int64), -1)
    bound = (2 * (q + 4) * 2.0 ** -24 * np.abs(P["delta"]) *
             (np.abs(P["alpha"]).sum(-1) + np.abs(P["zb"]) + np.abs(P["zu"])))[..., None]
    assert np.all(np.abs(rec - what.reshape(out, -1, P["g"])) <= bound)


@pytest.mark.parametrize("q", [1, 2, 3, 4])
def test_bitplane_round_trip_and_layout(q):
    rng = np.random.default_rng(q)
    codes = rng.integers(0, 1 << q, (5, 96)).astype(np.uint8)
    planes = O.pack_bitplanes(codes, q)
    assert planes.shape == (q, 5, 3) and planes.dtype == np.uint32
    assert np.array_equal(unpack_bitplanes(planes, 96), codes)
    # bit b of word t of plane j is c_{j+1} of column 32 t + b
    r, col, j = 3, 70, q - 1
    assert ((planes[j, r, col // 32] >> (col % 32)) & 1) == ((codes[r, col] >> j) & 1)


def test_eq4_matches_exact_brute_force():
    """Eq. 4 on dyadic values (exact fp32 arithmetic): the code is the nearest
    level of Theta_B*, ties to the lower level then the lower code word."""
    q, g = 3, 32
    rng = np.random.default_rng(3)
    W = (rng.integers(-200, 201, (2, 64)) / 128).astype(F32)
    delta = np.full((2, 2), 0.25, F32)
    zu = (rng.integers(0, 16, (2, 2)) / 4).astype(F32)
    alpha = (rng.integers(1, 9, (2, 2, q)) / 4).astype(F32)
    zb = (rng.integers(0, 16, (2, 2)) / 4).astype(F32)
    a_star, z_star = O.unify(delta, zu, alpha, zb)
    codes = O.codes_eq4(W, a_star, z_star, g)
    for r in range(2):
        for i in range(64):
            j = i // g
            cands = []
            for word in range(1 << q):
                c = [1 if (word >> b) & 1 else -1 for b in range(q)]
                lv = sum(Fraction(float(a)) * cb for a, cb in zip(a_star[r, j], c)) + Fraction(float(z_star[r, j]))
                cands.append((abs(Fraction(float(W[r, i])) - lv), lv, word))
            best = min(cands)
            assert codes[r, i] == best[2]


def test_export_sizes_match_memory_formula():
    """App. F.1: a k-bit group of g weights costs g k code bits plus k+1 reals
    (16-bit each in the paper's count)."""
    for case in GOLD["memory_cost"]["cases"]:
        g, k = case["g"], case["k"]
        codes = np.zeros((1, g), np.uint8)
        planes = O.pack_bitplanes(codes, k)
        a_star, z_star = O.unify(np.ones((1, 1), F32), np.zeros((1, 1), F32), np.ones((1, 1, k), F32),
                                 np.zeros((1, 1), F32))
        bits = planes.size * 32 + 16 * (a_star.size + z_star.size)
        assert bits == case["bits_per_group"]
        assert (bits - g * k) / g == case["overhead_bits_per_weight"]
