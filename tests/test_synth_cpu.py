"""The seeded synthetic inputs that stand in for the paper's model weights:
the shapes and settings of every workload, their distributions and outlier
columns, row-range reproducibility, and the bf16 rounding (nearest even),
checked against torch's own conversion."""

import numpy as np
import pytest
import torch
from scipy import stats

from paper_2506_03781_gb300 import synth

WL = synth.WORKLOADS


def shapes(name):
    return [(m.name, m.out, m.n_in) for m in WL[name].matrices]


def test_workload_shapes_and_settings():
    assert shapes("mat1k_f32") == [("w", 1024, 1024)]
    assert shapes("attn4k_bf16") == [("w", 4096, 4096)]
    assert shapes("mlp14336x4096_bf16") == [("w", 14336, 4096)]
    assert shapes("llama3_8b_block_bf16") == [
        ("q_proj", 4096, 4096), ("k_proj", 1024, 4096), ("v_proj", 1024, 4096), ("o_proj", 4096, 4096),
        ("gate_proj", 14336, 4096), ("up_proj", 14336, 4096), ("down_proj", 4096, 14336)]
    assert shapes("llama2_70b_mlp_bf16") == [
        ("gate_proj", 28672, 8192), ("up_proj", 28672, 8192), ("down_proj", 8192, 28672)]
    assert WL["llama3_8b_block_bf16"].n_elems == 218_103_808
    assert WL["llama2_70b_mlp_bf16"].n_elems == 704_643_072
    assert [(WL[n].q, WL[n].g) for n in WL] == [(3, 128), (3, 128), (3, 128), (2, 64), (3, 128)]
    assert WL["mlp14336x4096_bf16"].qs == (2, 3, 4) and WL["mlp14336x4096_bf16"].p == 2
    assert WL["mat1k_f32"].wdtype == "f32"
    assert all(WL[n].wdtype == "bf16" for n in WL if n != "mat1k_f32")


def test_outlier_columns():
    # round(0.001 in) columns x10 for the Llama-3 shapes, round(0.0005 in) x20 for Llama-2-70B
    for n_in, frac, k in ((4096, 0.001, 4), (8192, 0.0005, 4), (28672, 0.0005, 14), (14336, 0.0, 0)):
        cols = synth.outlier_columns(n_in, frac, 3)
        assert len(cols) == k and len(set(cols.tolist())) == k
        assert np.all(cols >= 0) and np.all(cols < n_in) and np.all(np.diff(cols) > 0)
    assert np.array_equal(synth.outlier_columns(4096, 0.001, 3), synth.outlier_columns(4096, 0.001, 3))
    assert not np.array_equal(synth.outlier_columns(4096, 0.01, 3), synth.outlier_columns(4096, 0.01, 4))
    m = WL["llama2_70b_mlp_bf16"].matrices[2]
    assert (m.outlier_frac, m.outlier_mult) == (0.0005, 20.0)
    m = WL["mlp14336x4096_bf16"].matrices[0]
    assert (m.dist, m.std, m.outlier_frac, m.outlier_mult) == ("t4", 0.02, 0.001, 10.0)


def test_normal_weights_have_the_stated_scale():
    _, W = synth.workload_weights(WL["mat1k_f32"], 0)
    assert W.dtype == np.float32 and W.shape == (1024, 1024)
    assert abs(W.std() - 0.02) < 0.02 * 0.01 and abs(W.mean()) < 1e-4


def test_student_t_weights_have_the_stated_scale_and_tails():
    """Student-t(4) scaled to std 0.02: the median of |w| is t_4's 0.75
    quantile times 0.02 / sqrt(2) (Var t_4 = 2); the tails are heavier than a
    normal's; the outlier columns are ten times wider."""
    m = WL["attn4k_bf16"].matrices[0]
    _, W = synth.workload_weights(WL["attn4k_bf16"], 0, slice(0, 1024))
    cols = synth.outlier_columns(m.n_in, m.outlier_frac, (WL["attn4k_bf16"].seed, 0))
    normal_cols = np.setdiff1d(np.arange(m.n_in), cols)
    body = np.abs(W[:, normal_cols].astype(np.float64))
    med = stats.t.ppf(0.75, 4) * 0.02 / np.sqrt(2.0)
    assert abs(np.median(body) / med - 1) < 0.02
    # heavy tails: beyond 5 standard deviations far more often than a normal
    assert (body > 5 * 0.02).mean() > 100 * 2 * stats.norm.sf(5)
    ratio = np.median(np.abs(W[:, cols])) / np.median(body)
    assert 9.0 < ratio < 11.0


def test_row_ranges_reproduce_the_full_draw():
    m = synth.Matrix("w", 700, 64, "t4", 0.02, 0.05, 10.0)
    full = synth.matrix_weights(m, (5, 0))
    for a, b in ((0, 1), (255, 257), (300, 700), (699, 700), (0, 700)):
        assert np.array_equal(synth.matrix_weights(m, (5, 0), slice(a, b)), full[a:b]), (a, b)


def test_bf16_rounding_is_nearest_even_like_torch():
    rng = np.random.default_rng(0)
    x = (rng.standard_normal(4096) * 0.02).astype(np.float32)
    bits = x.view(np.uint32)
    ties = (bits & np.uint32(0xFFFF0000)) | np.uint32(0x8000)     # exactly halfway between two bf16 values
    x = np.concatenate([x, ties.view(np.float32), np.float32([0.0, -0.0, 1.0, -3.5, 65504.0])])
    raw, vals = synth.bf16_round(x)
    t = torch.from_numpy(x).to(torch.bfloat16)
    assert np.array_equal(raw, t.view(torch.int16).numpy().view(np.uint16))
    assert np.array_equal(vals.view(np.uint32), t.float().numpy().view(np.uint32))
    # a tie goes to the even neighbour: the kept upper half has its lowest bit clear
    kept = raw[4096:8192]
    up = (ties >> 16).astype(np.uint16)
    assert np.all((kept == up) | (kept == up + 1)) and np.all((kept & 1) == 0)


@pytest.mark.parametrize("name", ["attn4k_bf16", "mlp14336x4096_bf16"])
def test_stored_bf16_weights_are_exactly_their_values(name):
    raw, vals = synth.workload_weights(WL[name], 0, slice(0, 8))
    assert raw.dtype == np.uint16 and vals.dtype == np.float32
    assert np.array_equal((raw.astype(np.uint32) << 16).view(np.float32), vals)
