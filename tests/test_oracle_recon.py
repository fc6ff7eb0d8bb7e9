"""Pins of the oracle's reconstruction loop (oracle.recon, Algorithm 1 around
the quantizer).

* attention: the batched causal grouped-query attention equals a brute-force
  loop over query positions and heads (softmax over the visible keys only,
  the key/value head of query head h is h // (heads / kv_heads));
* rotary embedding: preserves the norm of every pair and rotates position 0
  by nothing; the relative-position property of its dot products;
* the loss gradient: torch.autograd equals central finite differences of the
  fp64 loss in a few weight entries;
* the loss of W^ = W on X^ = X is zero;
* one step of the loop is train_step applied per weight to the gradient of
  the loss of the current W^ (composition, against the pieces called
  separately), and with the codes held the paper's learning rates lower the
  loss at every step (plain gradient descent on the block output error).
"""

import math

import numpy as np
import pytest
import torch

import oracle as O
from oracle import recon as R
from paper_2506_03781_gb300 import synth

F64 = torch.float64


def tiny():
    return synth.BLOCKS["tiny"]


def weights64(shape, seed=0):
    W = synth.block_weights(shape, seed)
    return {n: W[n][1] for n in R.NAMES}


def test_attention_equals_brute_force_loop():
    shape = tiny()
    W = {n: torch.tensor(v, dtype=F64) for n, v in weights64(shape).items()}
    X, _ = synth.block_inputs(shape, 1, 0)
    h = R.rms_norm(torch.tensor(X[0], dtype=F64), shape.eps)
    got = R.attention(h, W, shape)
    T, H, KV, hd = shape.seq, shape.heads, shape.kv_heads, shape.head_dim
    q = R.rotary((h @ W["q_proj"].T).reshape(T, H, hd).transpose(0, 1), shape.theta)
    k = R.rotary((h @ W["k_proj"].T).reshape(T, KV, hd).transpose(0, 1), shape.theta)
    v = (h @ W["v_proj"].T).reshape(T, KV, hd).transpose(0, 1)
    o = torch.zeros(T, H * hd, dtype=F64)
    for head in range(H):
        kvh = head // (H // KV)
        for i in range(T):
            s = [float(q[head, i] @ k[kvh, j]) / math.sqrt(hd) for j in range(i + 1)]
            m = max(s)
            e = [math.exp(x - m) for x in s]
            z = sum(e)
            o[i, head * hd:(head + 1) * hd] = sum((e[j] / z) * v[kvh, j] for j in range(i + 1))
    ref = o @ W["o_proj"].T
    assert torch.allclose(got, ref, rtol=1e-12, atol=1e-13)


def test_rotary_is_a_rotation_with_relative_phase():
    torch.manual_seed(0)
    x = torch.randn(2, 9, 16, dtype=F64)
    r = R.rotary(x, 10000.0)
    half = 8
    n0 = x[..., :half] ** 2 + x[..., half:] ** 2
    n1 = r[..., :half] ** 2 + r[..., half:] ** 2
    assert torch.allclose(n0, n1)
    assert torch.allclose(r[:, 0], x[:, 0])
    # <rot(a, p), rot(b, p')> depends on p - p' only
    a = torch.randn(1, 1, 16, dtype=F64).expand(1, 9, 16).clone()
    b = torch.randn(1, 1, 16, dtype=F64).expand(1, 9, 16).clone()
    ra, rb = R.rotary(a, 10000.0)[0], R.rotary(b, 10000.0)[0]
    assert torch.allclose(ra[5] @ rb[3], ra[4] @ rb[2])


def test_loss_gradient_matches_finite_differences():
    shape = tiny()
    W = weights64(shape)
    X, Xh = synth.block_inputs(shape, 1, 1, perturb=0.05)
    Y = R.targets(X, W, shape)[0]
    What = {n: (W[n] * (1 + 0.01 * np.random.default_rng(2).standard_normal(W[n].shape))).astype(np.float32)
            for n in R.NAMES}
    loss, G = R.loss_and_grads(Y, Xh[0], What, shape)
    rng = np.random.default_rng(3)

    def loss_of(Wd):
        Wt = {n: torch.tensor(np.asarray(Wd[n], np.float64)) for n in R.NAMES}
        out = R.block_forward(torch.tensor(Xh[0], dtype=F64), Wt, shape)
        return float(((out - torch.tensor(Y)) ** 2).mean())

    for n in ("q_proj", "v_proj", "down_proj"):
        for _ in range(3):
            i, j = rng.integers(W[n].shape[0]), rng.integers(W[n].shape[1])
            h = 1e-4
            Wp = {k: v.astype(np.float64).copy() for k, v in What.items()}
            Wm = {k: v.astype(np.float64).copy() for k, v in What.items()}
            Wp[n][i, j] += h
            Wm[n][i, j] -= h
            fd = (loss_of(Wp) - loss_of(Wm)) / (2 * h)
            assert abs(fd - G[n][i, j]) <= 1e-5 * max(abs(fd), 1e-9) + 1e-12, (n, i, j, fd, G[n][i, j])


def test_unquantized_block_has_zero_loss():
    shape = tiny()
    W = weights64(shape)
    X, _ = synth.block_inputs(shape, 1, 4)
    Y = R.targets(X, W, shape)[0]
    loss, G = R.loss_and_grads(Y, X[0], W, shape)
    assert loss == 0.0
    assert all(np.abs(G[n]).max() == 0.0 for n in R.NAMES)


def test_step_is_train_step_of_the_loss_gradient_and_lowers_the_loss():
    shape = tiny()
    q, g = 3, 32
    W = weights64(shape)
    X, Xh = synth.block_inputs(shape, 2, 5, perturb=0.02)
    Ys = R.targets(X, W, shape)
    state = R.init_state(W, q, g, G=4, T=3)
    loss0, G = R.loss_and_grads(Ys[0], Xh[0], {n: state[n][2] for n in R.NAMES}, shape)
    new, loss = R.recon_step(state, W, Ys[0], Xh[0], shape, g, 0)
    assert loss == loss0
    for n in R.NAMES:
        P, c, _ = state[n]
        P1, c1, w1 = O.train_step(W[n], P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], c, G[n], g, 0)
        assert all(np.array_equal(new[n][0][k], P1[k]) for k in P1)
        assert np.array_equal(new[n][1], c1) and np.array_equal(new[n][2], w1)
    # With the codes held (no remap: p larger than the number of steps) W^ is
    # a smooth function of Delta, z_U, alpha, z_B, and the steps are plain
    # gradient descent on it: the loss of the sample goes down at every step.
    # (Remap steps move codes and may raise it: the mapping is not descended.)
    st, losses = state, []
    for t in range(5):
        st, l = R.recon_step(st, W, Ys[0], Xh[0], shape, g, t, p=1000)
        losses.append(l)
    after, _ = R.loss_and_grads(Ys[0], Xh[0], {n: st[n][2] for n in R.NAMES}, shape)
    losses.append(after)
    assert all(b < a for a, b in zip(losses, losses[1:])), losses
