"""Plain CPU restatement of the block-wise reconstruction loop of Algorithm 1
around the UniQuan_F quantizer -- TEST INFRASTRUCTURE ONLY (see the package
docstring): the product path never imports this module.

Algorithm 1 quantizes one Transformer block f at a time.  For every sample
s it quantizes the block's weights Phi into Phi^ (Eq. 3), computes the
reconstruction loss || f(X_s; Phi) - f(X^_s; Phi^) ||^2, back-propagates
and updates Theta_IF.  Here:

* f is a Llama-style decoder block (RMSNorm, grouped-query attention with
  rotary position embedding and a causal mask, RMSNorm, SwiGLU MLP; norm
  weights one), evaluated in fp64 with plain torch CPU ops;
* the loss is the MEAN of the squared differences (the reading taken for
  the paper's squared Frobenius norm: the mean keeps the learning rates of
  the hyperparameter table meaningful for any block and sequence size);
* the quantizer step is oracle.train_step: the backward of step t, the SGD
  update, and the forward of step t + 1, so one optimisation step consumes
  W^_t and produces W^_{t+1}; the loop starts from W^_0 = Q(W; Theta_0) of
  the unified initialization.
"""

from __future__ import annotations

import math

import numpy as np
import torch

from . import uniquan as U

F64 = torch.float64
NAMES = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def rms_norm(x, eps):
    """x / sqrt(mean(x^2) + eps) over the hidden dimension (norm weight one)."""
    return x / torch.sqrt((x * x).mean(-1, keepdim=True) + eps)


def rotary(x, theta):
    """Rotary position embedding of x [heads, seq, head_dim]: the pair
    (x_i, x_{i+h/2}) of position p is rotated by the angle p / theta^(2i/h)."""
    _, T, hd = x.shape
    half = hd // 2
    inv = theta ** (-torch.arange(half, dtype=F64) * 2.0 / hd)
    ang = torch.arange(T, dtype=F64)[:, None] * inv[None, :]
    c, s = torch.cos(ang), torch.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * c - x2 * s, x1 * s + x2 * c], dim=-1)


def attention(h, W, shape):
    """Causal grouped-query self-attention of h [seq, d]."""
    T = h.shape[0]
    H, KV, hd = shape.heads, shape.kv_heads, shape.head_dim
    q = (h @ W["q_proj"].T).reshape(T, H, hd).transpose(0, 1)
    k = (h @ W["k_proj"].T).reshape(T, KV, hd).transpose(0, 1)
    v = (h @ W["v_proj"].T).reshape(T, KV, hd).transpose(0, 1)
    q, k = rotary(q, shape.theta), rotary(k, shape.theta)
    k = k.repeat_interleave(H // KV, dim=0)
    v = v.repeat_interleave(H // KV, dim=0)
    scores = q @ k.transpose(-1, -2) / math.sqrt(hd)
    mask = torch.triu(torch.ones(T, T, dtype=torch.bool), diagonal=1)
    scores = scores.masked_fill(mask, float("-inf"))
    o = torch.softmax(scores, dim=-1) @ v                      # [H, T, hd]
    return o.transpose(0, 1).reshape(T, H * hd) @ W["o_proj"].T


def block_forward(X, W, shape):
    """f(X; W): X [seq, d] fp64 tensor, W dict of fp64 tensors [out, in]."""
    X1 = X + attention(rms_norm(X, shape.eps), W, shape)
    h = rms_norm(X1, shape.eps)
    mlp = (torch.nn.functional.silu(h @ W["gate_proj"].T) * (h @ W["up_proj"].T)) @ W["down_proj"].T
    return X1 + mlp


def loss_and_grads(Y, Xh, What, shape):
    """Mean squared difference between the target Y = f(X; W) and
    f(X^; W^), and its gradient w.r.t. every W^ (fp64, returned as fp32
    arrays: the dL/dW^ the quantizer's backward takes)."""
    Wt = {n: torch.tensor(np.asarray(What[n], np.float64), requires_grad=True) for n in NAMES}
    out = block_forward(torch.tensor(np.asarray(Xh, np.float64)), Wt, shape)
    loss = ((out - torch.tensor(np.asarray(Y, np.float64))) ** 2).mean()
    loss.backward()
    return float(loss.detach()), {n: Wt[n].grad.numpy().astype(np.float32) for n in NAMES}


def targets(X, W, shape):
    """Y_s = f(X_s; W) for every sample (the unquantized block), fp64."""
    Wt = {n: torch.tensor(np.asarray(W[n], np.float64)) for n in NAMES}
    return [block_forward(torch.tensor(np.asarray(x, np.float64)), Wt, shape).numpy() for x in X]


def init_state(W, q, g, G=30, T=15):
    """Unified initialization of every weight (Algorithm 2) and the forward
    of step 0: state = {name: (params dict, codes, W^_0)}."""
    state = {}
    for n in NAMES:
        init = U.unified_init(W[n], q, g, G=G, T=T)
        P = {k: init[k] for k in ("delta", "zu", "s", "sr", "alpha", "zb")}
        what, codes = U.quantize_fwd(W[n], P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"],
                                     init["codes"], g, U.MAP_LOCAL_PERIODIC, 0, 2)
        state[n] = (P, codes, what)
    return state


def recon_step(state, W, Y, Xh, shape, g, t, lr_F=U.LR_F, lr_B=U.LR_B, mode=U.MAP_LOCAL_PERIODIC, p=2):
    """One optimisation step of Algorithm 1 on one sample: loss of W^_t,
    dL/dW^_t, then train_step of every weight.  Returns (new state, loss)."""
    loss, G = loss_and_grads(Y, Xh, {n: state[n][2] for n in NAMES}, shape)
    new = {}
    for n in NAMES:
        P, codes, _ = state[n]
        P1, c1, w1 = U.train_step(W[n], P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, G[n], g,
                                  t, lr_F, lr_B, mode, p)
        new[n] = (P1, c1, w1)
    return new, loss
