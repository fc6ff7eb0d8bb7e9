"""Algorithm 1 on the GPU: block-wise reconstruction of one Llama-style
decoder block with the UniQuan_F quantizer.

For every sample s and step t, with W^_t the quantizer output of step t:

    loss_t = mean( (f(X_s; W) - f(X^_s; W^_t))^2 )      (the block's output error)
    dL/dW^_t by back-propagation through the block
    uq_train_step per weight: backward of step t, SGD update of Theta_IF,
                              forward of step t + 1 -> W^_{t+1}, codes_{t+1}

The block itself (RMSNorm, rotary grouped-query attention with a causal
mask, RMSNorm, SwiGLU MLP; norm weights one) runs as torch operations in
`compute_dtype` (cuBLAS GEMMs and torch's fused attention): it is the model
being quantized, not the quantizer.  Every quantizer step -- the unified
initialization, the forward of step 0 and every fused step -- runs in the
library's kernels through the C ABI.  The unquantized outputs f(X_s; W) are
computed once per sample (they do not change during the optimisation).

The loss is the mean of the squared differences (a reading of the paper's
squared Frobenius norm that keeps the learning rates of its hyperparameter
table meaningful for any block and sequence size).
"""

from __future__ import annotations

import math

import torch
import torch.nn.functional as F

from . import api, checkpoint

NAMES = ("q_proj", "k_proj", "v_proj", "o_proj", "gate_proj", "up_proj", "down_proj")


def _rms_norm(x, eps):
    xf = x.float()
    return (xf * torch.rsqrt(xf.pow(2).mean(-1, keepdim=True) + eps)).to(x.dtype)


def _rotary(x, theta):
    # x [batch, heads, seq, head_dim]: pair (i, i + h/2) of position p rotated by p / theta^(2i/h)
    T, hd = x.shape[-2], x.shape[-1]
    half = hd // 2
    inv = theta ** (-torch.arange(half, device=x.device, dtype=torch.float32) * 2.0 / hd)
    ang = torch.arange(T, device=x.device, dtype=torch.float32)[:, None] * inv[None, :]
    c, s = torch.cos(ang).to(x.dtype), torch.sin(ang).to(x.dtype)
    x1, x2 = x[..., :half], x[..., half:]
    return torch.cat([x1 * c - x2 * s, x1 * s + x2 * c], dim=-1)


def block_forward(X, W, shape):
    """f(X; W) for X [seq, d] and a dict of weights [out, in], in X's dtype."""
    T = X.shape[0]
    H, KV, hd = shape.heads, shape.kv_heads, shape.head_dim
    h = _rms_norm(X, shape.eps)
    q = F.linear(h, W["q_proj"]).view(1, T, H, hd).transpose(1, 2)
    k = F.linear(h, W["k_proj"]).view(1, T, KV, hd).transpose(1, 2)
    v = F.linear(h, W["v_proj"]).view(1, T, KV, hd).transpose(1, 2)
    q, k = _rotary(q, shape.theta), _rotary(k, shape.theta)
    k = k.repeat_interleave(H // KV, dim=1)
    v = v.repeat_interleave(H // KV, dim=1)
    o = F.scaled_dot_product_attention(q, k, v, is_causal=True, scale=1.0 / math.sqrt(hd))
    X1 = X + F.linear(o.transpose(1, 2).reshape(T, H * hd), W["o_proj"])
    h2 = _rms_norm(X1, shape.eps)
    return X1 + F.linear(F.silu(F.linear(h2, W["gate_proj"])) * F.linear(h2, W["up_proj"]), W["down_proj"])


def level_ranks(alpha, zb, codes, g):
    """Index of every weight's level among its group's 2^q levels, as
    Algorithm 4 indexes them: the levels l(c) = c_1 a_1 + ... + c_q a_q + z_B
    (fp32, summed left to right) sorted ascending, equal levels in code-word
    order.  The index-change statistics of the paper's Table 2 compare these
    ranks between steps.  alpha [out, in/g, q], zb [out, in/g], codes
    [out, in] uint8 (bits at or above q ignored) -> uint8 ranks [out, in].
    Device tensors in, device tensor out; a report, outside the quantizer."""
    out, n_in = codes.shape
    q = alpha.shape[-1]
    L = 1 << q
    cw = torch.arange(L, device=codes.device)
    lv = None
    for j in range(q):
        cj = (((cw >> j) & 1) * 2 - 1).to(torch.float32)           # c_j of every code word
        term = alpha[..., j:j + 1] * cj                              # exact: c_j = +-1
        lv = term if lv is None else lv + term
    lv = lv + zb[..., None]
    order = torch.sort(lv, dim=-1, stable=True).indices              # ties keep code-word order
    rank_of_code = torch.empty_like(order)
    rank_of_code.scatter_(-1, order, cw.expand_as(order).contiguous())
    c = (codes.view(out, n_in // g, g).long() & (L - 1))
    return torch.gather(rank_of_code, -1, c).view(out, n_in).to(torch.uint8)


def index_change_shares(r_a, r_b):
    """Shares of weights whose level index moved by 0, 1, 2 and more than 2
    between two rank arrays (the four columns of Table 2)."""
    d = (r_a.to(torch.int16) - r_b.to(torch.int16)).abs()
    n = d.numel()
    c0, c1, c2 = int((d == 0).sum()), int((d == 1).sum()), int((d == 2).sum())
    return [c0 / n, c1 / n, c2 / n, (n - c0 - c1 - c2) / n]


class BlockReconstructor:
    """The quantizer state of one block and the steps of Algorithm 1.

    weights: {name: stored array} (raw bf16 bits as uint16, or fp32), shapes
    from `shape.matrices()`.  The shapes must be ones the fused step kernel
    takes (g in {32, 64, 128}; see uq_train_step).  init=True runs the
    unified initialization (G, T); otherwise load a state with set_state.
    """

    def __init__(self, shape, weights, q, g, device="cuda", compute_dtype=torch.bfloat16, G=30, T=15,
                 lr_F=api.LR_THETA_F, lr_B=api.LR_THETA_B, p=2, map_mode=api.MAP_LOCAL_PERIODIC, init=True):
        self.shape, self.q, self.g, self.p, self.map_mode = shape, q, g, p, map_mode
        self.lr_F, self.lr_B = lr_F, lr_B
        self.device = torch.device(device)
        self.dtype = compute_dtype
        # A bf16 block takes W^ and gives dL/dW^ in bf16 straight from the fused
        # step (uq_train_step_bf16): no conversion pass over the weights per step.
        self.bf16_io = compute_dtype == torch.bfloat16
        self.W, self.P, self.codes, self.what, self.G, self.qz = {}, {}, {}, {}, {}, {}
        self.what_c = {}
        for m in shape.matrices():
            n = m.name
            Wd = api.weights_tensor(weights[n], self.device)
            self.W[n] = Wd
            self.P[n] = api.empty_params(m.out, m.n_in, q, g, self.device)
            self.codes[n] = torch.empty(m.out, m.n_in, dtype=torch.uint8, device=self.device)
            self.what[n] = torch.empty(m.out, m.n_in, dtype=torch.float32, device=self.device)
            self.G[n] = torch.zeros(m.out, m.n_in, dtype=torch.float32, device=self.device)
            self.qz[n] = api.Quantizer(Wd, q, g, self.P[n], self.codes[n], self.what[n], self.G[n])
            if self.bf16_io:
                self.what_c[n] = torch.empty(m.out, m.n_in, dtype=torch.bfloat16, device=self.device)
            if init:
                api.uq_init_params(Wd, q, g, self.P[n], self.codes[n], G=G, T=T)
        # unquantized weights in the compute dtype, for the targets
        self.W_ref = {n: self.W[n].to(self.dtype) for n in NAMES}
        self.t = 0
        if init:
            self._forward0()

    def set_state(self, params, codes):
        """Load parameters and codes ({name: dict of arrays}, {name: array})
        and run the forward of step 0."""
        for n in NAMES:
            for k, v in params[n].items():
                self.P[n][k].copy_(torch.as_tensor(v))
            self.codes[n].copy_(torch.as_tensor(codes[n]))
        self._forward0()

    def _forward0(self):
        for n in NAMES:
            self.qz[n].fwd(0, self.p, self.map_mode)
        self._sync_compute_copy()
        self.t = 0

    def _sync_compute_copy(self):
        # the bf16 W^ the block reads, from the fp32 W^ of a separate forward
        # (step 0 or a resume; every later W^ comes from the fused step in bf16)
        if self.bf16_io:
            for n in NAMES:
                self.what_c[n].copy_(self.what[n])

    def quantizer_step(self, grads=None):
        """The fused steps of the seven weights (backward of step t, SGD, forward
        of t + 1), then t += 1.  grads: {name: dL/dW^} in bf16 for a bf16 block
        (uq_train_step_bf16); otherwise the fp32 buffers self.G are used."""
        for n in NAMES:
            if self.bf16_io:
                api.uq_train_step_bf16(self.W[n], self.q, self.g, self.P[n], self.codes[n], grads[n],
                                       self.what_c[n], self.t, self.lr_F, self.lr_B, self.map_mode, self.p)
            else:
                self.qz[n].train_step(self.t, self.lr_F, self.lr_B, self.p, self.map_mode)
        self.t += 1

    @torch.no_grad()
    def targets(self, X):
        """f(X_s; W) for every sample X_s [seq, d]."""
        return [block_forward(x.to(self.dtype), self.W_ref, self.shape) for x in X]

    def step(self, Y, Xh):
        """One optimisation step on one sample; returns the loss of W^_t
        (a 0-d tensor on the device, no synchronisation)."""
        leaves = {}
        if self.bf16_io:
            # W^ is already bf16; autograd hands back dL/dW^ in bf16
            for n in NAMES:
                leaves[n] = self.what_c[n].detach().requires_grad_(True)
            Wc = leaves
        else:
            for n in NAMES:
                leaf = self.what[n].detach().requires_grad_(True)
                self.G[n].zero_()
                leaf.grad = self.G[n]                   # back-propagation accumulates into dL/dW^
                leaves[n] = leaf
            Wc = {n: leaves[n].to(self.dtype) for n in NAMES}
        out = block_forward(Xh.to(self.dtype), Wc, self.shape)
        loss = (out.float() - Y.float()).pow(2).mean()
        loss.backward()
        grads = None
        if self.bf16_io:
            grads = {n: leaves[n].grad.contiguous() for n in NAMES}
        else:
            for n in NAMES:
                gr = leaves[n].grad
                if gr.data_ptr() != self.G[n].data_ptr():   # autograd replaced the buffer instead of adding into it
                    self.G[n].copy_(gr)
        for n in NAMES:
            leaves[n].grad = None
        self.quantizer_step(grads)
        return loss.detach()

    def ranks(self):
        """{name: level index of every weight} under the current parameters (level_ranks)."""
        return {n: level_ranks(self.P[n]["alpha"], self.P[n]["zb"], self.codes[n], self.g) for n in NAMES}

    def save(self, path):
        """Checkpoint: Theta_IF and the codes of the seven weights and the
        step counter (checkpoint.save_state)."""
        checkpoint.save_state(path, {n: (self.P[n], self.codes[n]) for n in NAMES}, self.t, q=self.q, g=self.g,
                              p=self.p, map_mode=self.map_mode, lr_F=float(self.lr_F), lr_B=float(self.lr_B))

    def load(self, path):
        """Resume from a checkpoint written by save(): loads Theta_IF, the
        codes and the step counter, and rebuilds W^ from them without
        mapping, so the next step() continues the saved run exactly."""
        mats, step, meta = checkpoint.load_state(path)
        if (meta.get("q"), meta.get("g")) != (self.q, self.g):
            raise ValueError(f"checkpoint has q={meta.get('q')}, g={meta.get('g')}; this block has "
                             f"q={self.q}, g={self.g}")
        if set(mats) != set(NAMES):
            raise ValueError(f"checkpoint holds {sorted(mats)}, expected {sorted(NAMES)}")
        for n in NAMES:
            checkpoint.restore_into(mats[n], self.P[n], self.codes[n])
        for n in NAMES:
            checkpoint.rebuild_what(self.qz[n])
        self._sync_compute_copy()
        self.t = step

    def state(self):
        """Host copies: ({name: params dict}, {name: codes}, {name: W^}); W^ is
        the block's copy (bf16 values as fp32 for a bf16 block)."""
        what = {n: (self.what_c[n].float() if self.bf16_io else self.what[n]).cpu().numpy() for n in NAMES}
        return ({n: {k: v.cpu().numpy() for k, v in self.P[n].items()} for n in NAMES},
                {n: self.codes[n].cpu().numpy() for n in NAMES}, what)
