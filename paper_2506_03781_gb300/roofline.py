"""Algorithmic HBM bytes of each kernel launch: what the method must move.

Per element: weights (2 B bf16 / 4 B fp32), s (4 B), code word (1 B),
w^ / dL/dw^ / ds (4 B each).  Per group: the parameters Delta, z_U, z_B and
alpha_1..q ((3 + q) * 4 B) read once, and the same number of gradient
values written by the backward.  Per row: s_r (4 B) read, ds_r written.
The fused optimisation step reads W, s, codes and dL/dw^ once and writes the
updated s, w^ of the next step and (on remap steps) its codes; every group
parameter and s_r is read and rewritten.
"""

from __future__ import annotations


def bytes_per_launch(kind: str, out: int, n_in: int, q: int, g: int, wbytes: int) -> int:
    n = out * n_in
    groups = out * (n_in // g)
    gp = groups * (3 + q) * 4
    if kind == "fwd_remap":        # read W, s, codes; write w^, codes
        return n * (wbytes + 4 + 1 + 4 + 1) + gp + out * 4
    if kind == "fwd_keep":         # read codes; write w^
        return n * (1 + 4) + gp
    if kind == "fwd_full":         # read W, s; write w^, codes
        return n * (wbytes + 4 + 4 + 1) + gp + out * 4
    if kind == "bwd":              # read W, s, codes, dL/dw^; write ds; group/row grads
        return n * (wbytes + 4 + 1 + 4 + 4) + 2 * gp + 2 * out * 4
    if kind in ("step_remap", "step_full"):  # read W, s, codes, dL/dw^; write s', w^, codes; params in/out
        return n * (wbytes + 4 + 1 + 4 + 4 + 4 + 1) + 2 * gp + 2 * out * 4
    if kind == "step_keep":        # as step_remap, codes not rewritten
        return n * (wbytes + 4 + 1 + 4 + 4 + 4) + 2 * gp + 2 * out * 4
    # OmniQuant maps: per group beta, gamma, alpha, z_B; no element-wise scale; W read on every step
    ogp = groups * (3 + q) * 4
    if kind == "omni_fwd_remap" or kind == "omni_fwd_full":   # read W, codes; write w^, codes
        return n * (wbytes + 1 + 4 + 1) + ogp
    if kind == "omni_fwd_keep":    # read W (for the group scales), codes; write w^
        return n * (wbytes + 1 + 4) + ogp
    if kind == "omni_bwd":         # read W, codes, dL/dw^; write the group gradients
        return n * (wbytes + 1 + 4) + 2 * ogp
    # AWQ maps: s_A per column, Delta_A, z_A, alpha, z_B per group
    if kind == "awq_fwd_remap" or kind == "awq_fwd_full":
        return n * (wbytes + 1 + 4 + 1) + gp + n_in * 4
    if kind == "awq_fwd_keep":     # read codes; write w^ (W not read)
        return n * (1 + 4) + gp + n_in * 4
    if kind == "awq_bwd":          # read W, codes, dL/dw^; write group gradients and ds_A
        return n * (wbytes + 1 + 4) + 2 * gp + 2 * n_in * 4
    if kind == "gemv":             # read planes, alpha*, z*, one token x (wbytes per value); write y
        return q * n // 8 + groups * (q + 1) * 4 + n_in * wbytes + out * 4
    if kind == "export_reuse":     # read codes; write planes, alpha*, z*
        return n * 1 + q * n // 8 + gp + groups * (q + 1) * 4
    if kind == "export_eq4":       # read W; write planes, alpha*, z*
        return n * wbytes + q * n // 8 + gp + groups * (q + 1) * 4
    raise ValueError(kind)


def step_bytes(out: int, n_in: int, q: int, g: int, wbytes: int, remap: bool) -> int:
    """One optimisation step of the quantizer: forward (remap or keep) + backward."""
    return (bytes_per_launch("fwd_remap" if remap else "fwd_keep", out, n_in, q, g, wbytes)
            + bytes_per_launch("bwd", out, n_in, q, g, wbytes))
