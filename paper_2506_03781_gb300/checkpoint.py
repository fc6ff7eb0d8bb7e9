"""Checkpoint and resume of the quantizer state.

A run of Algorithm 1 carries three things from one optimisation step to the
next, and nothing else:
- Theta_IF = (Delta, z_U, s, s_r, alpha, z_B) of every weight matrix, the
  parameters its SGD updates (Eq. 1, Eq. 3);
- the code array C: the local mapping M*_B of a remap step starts from the
  stored code of each weight and moves it by at most one rank (Algorithm 4),
  so the codes are state, not a function of Theta;
- the step counter t, which decides the steps that remap (t mod p = 0).
W is frozen (Algorithm 1 outputs only Theta*_B and C) and W^ is a function of
(Theta, C): W^ = Delta (l(C) - z_U) with the level l(c) = sum_j c_j alpha_j +
z_B (R_B, then D_R).  So a checkpoint holds Theta, C and t, and a resume
rebuilds W^ with the forward of a step that keeps the codes, which applies
R_B and D_R only and maps nothing.  A resumed run then continues exactly as
the uninterrupted one would have.

The file is a ``torch.save`` of plain tensors, ints, floats and strings, read
back with ``torch.load(weights_only=True)``.
"""

from __future__ import annotations

import torch

from . import api

FORMAT = "uniquan-f-quantizer-state/1"


def snapshot(params, codes):
    """Host copies of one matrix's state: ({name: tensor}, codes)."""
    missing = [k for k in api.PARAM_NAMES if k not in params]
    if missing:
        raise ValueError(f"params lack {missing}")
    return ({k: params[k].detach().to("cpu", copy=True) for k in api.PARAM_NAMES},
            codes.detach().to("cpu", copy=True))


def save_state(path, matrices, step, **meta):
    """Writes the state of several matrices and the step counter to ``path``.

    matrices: {name: (params dict, codes tensor)} on any device.  step: the
    step counter of the next optimisation step.  meta: ints, floats or
    strings kept beside the state (q, g, p, mapping mode, learning rates ...).
    """
    for k, v in meta.items():
        if not isinstance(v, (int, float, str, bool)):
            raise TypeError(f"meta[{k!r}] must be an int, float, str or bool, not {type(v).__name__}")
    if int(step) < 0:
        raise ValueError(f"step={step} must be >= 0")
    state = {"format": FORMAT, "step": int(step), "meta": dict(meta), "matrices": {}}
    for name, (params, codes) in matrices.items():
        p, c = snapshot(params, codes)
        state["matrices"][name] = {"params": p, "codes": c}
    torch.save(state, path)


def load_state(path):
    """Reads a file written by save_state: returns (matrices, step, meta),
    matrices = {name: (params dict, codes)} as host tensors."""
    state = torch.load(path, map_location="cpu", weights_only=True)
    if not isinstance(state, dict) or state.get("format") != FORMAT:
        raise ValueError(f"{path}: not a quantizer state file ({FORMAT})")
    mats = {name: (m["params"], m["codes"]) for name, m in state["matrices"].items()}
    return mats, state["step"], state["meta"]


def restore_into(saved, params, codes):
    """Copies one saved matrix state (params dict, codes) into existing
    buffers, after checking that every shape and dtype matches."""
    sp, sc = saved
    for k in api.PARAM_NAMES:
        if k not in sp:
            raise ValueError(f"saved state lacks {k}")
        if tuple(sp[k].shape) != tuple(params[k].shape) or sp[k].dtype != params[k].dtype:
            raise ValueError(f"{k}: saved {tuple(sp[k].shape)} {sp[k].dtype}, buffer "
                             f"{tuple(params[k].shape)} {params[k].dtype}")
    if tuple(sc.shape) != tuple(codes.shape) or sc.dtype != codes.dtype:
        raise ValueError(f"codes: saved {tuple(sc.shape)} {sc.dtype}, buffer {tuple(codes.shape)} {codes.dtype}")
    for k in api.PARAM_NAMES:
        params[k].copy_(sp[k])
    codes.copy_(sc)


def rebuild_what(qz: api.Quantizer, stream=None):
    """W^ = Delta (l(C) - z_U) from the current parameters and codes, with no
    mapping: the forward of a step that keeps the codes (local mapping, a
    step that is not a multiple of the period)."""
    qz.fwd(1, p_period=2, map_mode=api.MAP_LOCAL_PERIODIC, stream=stream)
