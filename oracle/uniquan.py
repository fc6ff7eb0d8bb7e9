"""Plain numpy restatement of the UniQuan_F per-element quantizer.

TEST INFRASTRUCTURE ONLY (see the package docstring): the product path never
imports this module.

Notation follows the paper: a weight group w (g values) is transformed by
FlexRound's T_F (Eq. 1), mapped to the nearest of the 2^q BCQ levels
(M_B, Sec. 2.3; or the local and periodic M*_B of Algorithm 4), reconstructed
by R_B (C alpha + z_B) and detransformed by D_R (Delta (w~ - z_U)).  The
bit-width is written q (the paper's k), L = 2^q.

Conventions shared with the CUDA library (they are readings of points the
paper leaves open; each one is listed with its reason in the design notes):

* a code word is an integer in [0, L); bit (j-1) set  <=>  c_j = +1;
* level of a code:  l(c) = ((c_1 a_1 + c_2 a_2) + ... + c_q a_q) + z_B,
  fp32, summed left to right (the matrix-vector product C alpha first, then
  the shift z_B, as R_B is written in Sec. 2.3);
* levels are sorted ascending; equal values keep ascending code-word order;
* full mapping M_B: argmin over ranks of |x - l|, fp32, ties -> lower rank;
* local mapping M*_B on a remap step (step % p == 0): candidates are the
  current rank d, then max(d-1, 0), then min(d+1, L-1); a candidate replaces
  the best only if strictly nearer;
* on a non-remap step the code word is kept and w~ = l(code) is recomputed
  with the current alpha, z_B;
* T_F: u = w / ((Delta * s) * s_r), x = u + z_U (fp32, IEEE division);
* D_R: w^ = Delta * (w~ - z_U) (fp32);
* gradient filter (App. C.1): tau = min_j |a_j|; the straight-through path
  of an element is zeroed when |x - w~| > tau.
"""

from __future__ import annotations

import itertools

import numpy as np

__all__ = [
    "MAP_FULL", "MAP_LOCAL_PERIODIC", "FILTER_STE", "FILTER_ELEMENT",
    "EXPORT_REUSE_CODES", "EXPORT_REMAP_EQ4",
    "CLIP_FIXED_MIN", "CLIP_FIXED_MAX", "CLIP_BALANCED",
    "signs", "levels", "sorted_levels",
    "transform_F", "map_full", "map_local", "reconstruct", "detransform",
    "quantize_fwd", "quantize_bwd", "bwd_l1_mass",
    "LR_F", "LR_B", "sgd_update", "train_step",
    "omni_params", "quantize_fwd_omni", "quantize_bwd_omni", "bwd_l1_mass_omni", "export_bcq_omni",
    "quantize_fwd_awq", "quantize_bwd_awq", "bwd_l1_mass_awq", "export_bcq_awq",
    "unify", "codes_eq4", "pack_bitplanes", "export_bcq", "export_bcq_half",
    "bcq_dequantize", "bcq_gemv",
    "clip_params", "greedy_init", "general_alternating", "init_error", "unified_init",
    "rtn",
]

F32 = np.float32
F64 = np.float64

MAP_FULL = 0
MAP_LOCAL_PERIODIC = 1
FILTER_STE = 0
FILTER_ELEMENT = 1
EXPORT_REUSE_CODES = 0
EXPORT_REMAP_EQ4 = 1
CLIP_FIXED_MIN = 0
CLIP_FIXED_MAX = 1
CLIP_BALANCED = 2


# ---------------------------------------------------------------------------
# BCQ levels (Sec. 2.3)
# ---------------------------------------------------------------------------

def signs(q: int, dtype=F32) -> np.ndarray:
    """Binary codes of all L = 2^q code words as a [L, q] array of +-1.

    Sec. 2.3: each weight carries c in {-1,+1}^q; row c of the result is the
    code of code word c (bit j-1 set  <=>  c_j = +1).
    """
    words = np.arange(1 << q)[:, None]
    bits = (words >> np.arange(q)[None, :]) & 1
    return np.where(bits == 1, 1, -1).astype(dtype)


def levels(alpha: np.ndarray, zb: np.ndarray) -> np.ndarray:
    """All 2^q quantization levels l(c) = c . alpha + z_B, fp32 (Sec. 2.3).

    alpha: [..., q]; zb: [...]  ->  [..., L] indexed by code word.
    The dot product is accumulated j = 1..q left to right, then z_B added.
    """
    alpha = np.asarray(alpha, F32)
    zb = np.asarray(zb, F32)
    q = alpha.shape[-1]
    S = signs(q)
    acc = S[:, 0] * alpha[..., None, 0]
    for j in range(1, q):
        acc = acc + S[:, j] * alpha[..., None, j]
    return acc + zb[..., None]


def sorted_levels(lv: np.ndarray):
    """Sort levels ascending (Algorithm 4 keeps the levels as an ordered list).

    Returns (sorted values [..., L], code_of_rank [..., L], rank_of_code
    [..., L]).  A stable sort orders equal levels by ascending code word.
    """
    code_of_rank = np.argsort(lv, axis=-1, kind="stable")
    srt = np.take_along_axis(lv, code_of_rank, axis=-1)
    rank_of_code = np.argsort(code_of_rank, axis=-1, kind="stable")
    return srt, code_of_rank, rank_of_code


# ---------------------------------------------------------------------------
# Transform / mapping / reconstruction / detransform (Sec. 3.1-3.3)
# ---------------------------------------------------------------------------

def transform_F(w, s, delta, zu, sr):
    """FlexRound transform T_F (Eq. 1): x = w / (Delta * s * s_r) + z_U.

    All arrays grouped: w, s [..., g]; delta, zu, sr broadcastable to [...].
    fp32, denominator formed left to right ((Delta * s) * s_r).
    Returns (x, u) with u = x - z_U before the shift (u is also what the
    backward pass differentiates).
    """
    w = np.asarray(w, F32)
    s = np.asarray(s, F32)
    denom = (np.asarray(delta, F32)[..., None] * s) * np.asarray(sr, F32)[..., None]
    u = w / denom
    x = u + np.asarray(zu, F32)[..., None]
    return x, u


def map_full(x, srt, code_of_rank):
    """Full nearest-level mapping M_B (Sec. 2.3; Eq. 2): argmin_l |x - l|.

    x [..., g]; srt, code_of_rank [..., L].  fp32 distances; the scan runs
    over ranks in ascending order and only a strictly smaller distance
    replaces the best, so ties go to the lower rank.  Returns code words.
    """
    x = np.asarray(x, F32)
    dist = np.abs(x[..., :, None] - srt[..., None, :])     # [..., g, L], fp32
    best_r = np.argmin(dist, axis=-1)                      # first minimum = lowest rank
    return np.take_along_axis(code_of_rank, best_r, axis=-1)


def map_local(x, codes, srt, code_of_rank, rank_of_code):
    """Local mapping step of M*_B (Algorithm 4, one remap step).

    Each element looks only at its current level d and the two neighbours
    max(d-1, 0), min(d+1, L-1) in the sorted level list and takes the
    nearest (|x - l|, fp32).  Candidates are examined in the order d, d-1,
    d+1 and replace the best only when strictly nearer.
    """
    x = np.asarray(x, F32)
    L = srt.shape[-1]
    d = np.take_along_axis(rank_of_code, codes.astype(np.int64), axis=-1)
    best_r = d
    best_d = np.abs(x - np.take_along_axis(srt, d, axis=-1))
    for cand in (np.maximum(d - 1, 0), np.minimum(d + 1, L - 1)):
        dc = np.abs(x - np.take_along_axis(srt, cand, axis=-1))
        upd = dc < best_d
        best_d = np.where(upd, dc, best_d)
        best_r = np.where(upd, cand, best_r)
    return np.take_along_axis(code_of_rank, best_r, axis=-1)


def reconstruct(codes, lv):
    """R_B per element: w~ = l(code) (Sec. 2.3, C alpha + z_B)."""
    return np.take_along_axis(lv, codes.astype(np.int64), axis=-1)


def detransform(wt, delta, zu):
    """D_R (Sec. 3.1): w^ = Delta * (w~ - z_U), fp32."""
    return np.asarray(delta, F32)[..., None] * (np.asarray(wt, F32) - np.asarray(zu, F32)[..., None])


def _grouped(a, out, g):
    return np.asarray(a).reshape(out, -1, g)


def quantize_fwd(W, s, sr, delta, zu, alpha, zb, codes, g, mode=MAP_LOCAL_PERIODIC, step=0, p=2):
    """UniQuan_F quantizer Q*_IF = D_R o M*_B o T_F (Eq. 3), or Q_IF (Eq. 2).

    W, s: [out, in] (W already as fp32 values); sr: [out]; delta, zu, zb:
    [out, in/g]; alpha: [out, in/g, q]; codes: [out, in] code words (ignored
    for MAP_FULL).  mode MAP_FULL re-maps every element to the nearest of all
    levels (Eq. 2); MAP_LOCAL_PERIODIC applies Algorithm 4 (re-map locally
    when step % p == 0, keep the codes otherwise).

    Returns (w_hat fp32 [out, in], codes uint8 [out, in]).
    """
    out, n_in = np.shape(W)
    Wg = _grouped(np.asarray(W, F32), out, g)
    sg = _grouped(np.asarray(s, F32), out, g)
    lv = levels(alpha, zb)
    srt, cor, roc = sorted_levels(lv)
    if mode == MAP_FULL:
        x, _ = transform_F(Wg, sg, delta, zu, np.asarray(sr)[:, None])
        new = map_full(x, srt, cor)
    elif step % p == 0:
        x, _ = transform_F(Wg, sg, delta, zu, np.asarray(sr)[:, None])
        new = map_local(x, _grouped(codes, out, g).astype(np.int64), srt, cor, roc)
    else:
        new = _grouped(codes, out, g).astype(np.int64)
    what = detransform(reconstruct(new, lv), delta, zu)
    return what.reshape(out, n_in).astype(F32), new.reshape(out, n_in).astype(np.uint8)


# ---------------------------------------------------------------------------
# Backward: straight-through estimator with gradient filtering (App. C.1)
# ---------------------------------------------------------------------------

def _bwd_terms(W, s, sr, delta, zu, alpha, zb, codes, Gup, g, filter_mode=FILTER_STE):
    out, n_in = np.shape(W)
    q = np.shape(alpha)[-1]
    Wg = _grouped(np.asarray(W, F32), out, g)
    sg = _grouped(np.asarray(s, F32), out, g)
    cg = _grouped(codes, out, g).astype(np.int64)
    # fp32 decision: the filter compares |x - w~| with tau = min_j |alpha_j|.
    x32, _ = transform_F(Wg, sg, delta, zu, np.asarray(sr)[:, None])
    m32 = reconstruct(cg, levels(alpha, zb))
    tau = np.min(np.abs(np.asarray(alpha, F32)), axis=-1)
    f = np.abs(x32 - m32) <= tau[..., None]
    # fp64 values.
    W64 = Wg.astype(F64)
    s64 = sg.astype(F64)
    d64 = np.asarray(delta, F64)[..., None]
    zu64 = np.asarray(zu, F64)[..., None]
    sr64 = np.asarray(sr, F64)
    u64 = W64 / (d64 * s64 * sr64[:, None, None])
    C = signs(q, F64)[cg]                                   # [out, Gr, g, q]
    m64 = (C * np.asarray(alpha, F64)[..., None, :]).sum(-1) + np.asarray(zb, F64)[..., None]
    G64 = _grouped(np.asarray(Gup, F64), out, g)
    if filter_mode == FILTER_ELEMENT:
        G64 = np.where(f, G64, 0.0)                         # a filtered element drops out entirely
    gbar = G64 * d64                                        # dL/dw~ = G * Delta
    fu = np.where(f, u64, 0.0)
    return dict(f=f, u=u64, m=m64, zu=zu64, s=s64, sr=sr64, G=G64, gbar=gbar, fu=fu, C=C)


def quantize_bwd(W, s, sr, delta, zu, alpha, zb, codes, Gup, g, filter_mode=FILTER_STE):
    """Gradients of L w.r.t. Theta_IF given G = dL/dW^ (App. C.1, Eq. 3).

    Differentiates w^ = Delta * (w~ - z_U) with
      w~ = c . alpha + z_B                   (codes held fixed),
      dw~/dx = 1 if |x - w~| <= tau else 0   (straight-through estimator,
                                              filtered as in App. C.1),
      x = w / (Delta s s_r) + z_U            (Eq. 1).
    With u = w / (Delta s s_r) and f the filter:
      ds_i    = -G_i Delta f_i u_i / s_i
      dDelta  = sum_i G_i ((w~_i - z_U) - f_i u_i)
      dz_U    = sum_i G_i Delta (f_i - 1)
      dz_B    = sum_i G_i Delta
      dalpha_j= sum_i G_i Delta c_ij
      ds_r    = -sum_{i in row} G_i Delta f_i u_i / s_r
    Filter decisions in fp32, values and sums in fp64.  Returns a dict of
    fp64 arrays shaped like the parameters.

    filter_mode FILTER_STE is the reading above (the filter cuts only the
    straight-through path); FILTER_ELEMENT is the alternative reading in
    which a filtered element drops out of every gradient: G_i is replaced by
    f_i G_i in all the sums (so dz_U is identically zero).
    """
    out, n_in = np.shape(W)
    t = _bwd_terms(W, s, sr, delta, zu, alpha, zb, codes, Gup, g, filter_mode)
    gbar, fu = t["gbar"], t["fu"]
    return dict(
        ds=(-gbar * fu / t["s"]).reshape(out, n_in),
        ddelta=(t["G"] * ((t["m"] - t["zu"]) - fu)).sum(-1),
        dzu=(gbar * (t["f"].astype(F64) - 1.0)).sum(-1),
        dzb=gbar.sum(-1),
        dalpha=(gbar[..., None] * t["C"]).sum(-2),
        dsr=-(gbar * fu).sum(axis=(1, 2)) / t["sr"],
    )


def bwd_l1_mass(W, s, sr, delta, zu, alpha, zb, codes, Gup, g, filter_mode=FILTER_STE):
    """L1 mass sum_i |term_i| of every reduction in quantize_bwd (fp64).

    A summation of n terms in any order cannot be trusted beyond a multiple
    of (unit roundoff) x (sum of |terms|); the parity tests scale their
    tolerance by this mass.  ds gets its own per-element values back.
    """
    t = _bwd_terms(W, s, sr, delta, zu, alpha, zb, codes, Gup, g, filter_mode)
    gbar, fu = t["gbar"], t["fu"]
    q = np.shape(alpha)[-1]
    mass_gbar = np.abs(gbar).sum(-1)
    return dict(
        ddelta=np.abs(t["G"] * ((t["m"] - t["zu"]) - fu)).sum(-1),
        dzu=np.abs(gbar * (t["f"].astype(F64) - 1.0)).sum(-1),
        dzb=mass_gbar,
        dalpha=np.repeat(mass_gbar[..., None], q, axis=-1),
        dsr=np.abs(gbar * fu).sum(axis=(1, 2)) / np.abs(t["sr"]),
    )


# ---------------------------------------------------------------------------
# OmniQuant unified into BCQ (App. E, extensibility): T_O / D_O
# ---------------------------------------------------------------------------

def omni_params(W, beta, gamma, q, g):
    """OmniQuant's learnable clipping as UniQuan's transformation parameters.

    Per group, with w_m and w_M the smallest and largest weight:
      Delta_O = (gamma w_M - beta w_m) / (2^q - 1),
      z_O     = -round(beta w_m / Delta_O)   (round half to even).
    fp32: each product rounded, then the difference, then the division.
    Returns (Delta_O, z_O), fp32 [out, in/g].
    """
    out, n_in = np.shape(W)
    Wg = _grouped(np.asarray(W, F32), out, g)
    wm, wM = Wg.min(-1), Wg.max(-1)
    beta, gamma = np.asarray(beta, F32), np.asarray(gamma, F32)
    num = (gamma * wM).astype(F32) - (beta * wm).astype(F32)
    delta = (num.astype(F32) / F32((1 << q) - 1)).astype(F32)
    zo = -np.rint(((beta * wm).astype(F32) / delta).astype(F32)).astype(F32)
    return delta.astype(F32), zo.astype(F32)


def quantize_fwd_omni(W, beta, gamma, alpha, zb, codes, g, mode=MAP_LOCAL_PERIODIC, step=0, p=2):
    """UniQuan with OmniQuant's maps: D_O(M*_B(T_O(w))) (or M_B with MAP_FULL).

    T_O(w) = w / Delta_O + z_O,  D_O(w~) = Delta_O (w~ - z_O)  (fp32, this
    op order); the mapping and its tie rules are those of quantize_fwd.
    Returns (w_hat fp32 [out, in], codes uint8 [out, in]).
    """
    out, n_in = np.shape(W)
    q = np.shape(alpha)[-1]
    delta, zo = omni_params(W, beta, gamma, q, g)
    Wg = _grouped(np.asarray(W, F32), out, g)
    lv = levels(alpha, zb)
    srt, cor, roc = sorted_levels(lv)
    x = ((Wg / delta[..., None]).astype(F32) + zo[..., None]).astype(F32)
    if mode == MAP_FULL:
        new = map_full(x, srt, cor)
    elif step % p == 0:
        new = map_local(x, _grouped(codes, out, g).astype(np.int64), srt, cor, roc)
    else:
        new = _grouped(codes, out, g).astype(np.int64)
    what = detransform(reconstruct(new, lv), delta, zo)
    return what.reshape(out, n_in).astype(F32), new.reshape(out, n_in).astype(np.uint8)


def _bwd_terms_omni(W, beta, gamma, alpha, zb, codes, Gup, g):
    out, n_in = np.shape(W)
    q = np.shape(alpha)[-1]
    delta, zo = omni_params(W, beta, gamma, q, g)
    Wg = _grouped(np.asarray(W, F32), out, g)
    cg = _grouped(codes, out, g).astype(np.int64)
    x32 = ((Wg / delta[..., None]).astype(F32) + zo[..., None]).astype(F32)
    m32 = reconstruct(cg, levels(alpha, zb))
    tau = np.min(np.abs(np.asarray(alpha, F32)), axis=-1)
    f = np.abs(x32 - m32) <= tau[..., None]
    d64, z64 = delta.astype(F64), zo.astype(F64)
    u = Wg.astype(F64) / d64[..., None]
    C = signs(q, F64)[cg]
    m64 = (C * np.asarray(alpha, F64)[..., None, :]).sum(-1) + np.asarray(zb, F64)[..., None]
    G = _grouped(np.asarray(Gup, F64), out, g)
    fu = np.where(f, u, 0.0)
    wm, wM = Wg.min(-1).astype(F64), Wg.max(-1).astype(F64)
    return dict(f=f, u=u, m=m64, C=C, G=G, fu=fu, d=d64, z=z64, wm=wm, wM=wM,
                beta=np.asarray(beta, F64), L1=float((1 << q) - 1))


def quantize_bwd_omni(W, beta, gamma, alpha, zb, codes, Gup, g):
    """Gradients of L w.r.t. (beta, gamma, alpha, z_B) given G = dL/dW^.

    w^ = Delta_O (w~ - z_O) with w~ = c . alpha + z_B (codes fixed), the
    straight-through path of x = w / Delta_O + z_O filtered as in App. C.1
    (tau = min_j |alpha_j|), and the rounding in z_O passed straight through
    (as OmniQuant trains its zero point).  With u = w / Delta_O:
      A = dL/dDelta_O (z_O held) = sum G ((m - z_O) - f u)
      B = dL/dz_O                = -Delta_O sum G (1 - f)
      dDelta/dbeta = -w_m / (2^q - 1),   dDelta/dgamma = w_M / (2^q - 1)
      dz/dbeta = -(w_m / Delta - beta w_m dDelta/dbeta / Delta^2)
      dz/dgamma = beta w_m dDelta/dgamma / Delta^2
      dbeta = A dDelta/dbeta + B dz/dbeta,  dgamma = A dDelta/dgamma + B dz/dgamma
      dalpha_j = Delta sum G c_j,  dz_B = Delta sum G.
    Decisions in fp32, values and sums in fp64 (dict of fp64 arrays).
    """
    t = _bwd_terms_omni(W, beta, gamma, alpha, zb, codes, Gup, g)
    d, z, G = t["d"], t["z"], t["G"]
    A = (G * ((t["m"] - z[..., None]) - t["fu"])).sum(-1)
    B = -d * (G * (1.0 - t["f"].astype(F64))).sum(-1)
    dDb, dDg = -t["wm"] / t["L1"], t["wM"] / t["L1"]
    dzb_ = -(t["wm"] / d - t["beta"] * t["wm"] * dDb / (d * d))
    dzg_ = t["beta"] * t["wm"] * dDg / (d * d)
    return dict(
        dbeta=A * dDb + B * dzb_, dgamma=A * dDg + B * dzg_,
        dalpha=(d[..., None, None] * G[..., None] * t["C"]).sum(-2), dzb=d * G.sum(-1),
    )


def bwd_l1_mass_omni(W, beta, gamma, alpha, zb, codes, Gup, g):
    """L1 mass of each reduction of quantize_bwd_omni (fp64), for tolerances."""
    t = _bwd_terms_omni(W, beta, gamma, alpha, zb, codes, Gup, g)
    d, z, G = t["d"], t["z"], t["G"]
    mA = np.abs(G * ((t["m"] - z[..., None]) - t["fu"])).sum(-1)
    mB = np.abs(d) * np.abs(G * (1.0 - t["f"].astype(F64))).sum(-1)
    dDb, dDg = -t["wm"] / t["L1"], t["wM"] / t["L1"]
    dzb_ = -(t["wm"] / d - t["beta"] * t["wm"] * dDb / (d * d))
    dzg_ = t["beta"] * t["wm"] * dDg / (d * d)
    q = np.shape(alpha)[-1]
    mG = np.abs(d) * np.abs(G).sum(-1)
    return dict(dbeta=mA * np.abs(dDb) + mB * np.abs(dzb_), dgamma=mA * np.abs(dDg) + mB * np.abs(dzg_),
                dalpha=np.repeat(mG[..., None], q, axis=-1), dzb=mG)


def export_bcq_omni(W, beta, gamma, alpha, zb, codes, g):
    """Theorem 1 for the OmniQuant maps: D_O has the same form as D_R, so
    alpha* = Delta_O alpha and z_B* = Delta_O (z_B - z_O); the stored codes.
    Returns (planes, alpha*, z_B*)."""
    q = np.shape(alpha)[-1]
    delta, zo = omni_params(W, beta, gamma, q, g)
    a_star, z_star = unify(delta, zo, alpha, zb)
    return pack_bitplanes(codes, q), a_star, z_star


# ---------------------------------------------------------------------------
# AWQ unified into BCQ (App. E, extensibility): T_A / D_A
# ---------------------------------------------------------------------------

def quantize_fwd_awq(W, sa, delta, za, alpha, zb, codes, g, mode=MAP_LOCAL_PERIODIC, step=0, p=2):
    """UniQuan with AWQ's maps: D_A(M*_B(T_A(w))) (or M_B with MAP_FULL).

    T_A(w) = (w * s_A) / Delta_A + z_A,  D_A(w~) = Delta_A (w~ - z_A) / s_A,
    s_A [in] one scale per column (shared by every row), Delta_A, z_A per
    group.  (The printed D_A subtracts z_O; it is read as z_A, the zero point
    of T_A.)  fp32, in this order: x = ((w s) / Delta) + z,
    w^ = (Delta (w~ - z)) / s.  Mapping and tie rules as quantize_fwd.
    """
    out, n_in = np.shape(W)
    Wg = _grouped(np.asarray(W, F32), out, g)
    sg = np.broadcast_to(np.asarray(sa, F32).reshape(1, -1, g), Wg.shape)
    delta, za = np.asarray(delta, F32), np.asarray(za, F32)
    lv = levels(alpha, zb)
    srt, cor, roc = sorted_levels(lv)
    x = (((Wg * sg).astype(F32) / delta[..., None]).astype(F32) + za[..., None]).astype(F32)
    if mode == MAP_FULL:
        new = map_full(x, srt, cor)
    elif step % p == 0:
        new = map_local(x, _grouped(codes, out, g).astype(np.int64), srt, cor, roc)
    else:
        new = _grouped(codes, out, g).astype(np.int64)
    wt = reconstruct(new, lv)
    what = ((delta[..., None] * (wt - za[..., None]).astype(F32)).astype(F32) / sg).astype(F32)
    return what.reshape(out, n_in), new.reshape(out, n_in).astype(np.uint8)


def _bwd_terms_awq(W, sa, delta, za, alpha, zb, codes, Gup, g):
    out, n_in = np.shape(W)
    q = np.shape(alpha)[-1]
    Wg = _grouped(np.asarray(W, F32), out, g)
    s32 = np.broadcast_to(np.asarray(sa, F32).reshape(1, -1, g), Wg.shape)
    cg = _grouped(codes, out, g).astype(np.int64)
    x32 = (((Wg * s32).astype(F32) / np.asarray(delta, F32)[..., None]).astype(F32)
           + np.asarray(za, F32)[..., None]).astype(F32)
    m32 = reconstruct(cg, levels(alpha, zb))
    tau = np.min(np.abs(np.asarray(alpha, F32)), axis=-1)
    f = np.abs(x32 - m32) <= tau[..., None]
    d, z = np.asarray(delta, F64)[..., None], np.asarray(za, F64)[..., None]
    s = s32.astype(F64)
    w = Wg.astype(F64)
    u = w * s / d
    C = signs(q, F64)[cg]
    m = (C * np.asarray(alpha, F64)[..., None, :]).sum(-1) + np.asarray(zb, F64)[..., None]
    G = _grouped(np.asarray(Gup, F64), out, g)
    return dict(f=f, fl=f.astype(F64), u=u, m=m, C=C, G=G, d=d, z=z, s=s, w=w)


def quantize_bwd_awq(W, sa, delta, za, alpha, zb, codes, Gup, g):
    """Gradients of L w.r.t. (Delta_A, z_A, s_A, alpha, z_B) given G = dL/dW^.

    w^ = Delta (w~ - z) / s with w~ = c . alpha + z_B (codes fixed) and the
    straight-through path of x = w s / Delta + z filtered as in App. C.1.
    With u = w s / Delta:
      dDelta = sum G ((m - z) - f u) / s
      dz_A   = -Delta sum G (1 - f) / s
      ds_A[col] = sum over the rows of G (f w - Delta (m - z) / s) / s
      dalpha_j = Delta sum G c_j / s,  dz_B = Delta sum G / s.
    Decisions in fp32, values and sums in fp64.
    """
    t = _bwd_terms_awq(W, sa, delta, za, alpha, zb, codes, Gup, g)
    G, s, d, z, m, fl = t["G"], t["s"], t["d"], t["z"], t["m"], t["fl"]
    out, n_in = np.shape(W)
    Gs = G / s
    return dict(
        ddelta=(Gs * ((m - z) - fl * t["u"])).sum(-1),
        dza=-(d[..., 0] * (Gs * (1.0 - fl)).sum(-1)),
        dsa=(Gs * (fl * t["w"] - d * (m - z) / s)).reshape(out, n_in).sum(0),
        dalpha=(d[..., None] * Gs[..., None] * t["C"]).sum(-2), dzb=d[..., 0] * Gs.sum(-1),
    )


def bwd_l1_mass_awq(W, sa, delta, za, alpha, zb, codes, Gup, g):
    """L1 mass of each reduction of quantize_bwd_awq (fp64), for tolerances."""
    t = _bwd_terms_awq(W, sa, delta, za, alpha, zb, codes, Gup, g)
    G, s, d, z, m, fl = t["G"], t["s"], t["d"], t["z"], t["m"], t["fl"]
    out, n_in = np.shape(W)
    q = np.shape(alpha)[-1]
    Gs = np.abs(G / s)
    mg = np.abs(d[..., 0]) * Gs.sum(-1)
    return dict(ddelta=(Gs * np.abs((m - z) - fl * t["u"])).sum(-1), dza=np.abs(d[..., 0]) * (Gs * (1.0 - fl)).sum(-1),
                dsa=(Gs * (np.abs(fl * t["w"]) + np.abs(d * (m - z) / s))).reshape(out, n_in).sum(0),
                dalpha=np.repeat(mg[..., None], q, axis=-1), dzb=mg)


def export_bcq_awq(sa, delta, za, alpha, zb, codes, g):
    """Theorem 1 for the AWQ maps: D_A = D_R followed by the column scale
    1 / s_A, so alpha* = Delta_A alpha, z_B* = Delta_A (z_B - z_A) and the
    column scale stays outside the BCQ weights (AWQ folds 1/s_A into the
    activations: W^ x = (C alpha* + z_B*) (x / s_A)).
    Returns (planes, alpha*, z_B*, 1 / s_A)."""
    q = np.shape(alpha)[-1]
    a_star, z_star = unify(delta, za, alpha, zb)
    inv = (F32(1.0) / np.asarray(sa, F32)).astype(F32)
    return pack_bitplanes(codes, q), a_star, z_star, inv


# ---------------------------------------------------------------------------
# One optimisation step around the quantizer (the inner loop of Algorithm 1)
# ---------------------------------------------------------------------------

LR_F = 0.005     # learning rate of Theta_F = {Delta, z_U, s, s_r} (hyperparameter table, App. C.1)
LR_B = 0.0005    # learning rate of Theta_B = {alpha, z_B} (same table)


def sgd_update(s, sr, delta, zu, alpha, zb, grads, lr_F=LR_F, lr_B=LR_B):
    """Plain SGD on Theta_IF = Theta_F u Theta_B.

    FlexRound trains Theta_F by stochastic gradient descent (Sec. 3.1);
    Algorithm 1 updates Theta_IF once per data point (batch size 1) with one
    learning rate for Theta_F and one for Theta_B (hyperparameter table,
    App. C.1):  theta <- theta - eta * dL/dtheta.  Evaluated in fp64 from
    the fp64 gradients of quantize_bwd, stored as fp32.
    """
    def upd(theta, grad, lr):
        return (np.asarray(theta, F64) - lr * np.asarray(grad, F64)).astype(F32)

    return dict(
        s=upd(s, grads["ds"], lr_F), sr=upd(sr, grads["dsr"], lr_F),
        delta=upd(delta, grads["ddelta"], lr_F), zu=upd(zu, grads["dzu"], lr_F),
        alpha=upd(alpha, grads["dalpha"], lr_B), zb=upd(zb, grads["dzb"], lr_B),
    )


def train_step(W, s, sr, delta, zu, alpha, zb, codes, Gup, g, step, lr_F=LR_F, lr_B=LR_B,
               mode=MAP_LOCAL_PERIODIC, p=2):
    """One pass of Algorithm 1's inner loop as the quantizer sees it.

    `codes` are the codes the forward of step `step` produced and Gup is
    dL/dW^ of that forward.  The step back-propagates Gup (quantize_bwd),
    updates Theta_IF (sgd_update) and quantizes W again for step `step + 1`
    with the updated parameters (quantize_fwd; under M*_B that forward
    remaps only when (step + 1) % p == 0).
    Returns (dict of the updated fp32 parameters, codes and W^ of step + 1).
    """
    grads = quantize_bwd(W, s, sr, delta, zu, alpha, zb, codes, Gup, g)
    new = sgd_update(s, sr, delta, zu, alpha, zb, grads, lr_F, lr_B)
    what, codes1 = quantize_fwd(W, new["s"], new["sr"], new["delta"], new["zu"], new["alpha"], new["zb"],
                                codes, g, mode, step + 1, p)
    return new, codes1, what


# ---------------------------------------------------------------------------
# Export: unification theorem (Theorem 1) and final codes (Eq. 4)
# ---------------------------------------------------------------------------

def unify(delta, zu, alpha, zb):
    """Theorem 1 (proof in App. E.5): alpha* = Delta alpha, z_B* = Delta (z_B - z_U).

    fp32; z_B - z_U is formed first, then scaled.
    """
    delta = np.asarray(delta, F32)
    alpha_star = delta[..., None] * np.asarray(alpha, F32)
    zb_star = delta * (np.asarray(zb, F32) - np.asarray(zu, F32))
    return alpha_star.astype(F32), zb_star.astype(F32)


def codes_eq4(W, alpha_star, zb_star, g):
    """Eq. 4: C = argmin_C' || w - (C' alpha* + z_B*) ||^2, per element.

    Same nearest-level rule as map_full, on the levels of Theta_B* and the
    original weights (no s, no s_r).
    """
    out, n_in = np.shape(W)
    Wg = _grouped(np.asarray(W, F32), out, g)
    srt, cor, _ = sorted_levels(levels(alpha_star, zb_star))
    return map_full(Wg, srt, cor).reshape(out, n_in).astype(np.uint8)


def pack_bitplanes(codes, q):
    """Bit-plane layout of the binary code matrix C (App. F.1: 1 bit per code).

    codes [out, in] uint8 -> planes uint32 [q, out, in/32] with
    bit b of planes[j, r, t] = 1  <=>  c_{j+1} = +1 for column 32 t + b.
    """
    codes = np.asarray(codes, np.uint32)
    out, n_in = codes.shape
    bits = (codes[None, :, :] >> np.arange(q, dtype=np.uint32)[:, None, None]) & 1
    bits = bits.reshape(q, out, n_in // 32, 32)
    weights = (np.uint64(1) << np.arange(32, dtype=np.uint64))
    return (bits.astype(np.uint64) * weights).sum(-1).astype(np.uint32)


def export_bcq_half(W, delta, zu, alpha, zb, codes, g, mode=EXPORT_REUSE_CODES):
    """export_bcq with alpha* and z_B* stored as 16-bit reals (App. F.1 counts
    16 bits per real of Theta_B*): the fp32 values of export_bcq rounded to
    IEEE half precision, nearest even.  Returns (planes, alpha* bits uint16,
    z_B* bits uint16, codes used)."""
    planes, a_s, z_s, c = export_bcq(W, delta, zu, alpha, zb, codes, g, mode)
    return planes, a_s.astype(np.float16).view(np.uint16), z_s.astype(np.float16).view(np.uint16), c


def export_bcq(W, delta, zu, alpha, zb, codes, g, mode=EXPORT_REUSE_CODES):
    """The last two steps of Algorithm 1: Theta_B* by Theorem 1, then the code matrix.

    mode EXPORT_REUSE_CODES keeps the codes of the last quantizer step (for
    which Theorem 1 makes R_B(C; Theta_B*) equal the quantizer output);
    EXPORT_REMAP_EQ4 recomputes them from the original weights by Eq. 4.
    Returns (planes [q, out, in/32] uint32, alpha* [out, in/g, q], z_B*
    [out, in/g], codes used [out, in] uint8).
    """
    q = np.shape(alpha)[-1]
    a_star, z_star = unify(delta, zu, alpha, zb)
    if mode == EXPORT_REMAP_EQ4:
        c = codes_eq4(W, a_star, z_star, g)
    else:
        c = np.asarray(codes, np.uint8)
    return pack_bitplanes(c, q), a_star, z_star, c


# ---------------------------------------------------------------------------
# Deployment: the BCQ product from the exported format
# ---------------------------------------------------------------------------

def bcq_dequantize(planes, alpha_star, zb_star, g, rows=slice(None)):
    """R_B(C; Theta_B*) = C alpha* + z_B* (Sec. 2.3) read back from the
    exported format: bit b of planes[j, r, t] is c_{j+1} = +1 for column
    32 t + b (App. F.1 stores one bit per code and weight).  fp64, [rows, in].
    """
    planes = np.asarray(planes, np.uint32)[:, rows]
    q, out, words = planes.shape
    n_in = words * 32
    bits = (planes[..., None] >> np.arange(32, dtype=np.uint32)) & 1          # [q, out, words, 32]
    c = np.where(bits.reshape(q, out, n_in) == 1, 1.0, -1.0)                 # c_{j+1} per element
    a = np.repeat(np.asarray(alpha_star, F64)[rows], g, axis=1)             # [out, in, q]
    z = np.repeat(np.asarray(zb_star, F64)[rows], g, axis=1)                # [out, in]
    return np.einsum("jri,rij->ri", c, a) + z


def bcq_gemv(planes, alpha_star, zb_star, x, g, row_block=256):
    """y = W~ x for every row x of `x` [batch, in], with W~ = C alpha* + z_B*
    the exported BCQ weights: the product a BCQ inference kernel computes
    (Sec. 2.3; the deployment format of App. F.1).  fp64, [batch, out].

    Each output is the fp64 sum over the row of W~_ri x_i (numpy's sum along
    the contiguous axis, the same for every row); the rows of W~ are
    dequantized `row_block` at a time only to bound the memory.
    """
    x = np.atleast_2d(np.asarray(x, F64))
    out = np.shape(planes)[1]
    y = np.empty((x.shape[0], out), F64)
    for r0 in range(0, out, row_block):
        rows = slice(r0, min(out, r0 + row_block))
        Wt = bcq_dequantize(planes, alpha_star, zb_star, g, rows)
        for b in range(x.shape[0]):
            y[b, rows] = (Wt * x[b][None, :]).sum(-1)
    return y


# ---------------------------------------------------------------------------
# Unified initialization (Algorithm 2, App. E.2 clipping, Algorithm 3)
# ---------------------------------------------------------------------------

def clip_params(wm, wM, gamma, q, strategy=CLIP_FIXED_MIN):
    """Candidate Delta', z'_U for clipping ratio gamma (App. E.2), fp32.

    Delta' = gamma (w_M - w_m) / (2^q - 1) with w_M - w_m floored at 1e-12
    (a constant group would otherwise divide by zero);
      Fixed-minimum:  z'_U = -w_m / Delta'            (T_F(w_m) = 0)
      Fixed-maximum:  z'_U = (2^q - 1) - w_M / Delta'  (T_F(w_M) = 2^q - 1)
      Balanced:       z'_U = -(gamma w_m) / Delta'     (T_F(gamma w_m) = 0)
    """
    wm = np.asarray(wm, F32)
    wM = np.asarray(wM, F32)
    gamma = F32(gamma)
    top = F32((1 << q) - 1)
    rng = np.maximum(wM - wm, F32(1e-12))
    delta = (gamma * rng) / top
    if strategy == CLIP_FIXED_MIN:
        zu = (-wm) / delta
    elif strategy == CLIP_FIXED_MAX:
        zu = top - wM / delta
    elif strategy == CLIP_BALANCED:
        zu = (-(gamma * wm)) / delta
    else:
        raise ValueError(f"unknown clipping strategy {strategy}")
    return delta.astype(F32), zu.astype(F32)


def greedy_init(x, zb, q):
    """Greedy BCQ initialisation used by Algorithm 3 (one bit at a time).

    With r = x - z_B: for j = 1..q, c_j = sign(r) (r >= 0 -> +1),
    alpha_j = mean |r| (fp64 sum, stored fp32), r <- r - c_j alpha_j (fp32).
    x [NG, g] fp32; zb [NG].  Returns (alpha [NG, q] fp32, codes [NG, g]).
    """
    x = np.asarray(x, F32)
    NG, g = x.shape
    r = x - np.asarray(zb, F32)[:, None]
    alpha = np.zeros((NG, q), F32)
    codes = np.zeros((NG, g), np.int64)
    for j in range(q):
        pos = r >= 0
        a = (np.abs(r).astype(F64).sum(-1) / g).astype(F32)
        alpha[:, j] = a
        codes |= pos.astype(np.int64) << j
        r = r - np.where(pos, F32(1), F32(-1)) * a[:, None]
    return alpha, codes


def _sq_err(x64, C, alpha, zb):
    rec = (C * np.asarray(alpha, F64)[:, None, :]).sum(-1) + np.asarray(zb, F64)[:, None]
    return ((x64 - rec) ** 2).sum(-1)


def _int_det(M):
    """Exact determinant of integer matrices M [..., q, q] (Leibniz formula).

    Used only to decide whether C^T C is singular.  C^T C is a Gram matrix of
    +-1 columns, so by Hadamard's inequality |det| <= g^q < 2^63 for g <= 2^15;
    int64 products and sums may wrap but the result is exact modulo 2^64 and
    therefore exact.
    """
    M = np.asarray(M).astype(np.int64)
    q = M.shape[-1]
    total = np.zeros(M.shape[:-2], np.int64)
    with np.errstate(over="ignore"):
        for perm in itertools.permutations(range(q)):
            inversions = sum(1 for a in range(q) for b in range(a + 1, q) if perm[a] > perm[b])
            term = np.ones(M.shape[:-2], np.int64)
            for i, j in enumerate(perm):
                term = term * M[..., i, j]
            total = total - term if inversions % 2 else total + term
    return total


def _solve(A, b):
    """Solves the stacked systems A x = b (fp64): Gaussian elimination with
    partial pivoting (the first largest |pivot| wins), then back substitution;
    every product and difference rounded separately."""
    A = np.array(A, F64)
    b = np.array(b, F64)
    n, q = b.shape
    rows = np.arange(n)
    for k in range(q):
        p = k + np.argmax(np.abs(A[:, k:, k]), axis=1)
        Ak, Ap = A[rows, k].copy(), A[rows, p].copy()
        A[rows, k], A[rows, p] = Ap, Ak
        bk, bp = b[rows, k].copy(), b[rows, p].copy()
        b[rows, k], b[rows, p] = bp, bk
        for i in range(k + 1, q):
            f = A[:, i, k] / A[:, k, k]
            A[:, i, k:] = A[:, i, k:] - f[:, None] * A[:, k, k:]
            b[:, i] = b[:, i] - f * b[:, k]
    xs = np.zeros((n, q), F64)
    for i in range(q - 1, -1, -1):
        acc = b[:, i].copy()
        for j in range(i + 1, q):
            acc = acc - A[:, i, j] * xs[:, j]
        xs[:, i] = acc / A[:, i, i]
    return xs


def general_alternating(x, zb, G, T, q, trace=False):
    """General alternating update (Algorithm 3) on transformed groups x.

    Greedy start, then T rounds of
      alpha <- (C^T C)^{-1} C^T (x - z_B 1)     (fp64 normal equations solved
                                                  by Gaussian elimination; if
                                                  C^T C is singular alpha is
                                                  left unchanged)
      C     <- argmin_C' || x - (C' alpha + z_B 1) ||^2   (= map_full)
      z_B   <- sum_i (x_i - C_i alpha) / g       (only when G == 1)
    alpha and z_B are stored in fp32 after each update.
    x [NG, g]; zb [NG].  Returns (alpha, zb, codes[, errors per round]).
    """
    x = np.asarray(x, F32)
    NG, g = x.shape
    zb = np.array(zb, F32, copy=True).reshape(NG)
    x64 = x.astype(F64)
    S = signs(q, F64)
    alpha, codes = greedy_init(x, zb, q)
    errs = []
    for _ in range(T):
        C = S[codes]                                         # [NG, g, q]
        Ct = C.transpose(0, 2, 1)
        CtC = Ct @ C
        Cty = (Ct @ (x64 - zb.astype(F64)[:, None])[..., None])[..., 0]
        ok = _int_det(np.rint(CtC)) != 0                     # exact integer test
        if ok.any():
            alpha[ok] = _solve(CtC[ok], Cty[ok]).astype(F32)
        srt, cor, _ = sorted_levels(levels(alpha, zb))
        codes = map_full(x, srt, cor)
        if G == 1:
            C = S[codes]
            resid = x64 - (C * alpha.astype(F64)[:, None, :]).sum(-1)
            zb = (resid.sum(-1) / g).astype(F32)
        if trace:
            errs.append(_sq_err(x64, S[codes], alpha, zb))
    if trace:
        return alpha, zb, codes, errs
    return alpha, zb, codes


def init_error(w, delta, zu, alpha, zb):
    """Candidate error of Algorithm 2, e' = ||w - w^||^2 per group (fp64 sum).

    w [NG, g] fp32 groups; delta, zu, zb [NG]; alpha [NG, q].  w^ is the
    quantizer output under these parameters with s = s_r = 1 and the full
    mapping (reading R10): T_F, M_B over all 2^q levels, R_B, D_R.
    """
    w = np.asarray(w, F32)
    NG, g = w.shape
    x, _ = transform_F(w, np.ones((NG, g), F32), np.asarray(delta, F32), np.asarray(zu, F32), np.ones(NG, F32))
    lv = levels(np.asarray(alpha, F32), np.asarray(zb, F32))
    srt, cor, _ = sorted_levels(lv)
    what = detransform(reconstruct(map_full(x, srt, cor), lv), np.asarray(delta, F32), np.asarray(zu, F32))
    return ((w.astype(F64) - what.astype(F64)) ** 2).sum(-1)


def unified_init(W, q, g, G=30, T=15, clip=CLIP_FIXED_MIN, return_errors=False):
    """Unified initialization (Algorithm 2) of every group of W [out, in].

    s = 1, s_r = 1, z_B starts at (2^q - 1)/2.  For gamma = 1/G, 2/G, ..., 1
    (gamma_i = float32(i) / float32(G)): clip (App. E.2) -> T_F -> general
    alternating update (Algorithm 3) -> quantize with the full mapping ->
    e' = ||w - w^||^2 (fp64); a candidate replaces the kept one only when
    e' < e.  The initial codes are the full mapping of T_F(w) under the kept
    parameters (App. E.4: the mapping starts from distances to all levels).

    Returns dict(delta, zu, alpha, zb [per group], s [out, in], sr [out],
    codes [out, in] uint8) and, if return_errors, the per-candidate errors
    [G, NG] and the chosen candidate index per group.
    """
    W = np.asarray(W, F32)
    out, n_in = W.shape
    Gr = n_in // g
    NG = out * Gr
    w = W.reshape(NG, g)
    wm = w.min(-1)
    wM = w.max(-1)
    ones_g = np.ones((NG, g), F32)
    ones_r = np.ones(NG, F32)
    zb = np.full(NG, F32(((1 << q) - 1) / 2), F32)
    best = dict(delta=np.zeros(NG, F32), zu=np.zeros(NG, F32),
                alpha=np.zeros((NG, q), F32), zb=zb.copy())
    e_best = np.full(NG, np.inf)
    chosen = np.full(NG, -1, np.int64)
    all_errs = []
    for i in range(1, G + 1):
        gamma = F32(i) / F32(G)
        d_c, zu_c = clip_params(wm, wM, gamma, q, clip)
        x, _ = transform_F(w, ones_g, d_c, zu_c, ones_r)
        a_c, zb_c, _ = general_alternating(x, best["zb"], G, T, q)
        e = init_error(w, d_c, zu_c, a_c, zb_c)
        all_errs.append(e)
        acc = e < e_best
        best["delta"] = np.where(acc, d_c, best["delta"])
        best["zu"] = np.where(acc, zu_c, best["zu"])
        best["alpha"] = np.where(acc[:, None], a_c, best["alpha"])
        best["zb"] = np.where(acc, zb_c, best["zb"])
        e_best = np.where(acc, e, e_best)
        chosen = np.where(acc, i - 1, chosen)
    x, _ = transform_F(w, ones_g, best["delta"], best["zu"], ones_r)
    srt, cor, _ = sorted_levels(levels(best["alpha"], best["zb"]))
    codes = map_full(x, srt, cor)
    res = dict(
        delta=best["delta"].reshape(out, Gr).astype(F32),
        zu=best["zu"].reshape(out, Gr).astype(F32),
        alpha=best["alpha"].reshape(out, Gr, q).astype(F32),
        zb=best["zb"].reshape(out, Gr).astype(F32),
        s=np.ones((out, n_in), F32),
        sr=np.ones(out, F32),
        codes=codes.reshape(out, n_in).astype(np.uint8),
    )
    if return_errors:
        return res, np.stack(all_errs), chosen.reshape(out, Gr)
    return res


# ---------------------------------------------------------------------------
# Round-to-nearest (Sec. 2.2) -- only used to pin M_B by reduction
# ---------------------------------------------------------------------------

def rtn(w, delta, zu, q):
    """RTN quantizer Q_R (Sec. 2.2): Delta (Clip(round(w/Delta + z_U), 0, 2^q-1) - z_U).

    fp32; round half to even.  Not part of the product: the tests use it to
    pin the full mapping on the uniform BCQ level set.
    """
    w = np.asarray(w, F32)
    delta = np.asarray(delta, F32)[..., None]
    zu = np.asarray(zu, F32)[..., None]
    wt = np.clip(np.rint(w / delta + zu), 0, (1 << q) - 1).astype(F32)
    return delta * (wt - zu)
