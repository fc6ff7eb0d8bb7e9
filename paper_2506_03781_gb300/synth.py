"""Seeded synthetic inputs for the quantizer workloads.

The paper quantizes Llama-3 8B/70B and Mistral 7B weights; none of those
weights (nor C4, GSM8K, MMLU or WikiText2) are available here, so every
workload is a synthetic matrix with the same shape and a heavy-tailed,
outlier-column value distribution.  This module holds only random draws,
dtype casts and the bf16 rounding of stored weights -- none of the
quantizer's arithmetic -- and is the one module that both the CUDA tests and
the CPU oracle tests use for their inputs.

All draws use numpy's PCG64 (``numpy.random.default_rng``) in fp64, then cast
to fp32; bf16 storage rounds the fp32 values to nearest-even.
"""

from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

F32 = np.float32


def bf16_round(x) -> tuple[np.ndarray, np.ndarray]:
    """Round fp32 values to bf16 (nearest-even).

    Returns (raw uint16 bit patterns, the same values widened back to fp32).
    Inputs must be finite.
    """
    x = np.ascontiguousarray(x, F32)
    b = x.view(np.uint32).astype(np.uint64)
    b = b + 0x7FFF + ((b >> 16) & 1)
    hi = ((b >> 16) & 0xFFFF).astype(np.uint16)
    vals = (hi.astype(np.uint32) << 16).view(F32)
    return hi, vals


def _rng(*seed):
    flat = []
    for x in seed:
        flat.extend(np.atleast_1d(x).tolist())
    return np.random.default_rng([int(v) for v in flat])


ROW_BLOCK = 256


def _block_draw(kind: str, out: int, n_in: int, std: float, seed, rows: slice, nu: float = 4.0):
    """Draw rows ``rows`` of an [out, n_in] matrix, one generator per block of
    ROW_BLOCK rows, so any row range costs only the blocks it touches."""
    r0, r1 = rows.start or 0, min(rows.stop if rows.stop is not None else out, out)
    res = np.empty((max(r1 - r0, 0), n_in), F32)
    for b in range(r0 // ROW_BLOCK, (r1 + ROW_BLOCK - 1) // ROW_BLOCK):
        b0, b1 = b * ROW_BLOCK, min((b + 1) * ROW_BLOCK, out)
        rng = _rng(*np.atleast_1d(seed).tolist(), 0, b)
        if kind == "normal":
            blk = rng.standard_normal((b1 - b0, n_in)) * std
        else:
            blk = rng.standard_t(nu, (b1 - b0, n_in)) * (std / np.sqrt(nu / (nu - 2.0)))
        lo, hi = max(b0, r0), min(b1, r1)
        res[lo - r0:hi - r0] = blk[lo - b0:hi - b0].astype(F32)
    return res


def normal_weights(out: int, n_in: int, std: float, seed, rows: slice = slice(None)) -> np.ndarray:
    """W ~ N(0, std^2), fp32."""
    return _block_draw("normal", out, n_in, std, seed, rows)


def student_t_weights(out: int, n_in: int, std: float, nu: float, seed,
                      rows: slice = slice(None)) -> np.ndarray:
    """Student-t(nu) entries scaled to standard deviation std, fp32."""
    return _block_draw("t", out, n_in, std, seed, rows, nu)


def outlier_columns(n_in: int, frac: float, seed) -> np.ndarray:
    """round(frac * n_in) distinct input columns chosen by a seeded permutation."""
    k = int(round(frac * n_in))
    return np.sort(_rng(seed, 1).permutation(n_in)[:k])


def scale_columns(W: np.ndarray, cols: np.ndarray, mult: float) -> np.ndarray:
    W = W.copy()
    W[:, cols] = (W[:, cols].astype(np.float64) * mult).astype(F32)
    return W


def perturb_factors(shapes: dict, eps: float, seed) -> dict:
    """Multipliers 1 + eps * N(0, 1), one independent fp32 array per name.

    Drawn in the order of ``shapes`` from one generator seeded by ``seed``.
    """
    rng = _rng(seed, 7)
    return {k: (1.0 + eps * rng.standard_normal(shp)).astype(F32) for k, shp in shapes.items()}


def upstream_grad(out: int, n_in: int, var: float, seed) -> np.ndarray:
    """dL/dW^ ~ N(0, var), fp32."""
    return (_rng(seed, 3).standard_normal((out, n_in)) * np.sqrt(var)).astype(F32)


@dataclass
class Matrix:
    """One weight matrix of a workload."""
    name: str
    out: int
    n_in: int
    dist: str            # "normal" | "t4"
    std: float
    outlier_frac: float = 0.0
    outlier_mult: float = 1.0


@dataclass
class Workload:
    """A quantizer workload: matrices plus quantizer settings."""
    name: str
    matrices: list
    q: int
    g: int
    wdtype: str          # "f32" | "bf16"
    seed: int
    qs: tuple = ()       # bit-width sweep, if any
    G: int = 30          # grid-search iterations (App. C.1 setting)
    T: int = 15          # alternating iterations
    p: int = 2           # remapping period
    init_eps: float = 0.01     # multiplicative jitter of the initial parameters
    grad_var: float = 1e-4     # variance of dL/dW^
    step_eps: float = 0.0      # per-iteration jitter (stands in for the SGD update)
    iters: int = 1
    notes: str = ""
    extra: dict = field(default_factory=dict)

    @property
    def n_elems(self) -> int:
        return sum(m.out * m.n_in for m in self.matrices)


def _llama3_8b_block():
    mk = lambda n, o, i: Matrix(n, o, i, "t4", 0.02)
    return [mk("q_proj", 4096, 4096), mk("k_proj", 1024, 4096), mk("v_proj", 1024, 4096),
            mk("o_proj", 4096, 4096), mk("gate_proj", 14336, 4096), mk("up_proj", 14336, 4096),
            mk("down_proj", 4096, 14336)]


# Step jitter chosen so that about 0.03 % of the codes move per remap step
# under the local mapping, the per-step rate the paper reports for
# Llama-3 8B (Sec. 3.3, index-change table).
STEP_EPS = 3e-4

WORKLOADS = {
    "mat1k_f32": Workload(
        "mat1k_f32", [Matrix("w", 1024, 1024, "normal", 0.02)], q=3, g=128, wdtype="f32", seed=0,
        notes="1024x1024 fp32 N(0, 0.02^2)"),
    "attn4k_bf16": Workload(
        "attn4k_bf16", [Matrix("w", 4096, 4096, "t4", 0.02, 0.001, 10.0)], q=3, g=128,
        wdtype="bf16", seed=1,
        notes="Llama-3-8B attention projection shape, Student-t(4) std 0.02, 0.1% outlier columns x10"),
    "mlp14336x4096_bf16": Workload(
        "mlp14336x4096_bf16", [Matrix("w", 14336, 4096, "t4", 0.02, 0.001, 10.0)], q=3, g=128,
        wdtype="bf16", seed=2, qs=(2, 3, 4), step_eps=STEP_EPS, iters=100,
        notes="Llama-3-8B MLP shape, Student-t(4) std 0.02, 0.1% outlier columns x10, local mapping p=2"),
    "llama3_8b_block_bf16": Workload(
        "llama3_8b_block_bf16", _llama3_8b_block(), q=2, g=64, wdtype="bf16", seed=3,
        notes="Llama-3-8B block (q,k,v,o,gate,up,down), Student-t(4) std 0.02"),
    "llama2_70b_mlp_bf16": Workload(
        "llama2_70b_mlp_bf16",
        [Matrix("gate_proj", 28672, 8192, "normal", 0.015, 0.0005, 20.0),
         Matrix("up_proj", 28672, 8192, "normal", 0.015, 0.0005, 20.0),
         Matrix("down_proj", 8192, 28672, "normal", 0.015, 0.0005, 20.0)],
        q=3, g=128, wdtype="bf16", seed=4,
        notes="Llama-2-70B MLP shapes, N(0, 0.015^2), 0.05% outlier columns x20"),
}


def matrix_weights(m: Matrix, seed, rows: slice = slice(None)):
    """fp32 values of rows ``rows`` of one matrix (bf16 rounding is the caller's).

    Any row range gives the same values as the same rows of the full draw.
    """
    if m.dist == "normal":
        W = normal_weights(m.out, m.n_in, m.std, seed, rows)
    elif m.dist == "t4":
        W = student_t_weights(m.out, m.n_in, m.std, 4.0, seed, rows)
    else:
        raise ValueError(m.dist)
    if m.outlier_frac > 0:
        W = scale_columns(W, outlier_columns(m.n_in, m.outlier_frac, seed), m.outlier_mult)
    return W


def workload_weights(wl: Workload, index: int = 0, rows: slice = slice(None)):
    """(stored array, fp32 values) of rows ``rows`` of matrix ``index``.

    The stored array is fp32 for wdtype "f32" and raw uint16 bf16 bits for
    "bf16"; the fp32 values are exactly what the stored array holds.
    """
    W = matrix_weights(wl.matrices[index], (wl.seed, index), rows)
    if wl.wdtype == "bf16":
        return bf16_round(W)
    return W, W


def param_shapes(out: int, n_in: int, g: int, q: int) -> dict:
    """Shapes of the multiplicatively jittered parameters (Delta, s, s_r, alpha)."""
    return {"delta": (out, n_in // g), "s": (out, n_in), "sr": (out,), "alpha": (out, n_in // g, q)}


def jitter(params: dict, factors: dict) -> dict:
    """Apply multiplicative jitter factors to a parameter dict (fp32 product)."""
    outp = dict(params)
    for k, f in factors.items():
        outp[k] = (np.asarray(params[k], F32) * f).astype(F32)
    return outp


# ---------------------------------------------------------------------------
# Synthetic decoder block for the reconstruction loop (Algorithm 1)
# ---------------------------------------------------------------------------

@dataclass
class BlockShape:
    """Shape of a Llama-style decoder block: RMSNorm, grouped-query
    attention with rotary position embedding, RMSNorm, SwiGLU MLP.  Only the
    seven linear weights are quantized (norm weights are one)."""
    name: str
    d: int               # hidden size
    heads: int
    kv_heads: int
    head_dim: int
    mlp: int
    seq: int             # tokens per sample
    theta: float = 500000.0
    eps: float = 1e-5

    def matrices(self, std: float = 0.02):
        """The seven linear weights as (name, out, in) Matrix records."""
        qd, kd = self.heads * self.head_dim, self.kv_heads * self.head_dim
        mk = lambda n, o, i: Matrix(n, o, i, "t4", std)
        return [mk("q_proj", qd, self.d), mk("k_proj", kd, self.d), mk("v_proj", kd, self.d),
                mk("o_proj", self.d, qd), mk("gate_proj", self.mlp, self.d), mk("up_proj", self.mlp, self.d),
                mk("down_proj", self.d, self.mlp)]


BLOCKS = {
    # Llama-3-8B block, one calibration sample of 2048 tokens (Sec. 4.1)
    "llama3_8b": BlockShape("llama3_8b", d=4096, heads=32, kv_heads=8, head_dim=128, mlp=14336, seq=2048),
    # small blocks of the same structure, for tests
    "tiny": BlockShape("tiny", d=256, heads=4, kv_heads=2, head_dim=64, mlp=512, seq=16),
    "small": BlockShape("small", d=512, heads=8, kv_heads=2, head_dim=64, mlp=1024, seq=64),
}


def block_weights(shape: BlockShape, seed):
    """fp32 values of the seven weights, bf16-rounded (stored raw bits, values)."""
    out = {}
    for i, m in enumerate(shape.matrices()):
        out[m.name] = bf16_round(matrix_weights(m, (seed, i)))
    return out


def block_inputs(shape: BlockShape, n: int, seed, perturb: float = 0.0):
    """n samples X [seq, d] ~ N(0, 1) (the block's input hidden states) and
    X^ = X (1 + perturb N(0, 1)), standing for the input of the quantized
    block after quantized predecessors (Algorithm 1's X^).  fp32."""
    rng = _rng(seed, 11)
    X = rng.standard_normal((n, shape.seq, shape.d)).astype(F32)
    Xh = (X * (1.0 + perturb * rng.standard_normal(X.shape))).astype(F32)
    return X, Xh
