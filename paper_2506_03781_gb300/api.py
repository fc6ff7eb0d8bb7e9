"""ctypes binding of the C ABI declared in ``include/uq_api.h``.

Same entry-point names as the C library; the only work done here is
argument marshalling (tensor -> device pointer, shape/dtype/device checks so
that no call can hand the kernels a buffer of the wrong size).  Every step of
the quantizer runs in the CUDA library: if ``_build/libuq.so`` is missing,
the first call raises -- there is no other implementation to fall back to.

Tensors are ``torch`` tensors on a CUDA device, contiguous, with the layouts
of the header: W [out, in] fp32 or bf16; s [out, in]; sr [out];
delta, zu, zb [out, in/g]; alpha [out, in/g, q]; codes [out, in] uint8.
"""

from __future__ import annotations

import ctypes
import os

import torch

from .build import LIB

UQ_OK, UQ_ERR_ARG, UQ_ERR_UNSUPPORTED, UQ_ERR_ALIGN, UQ_ERR_CUDA = range(5)
W_F32, W_BF16 = 0, 1
CLIP_FIXED_MIN, CLIP_FIXED_MAX, CLIP_BALANCED = 0, 1, 2
MAP_FULL, MAP_LOCAL_PERIODIC = 0, 1
LR_THETA_F, LR_THETA_B = 0.005, 0.0005     # learning rates of the hyperparameter table (App. C.1)
EXPORT_REUSE_CODES, EXPORT_REMAP_EQ4 = 0, 1
FILTER_STE, FILTER_ELEMENT = 0, 1

PARAM_NAMES = ("delta", "zu", "s", "sr", "alpha", "zb")
OMNI_PARAM_NAMES = ("beta", "gamma", "alpha", "zb")
OMNI_GRAD_NAMES = ("dbeta", "dgamma", "dalpha", "dzb")
AWQ_PARAM_NAMES = ("sa", "delta", "za", "alpha", "zb")
AWQ_GRAD_NAMES = ("dsa", "ddelta", "dza", "dalpha", "dzb")
GRAD_NAMES = ("ddelta", "dzu", "ds", "dsr", "dalpha", "dzb")
ENTRY_POINTS = ("uq_init_params", "uq_quantize_fwd", "uq_quantize_bwd", "uq_train_step", "uq_train_step_bf16",
                "uq_export_bcq",
                "uq_quantize_bwd_ex", "uq_export_bcq_half",
                "uq_quantize_fwd_omni", "uq_quantize_bwd_omni", "uq_omni_scales",
                "uq_quantize_fwd_awq", "uq_quantize_bwd_awq", "uq_awq_bwd_workspace_bytes", "uq_bcq_gemv",
                "uq_bcq_gemv_workspace_bytes", "uq_bcq_gemv_noalloc",
                "uq_check_device", "uq_selftest_wait_timeout", "uq_last_error", "uq_abi_version")


class UQError(RuntimeError):
    """A C entry point returned a non-OK status."""

    def __init__(self, status: int, message: str):
        super().__init__(f"uq status {status}: {message}")
        self.status = status


class uq_params(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in PARAM_NAMES]


class uq_grads(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in GRAD_NAMES]


class uq_params_omni(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in OMNI_PARAM_NAMES]


class uq_grads_omni(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in OMNI_GRAD_NAMES]


class uq_params_awq(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in AWQ_PARAM_NAMES]


class uq_grads_awq(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in AWQ_GRAD_NAMES]


_lib = None


def lib() -> ctypes.CDLL:
    """The loaded C library (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB):
            raise RuntimeError(f"{LIB} is missing: build it with `python -m paper_2506_03781_gb300.build` "
                               "(or __graft_entry__.build()); there is no fallback implementation")
        L = ctypes.CDLL(LIB)
        i64, i32, vp = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p
        L.uq_init_params.argtypes = [vp, i32, i64, i64, i32, i32, i32, i32, i32, uq_params, vp, vp]
        L.uq_quantize_fwd.argtypes = [vp, i32, i64, i64, i32, i32, uq_params, vp, i32, i64, i32, vp, vp]
        L.uq_quantize_bwd.argtypes = [vp, i32, i64, i64, i32, i32, uq_params, vp, vp, uq_grads, vp]
        L.uq_export_bcq.argtypes = [vp, i32, i64, i64, i32, i32, uq_params, vp, i32, vp, vp, vp, vp]
        L.uq_quantize_bwd_ex.argtypes = [vp, i32, i64, i64, i32, i32, uq_params, vp, vp, uq_grads, i32, vp]
        L.uq_export_bcq_half.argtypes = [vp, i32, i64, i64, i32, i32, uq_params, vp, i32, vp, vp, vp, vp]
        L.uq_quantize_fwd_omni.argtypes = [vp, i32, i64, i64, i32, i32, uq_params_omni, vp, i32, i64, i32, vp, vp]
        L.uq_quantize_bwd_omni.argtypes = [vp, i32, i64, i64, i32, i32, uq_params_omni, vp, vp, uq_grads_omni, vp]
        L.uq_omni_scales.argtypes = [vp, i32, i64, i64, i32, i32, vp, vp, vp, vp, vp]
        L.uq_quantize_fwd_awq.argtypes = [vp, i32, i64, i64, i32, i32, uq_params_awq, vp, i32, i64, i32, vp, vp]
        L.uq_quantize_bwd_awq.argtypes = [vp, i32, i64, i64, i32, i32, uq_params_awq, vp, vp, uq_grads_awq, vp, i64,
                                          vp]
        L.uq_awq_bwd_workspace_bytes.argtypes = [i64, i64, i32, i32]
        L.uq_awq_bwd_workspace_bytes.restype = i64
        L.uq_bcq_gemv.argtypes = [vp, vp, vp, i64, i64, i32, i32, vp, i32, i32, vp, vp, i64, vp]
        L.uq_bcq_gemv_workspace_bytes.argtypes = [i64, i64, i32]
        L.uq_bcq_gemv_workspace_bytes.restype = i64
        L.uq_bcq_gemv_noalloc.argtypes = [vp, vp, vp, i64, i64, i32, i32, vp, i32, i32, vp, vp]
        f32 = ctypes.c_float
        L.uq_train_step.argtypes = [vp, i32, i64, i64, i32, i32, uq_params, vp, vp, f32, f32, i32, i64, i32, vp,
                                    vp]
        L.uq_train_step_bf16.argtypes = [vp, i32, i64, i64, i32, i32, uq_params, vp, vp, f32, f32, i32, i64, i32,
                                         vp, vp]
        for name in ("uq_init_params", "uq_quantize_fwd", "uq_quantize_bwd", "uq_export_bcq"):
            getattr(L, name).restype = ctypes.c_int
        L.uq_last_error.argtypes = []
        L.uq_last_error.restype = ctypes.c_char_p
        L.uq_check_device.argtypes = [vp]
        L.uq_check_device.restype = ctypes.c_int
        L.uq_selftest_wait_timeout.argtypes = [vp]
        L.uq_selftest_wait_timeout.restype = ctypes.c_int
        L.uq_abi_version.argtypes = []
        L.uq_abi_version.restype = ctypes.c_int
        _lib = L
    return _lib


def uq_last_error() -> str:
    return lib().uq_last_error().decode()


def uq_abi_version() -> int:
    return lib().uq_abi_version()


def uq_selftest_wait_timeout(stream=None, device=None):
    """Launches the bounded-wait self-test (a wait that runs out after ~8 ms)."""
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else device
    _raise(lib().uq_selftest_wait_timeout(_stream(stream, dev)))


def uq_check_device(stream=None, device=None):
    """Synchronises ``stream`` and raises UQError if a pipelined kernel's
    bounded wait ran out since the last check."""
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else device
    _raise(lib().uq_check_device(_stream(stream, dev)))


# ---------------------------------------------------------------------------
# marshalling helpers
# ---------------------------------------------------------------------------

def _check(t, name, shape, dtype, device):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.device.type != "cuda" or (device is not None and t.device != device):
        raise ValueError(f"{name} must be on {device or 'a CUDA device'} (got {t.device})")
    if t.device.index != torch.cuda.current_device():
        raise ValueError(f"{name} is on {t.device} but the current device is cuda:{torch.cuda.current_device()}; "
                         "the library launches on the current device (call it under torch.cuda.device(...))")
    if tuple(t.shape) != tuple(shape):
        raise ValueError(f"{name} has shape {tuple(t.shape)}, expected {tuple(shape)}")
    if t.dtype != dtype:
        raise ValueError(f"{name} has dtype {t.dtype}, expected {dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _wdtype(W):
    if W.dtype == torch.float32:
        return W_F32
    if W.dtype == torch.bfloat16:
        return W_BF16
    raise ValueError(f"W must be float32 or bfloat16 (got {W.dtype})")


def _stream(stream, device):
    if stream is None:
        return torch.cuda.current_stream(device).cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _params(p, out, n_in, q, g, device, need=PARAM_NAMES):
    Gr = n_in // g
    shapes = {"delta": (out, Gr), "zu": (out, Gr), "s": (out, n_in), "sr": (out,),
              "alpha": (out, Gr, q), "zb": (out, Gr)}
    ptrs = {}
    for n in PARAM_NAMES:
        if n in need:
            ptrs[n] = _check(p[n], f"params['{n}']", shapes[n], torch.float32, device)
        else:
            t = p.get(n) if p is not None else None
            ptrs[n] = _check(t, f"params['{n}']", shapes[n], torch.float32, device) if t is not None else None
    return uq_params(**ptrs)


def _raise(status):
    if status != UQ_OK:
        raise UQError(status, uq_last_error())


def _dims(W, g):
    if W.dim() != 2:
        raise ValueError("W must be 2-D [out, in]")
    return W.shape[0], W.shape[1]


# ---------------------------------------------------------------------------
# entry points
# ---------------------------------------------------------------------------

def uq_init_params(W, q, g, params, codes, G=30, T=15, clip=CLIP_FIXED_MIN, stream=None):
    """Unified initialization (Algorithm 2); writes every tensor of ``params`` and ``codes``."""
    out, n_in = _dims(W, g)
    dev = W.device
    st = lib().uq_init_params(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, G, T, clip,
        _params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev), _stream(stream, dev))
    _raise(st)


def uq_quantize_fwd(W, q, g, params, codes, W_hat, map_mode=MAP_LOCAL_PERIODIC, step=0, p_period=2,
                    stream=None, shape=None, wdtype=None):
    """Quantizer forward Q*_IF (Eq. 3) / Q_IF (Eq. 2) into ``W_hat``; updates ``codes`` on remap steps.

    On a non-remap step of the local mapping W may be None (pass ``shape`` =
    (out, in) and ``wdtype``)."""
    if W is not None:
        out, n_in = _dims(W, g)
        wd, dev, wptr = _wdtype(W), W.device, W.data_ptr()
    else:
        out, n_in = shape
        wd, dev, wptr = (W_BF16 if wdtype is None else wdtype), codes.device, None
    keep = map_mode == MAP_LOCAL_PERIODIC and p_period >= 1 and step % p_period != 0
    need = ("delta", "zu", "alpha", "zb") if keep else PARAM_NAMES
    st = lib().uq_quantize_fwd(
        wptr, wd, out, n_in, q, g, _params(params, out, n_in, q, g, dev, need),
        _check(codes, "codes", (out, n_in), torch.uint8, dev), map_mode, step, p_period,
        _check(W_hat, "W_hat", (out, n_in), torch.float32, dev), _stream(stream, dev))
    _raise(st)


def uq_quantize_bwd(W, q, g, params, codes, dL_dWhat, grads, stream=None):
    """Backward (App. C.1 STE with gradient filtering); overwrites every tensor of ``grads``."""
    out, n_in = _dims(W, g)
    dev = W.device
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    shapes = {"ddelta": (out, Gr), "dzu": (out, Gr), "ds": (out, n_in), "dsr": (out,),
              "dalpha": (out, Gr, q), "dzb": (out, Gr)}
    gp = uq_grads(**{n: _check(grads[n], f"grads['{n}']", shapes[n], torch.float32, dev) for n in GRAD_NAMES})
    st = lib().uq_quantize_bwd(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev),
        _check(dL_dWhat, "dL_dWhat", (out, n_in), torch.float32, dev), gp, _stream(stream, dev))
    _raise(st)


def uq_train_step(W, q, g, params, codes, dL_dWhat, W_hat, step, lr_F=LR_THETA_F, lr_B=LR_THETA_B,
                  map_mode=MAP_LOCAL_PERIODIC, p_period=2, stream=None):
    """Fused step: backward of ``step``, SGD update of ``params`` in place, forward of ``step + 1``.

    ``codes`` holds the codes of the forward of ``step`` on entry and those
    of ``step + 1`` on return; ``W_hat`` receives W^ of ``step + 1``."""
    out, n_in = _dims(W, g)
    dev = W.device
    st = lib().uq_train_step(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev),
        _check(dL_dWhat, "dL_dWhat", (out, n_in), torch.float32, dev), float(lr_F), float(lr_B), map_mode, step,
        p_period, _check(W_hat, "W_hat", (out, n_in), torch.float32, dev), _stream(stream, dev))
    _raise(st)


def uq_train_step_bf16(W, q, g, params, codes, dL_dWhat, W_hat, step, lr_F=LR_THETA_F, lr_B=LR_THETA_B,
                       map_mode=MAP_LOCAL_PERIODIC, p_period=2, stream=None):
    """uq_train_step with bf16 ``dL_dWhat`` (read exactly) and bf16 ``W_hat``
    (W^ of ``step + 1`` rounded to nearest even), for a block computed in bf16."""
    out, n_in = _dims(W, g)
    dev = W.device
    st = lib().uq_train_step_bf16(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev),
        _check(dL_dWhat, "dL_dWhat", (out, n_in), torch.bfloat16, dev), float(lr_F), float(lr_B), map_mode, step,
        p_period, _check(W_hat, "W_hat", (out, n_in), torch.bfloat16, dev), _stream(stream, dev))
    _raise(st)


def uq_quantize_bwd_ex(W, q, g, params, codes, dL_dWhat, grads, filter=FILTER_STE, stream=None):
    """uq_quantize_bwd with a choice of gradient filter (FILTER_STE or FILTER_ELEMENT)."""
    out, n_in = _dims(W, g)
    dev = W.device
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    shapes = {"ddelta": (out, Gr), "dzu": (out, Gr), "ds": (out, n_in), "dsr": (out,),
              "dalpha": (out, Gr, q), "dzb": (out, Gr)}
    gp = uq_grads(**{n: _check(grads[n], f"grads['{n}']", shapes[n], torch.float32, dev) for n in GRAD_NAMES})
    st = lib().uq_quantize_bwd_ex(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev),
        _check(dL_dWhat, "dL_dWhat", (out, n_in), torch.float32, dev), gp, filter, _stream(stream, dev))
    _raise(st)


def uq_export_bcq_half(W, q, g, params, codes, bitplanes, alpha_star, zb_star, mode=EXPORT_REUSE_CODES,
                       stream=None, shape=None, wdtype=None):
    """uq_export_bcq with alpha*, z_B* as IEEE half: ``alpha_star``, ``zb_star`` are torch.float16 tensors."""
    if W is not None:
        out, n_in = _dims(W, g)
        wd, dev, wptr = _wdtype(W), W.device, W.data_ptr()
    else:
        out, n_in = shape if shape is not None else codes.shape
        wd, dev, wptr = (W_BF16 if wdtype is None else wdtype), codes.device, None
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    cptr = _check(codes, "codes", (out, n_in), torch.uint8, dev) if codes is not None else None
    st = lib().uq_export_bcq_half(
        wptr, wd, out, n_in, q, g, _params(params, out, n_in, q, g, dev, ("delta", "zu", "alpha", "zb")),
        cptr, mode, _check(bitplanes, "bitplanes", (q, out, n_in // 32), torch.int32, dev),
        _check(alpha_star, "alpha_star", (out, Gr, q), torch.float16, dev),
        _check(zb_star, "zb_star", (out, Gr), torch.float16, dev), _stream(stream, dev))
    _raise(st)


def uq_export_bcq(W, q, g, params, codes, bitplanes, alpha_star, zb_star, mode=EXPORT_REUSE_CODES,
                  stream=None, shape=None, wdtype=None):
    """Theorem 1 + bit-plane export; writes ``bitplanes`` [q, out, in/32], ``alpha_star``, ``zb_star``."""
    if W is not None:
        out, n_in = _dims(W, g)
        wd, dev, wptr = _wdtype(W), W.device, W.data_ptr()
    else:
        out, n_in = shape if shape is not None else codes.shape
        wd, dev, wptr = (W_BF16 if wdtype is None else wdtype), codes.device, None
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    cptr = _check(codes, "codes", (out, n_in), torch.uint8, dev) if codes is not None else None
    st = lib().uq_export_bcq(
        wptr, wd, out, n_in, q, g, _params(params, out, n_in, q, g, dev, ("delta", "zu", "alpha", "zb")),
        cptr, mode, _check(bitplanes, "bitplanes", (q, out, n_in // 32), torch.int32, dev),
        _check(alpha_star, "alpha_star", (out, Gr, q), torch.float32, dev),
        _check(zb_star, "zb_star", (out, Gr), torch.float32, dev), _stream(stream, dev))
    _raise(st)


def _omni_params(p, out, n_in, q, g, device):
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    shapes = {"beta": (out, Gr), "gamma": (out, Gr), "alpha": (out, Gr, q), "zb": (out, Gr)}
    return uq_params_omni(**{n: _check(p[n], f"params['{n}']", shapes[n], torch.float32, device)
                             for n in OMNI_PARAM_NAMES})


def uq_quantize_fwd_omni(W, q, g, params, codes, W_hat, map_mode=MAP_LOCAL_PERIODIC, step=0, p_period=2,
                         stream=None):
    """UniQuan with OmniQuant's T_O / D_O (params: beta, gamma, alpha, zb) into ``W_hat``."""
    out, n_in = _dims(W, g)
    dev = W.device
    st = lib().uq_quantize_fwd_omni(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _omni_params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev), map_mode, step, p_period,
        _check(W_hat, "W_hat", (out, n_in), torch.float32, dev), _stream(stream, dev))
    _raise(st)


def uq_quantize_bwd_omni(W, q, g, params, codes, dL_dWhat, grads, stream=None):
    """Gradients w.r.t. beta, gamma, alpha, zb of the OmniQuant-unified quantizer."""
    out, n_in = _dims(W, g)
    dev = W.device
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    shapes = {"dbeta": (out, Gr), "dgamma": (out, Gr), "dalpha": (out, Gr, q), "dzb": (out, Gr)}
    gp = uq_grads_omni(**{n: _check(grads[n], f"grads['{n}']", shapes[n], torch.float32, dev)
                          for n in OMNI_GRAD_NAMES})
    st = lib().uq_quantize_bwd_omni(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _omni_params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev),
        _check(dL_dWhat, "dL_dWhat", (out, n_in), torch.float32, dev), gp, _stream(stream, dev))
    _raise(st)


def uq_omni_scales(W, q, g, beta, gamma, delta, zo, stream=None):
    """Delta_O and z_O of every group (for uq_export_bcq with delta/zu = delta/zo)."""
    out, n_in = _dims(W, g)
    dev = W.device
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    st = lib().uq_omni_scales(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _check(beta, "beta", (out, Gr), torch.float32, dev),
        _check(gamma, "gamma", (out, Gr), torch.float32, dev), _check(delta, "delta", (out, Gr), torch.float32, dev),
        _check(zo, "zo", (out, Gr), torch.float32, dev), _stream(stream, dev))
    _raise(st)


def _awq_params(p, out, n_in, q, g, device, need=AWQ_PARAM_NAMES):
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    shapes = {"sa": (n_in,), "delta": (out, Gr), "za": (out, Gr), "alpha": (out, Gr, q), "zb": (out, Gr)}
    return uq_params_awq(**{n: _check(p[n], f"params['{n}']", shapes[n], torch.float32, device)
                            for n in AWQ_PARAM_NAMES})


def uq_quantize_fwd_awq(W, q, g, params, codes, W_hat, map_mode=MAP_LOCAL_PERIODIC, step=0, p_period=2,
                        stream=None):
    """UniQuan with AWQ's T_A / D_A (params: sa [in], delta, za, alpha, zb) into ``W_hat``."""
    out, n_in = _dims(W, g)
    dev = W.device
    st = lib().uq_quantize_fwd_awq(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _awq_params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev), map_mode, step, p_period,
        _check(W_hat, "W_hat", (out, n_in), torch.float32, dev), _stream(stream, dev))
    _raise(st)


def uq_awq_bwd_workspace_bytes(out, n_in, q, g) -> int:
    """Bytes of device workspace uq_quantize_bwd_awq needs on the current device (-1: invalid shape)."""
    return int(lib().uq_awq_bwd_workspace_bytes(out, n_in, q, g))


def uq_quantize_bwd_awq(W, q, g, params, codes, dL_dWhat, grads, workspace=None, stream=None):
    """Gradients w.r.t. sa, delta, za, alpha, zb of the AWQ-unified quantizer (workspace allocated if None)."""
    out, n_in = _dims(W, g)
    dev = W.device
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    shapes = {"dsa": (n_in,), "ddelta": (out, Gr), "dza": (out, Gr), "dalpha": (out, Gr, q), "dzb": (out, Gr)}
    gp = uq_grads_awq(**{n: _check(grads[n], f"grads['{n}']", shapes[n], torch.float32, dev)
                         for n in AWQ_GRAD_NAMES})
    if workspace is None:
        nbytes = uq_awq_bwd_workspace_bytes(out, n_in, q, g)
        workspace = torch.empty(max(nbytes // 4, 4), dtype=torch.float32, device=dev)
    st = lib().uq_quantize_bwd_awq(
        W.data_ptr(), _wdtype(W), out, n_in, q, g, _awq_params(params, out, n_in, q, g, dev),
        _check(codes, "codes", (out, n_in), torch.uint8, dev),
        _check(dL_dWhat, "dL_dWhat", (out, n_in), torch.float32, dev), gp, workspace.data_ptr(),
        workspace.numel() * 4, _stream(stream, dev))
    _raise(st)


def uq_bcq_gemv_workspace_bytes(out, n_in, batch=1) -> int:
    """Bytes of device workspace uq_bcq_gemv needs (-1 for an invalid shape)."""
    return int(lib().uq_bcq_gemv_workspace_bytes(out, n_in, batch))


def bcq_gemv_workspace(out, n_in, batch=1, device="cuda"):
    """A workspace tensor large enough for uq_bcq_gemv on this shape."""
    nbytes = uq_bcq_gemv_workspace_bytes(out, n_in, batch)
    if nbytes < 0:
        raise ValueError(f"invalid shape for the BCQ product: out={out} in={n_in} batch={batch}")
    return torch.empty(max(nbytes // 4, 4), dtype=torch.float32, device=device)


def uq_bcq_gemv(bitplanes, alpha_star, zb_star, x, y, g, workspace=None, stream=None):
    """BCQ product y = W~ x from the exported format (``bitplanes`` int32 [q, out, in/32],
    ``alpha_star`` [out, in/g, q], ``zb_star`` [out, in/g]); x [batch, in] fp32/bf16, y [batch, out] fp32.
    ``workspace``: a float32 device tensor of at least uq_bcq_gemv_workspace_bytes bytes
    (allocated here when None)."""
    if bitplanes.dim() != 3 or x.dim() != 2:
        raise ValueError("bitplanes must be [q, out, in/32] and x [batch, in]")
    q, out, words = bitplanes.shape
    batch, n_in = x.shape
    if n_in != 32 * words:
        raise ValueError(f"x has {n_in} columns, the planes {32 * words}")
    dev = x.device
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    if workspace is None:
        workspace = bcq_gemv_workspace(out, n_in, batch, dev)
    if workspace.dtype != torch.float32 or workspace.device != dev or not workspace.is_contiguous():
        raise ValueError("workspace must be a contiguous float32 tensor on the device of x")
    st = lib().uq_bcq_gemv(
        _check(bitplanes, "bitplanes", (q, out, words), torch.int32, dev),
        _check(alpha_star, "alpha_star", (out, Gr, q), torch.float32, dev),
        _check(zb_star, "zb_star", (out, Gr), torch.float32, dev), out, n_in, q, g,
        _check(x, "x", (batch, n_in), x.dtype, dev), _wdtype(x), batch,
        _check(y, "y", (batch, out), torch.float32, dev), workspace.data_ptr(), workspace.numel() * 4,
        _stream(stream, dev))
    _raise(st)


def uq_bcq_gemv_noalloc(bitplanes, alpha_star, zb_star, x, y, g, stream=None):
    """The BCQ product of uq_bcq_gemv without a workspace: for callers that
    cannot allocate device memory, it uses 4 MiB of scratch built into the
    library (shared by all calls; calls that overlap on the GPU race on it).
    Larger shapes raise UQError (UQ_ERR_UNSUPPORTED)."""
    if bitplanes.dim() != 3 or x.dim() != 2:
        raise ValueError("bitplanes must be [q, out, in/32] and x [batch, in]")
    q, out, words = bitplanes.shape
    batch, n_in = x.shape
    if n_in != 32 * words:
        raise ValueError(f"x has {n_in} columns, the planes {32 * words}")
    dev = x.device
    Gr = n_in // g if g > 0 and n_in % g == 0 else 0
    st = lib().uq_bcq_gemv_noalloc(
        _check(bitplanes, "bitplanes", (q, out, words), torch.int32, dev),
        _check(alpha_star, "alpha_star", (out, Gr, q), torch.float32, dev),
        _check(zb_star, "zb_star", (out, Gr), torch.float32, dev), out, n_in, q, g,
        _check(x, "x", (batch, n_in), x.dtype, dev), _wdtype(x), batch,
        _check(y, "y", (batch, out), torch.float32, dev), _stream(stream, dev))
    _raise(st)


class RowSlabs:
    """Several weight matrices quantized with one launch per input width.

    Rows are independent (groups lie inside rows and s_r is per row), so the
    matrices that share a number of columns are stored as consecutive row
    ranges of one slab: W, Theta_IF, the codes, W^, dL/dW^ (and, on request,
    the gradients and the export outputs) are one [sum of rows, in] tensor
    per width, and every matrix's tensors are row views into them.  One call
    per width then runs the forward, backward, fused step or export of all
    its matrices with the persistent grid filled (a Llama-3-8B block's
    1024-row k and v projections alone would leave most of the GPU idle),
    and the results are bit for bit those of one call per matrix.  The views
    of a matrix start on 16-byte boundaries when every matrix before it in
    the slab has a multiple of 4 rows (true of the model shapes).

    shapes: {name: (out, in)} in the order the matrices are laid out.
    """

    def __init__(self, shapes, q, g, w_dtype=torch.bfloat16, device="cuda", with_grads=True, with_export=False):
        self.q, self.g, self.device = q, g, torch.device(device)
        self.rows, widths = {}, {}
        for name, (out, n_in) in shapes.items():
            r0 = widths.get(n_in, 0)
            self.rows[name] = (n_in, r0, r0 + out)
            widths[n_in] = r0 + out
        self.slabs = {}
        for n_in, total in widths.items():
            d = {"W": torch.empty(total, n_in, dtype=w_dtype, device=self.device),
                 "params": empty_params(total, n_in, q, g, self.device),
                 "codes": torch.empty(total, n_in, dtype=torch.uint8, device=self.device),
                 "W_hat": torch.empty(total, n_in, dtype=torch.float32, device=self.device),
                 "dL_dWhat": torch.zeros(total, n_in, dtype=torch.float32, device=self.device),
                 "grads": empty_grads(total, n_in, q, g, self.device) if with_grads else None}
            if with_export:
                d["export"] = (torch.empty(q, total, n_in // 32, dtype=torch.int32, device=self.device),
                               torch.empty(total, n_in // g, q, dtype=torch.float32, device=self.device),
                               torch.empty(total, n_in // g, dtype=torch.float32, device=self.device))
            d["qz"] = Quantizer(d["W"], q, g, d["params"], d["codes"], d["W_hat"], d["dL_dWhat"], d["grads"])
            self.slabs[n_in] = d

    def view(self, name):
        """The matrix's tensors: row views of its slab (W, params, codes,
        W_hat, dL_dWhat, grads, export)."""
        n_in, r0, r1 = self.rows[name]
        d = self.slabs[n_in]
        v = {k: d[k][r0:r1] for k in ("W", "codes", "W_hat", "dL_dWhat")}
        v["params"] = {k: t[r0:r1] for k, t in d["params"].items()}
        v["grads"] = None if d["grads"] is None else {k: t[r0:r1] for k, t in d["grads"].items()}
        if "export" in d:
            planes, a_s, z_s = d["export"]
            v["export"] = (planes[:, r0:r1], a_s[r0:r1], z_s[r0:r1])
        return v

    def init_params(self, G=30, T=15, clip=CLIP_FIXED_MIN, stream=None):
        """Unified initialization of every matrix (one call per width)."""
        for d in self.slabs.values():
            uq_init_params(d["W"], self.q, self.g, d["params"], d["codes"], G=G, T=T, clip=clip, stream=stream)

    def fwd(self, step, p_period=2, map_mode=MAP_LOCAL_PERIODIC, stream=None):
        for d in self.slabs.values():
            d["qz"].fwd(step, p_period, map_mode, stream)

    def bwd(self, stream=None):
        for d in self.slabs.values():
            d["qz"].bwd(stream)

    def train_step(self, step, lr_F=LR_THETA_F, lr_B=LR_THETA_B, p_period=2, map_mode=MAP_LOCAL_PERIODIC,
                   stream=None):
        for d in self.slabs.values():
            d["qz"].train_step(step, lr_F, lr_B, p_period, map_mode, stream)

    def export(self, mode=EXPORT_REUSE_CODES, stream=None):
        for d in self.slabs.values():
            d["qz"].export(*d["export"], mode=mode, stream=stream)


# ---------------------------------------------------------------------------
# buffer helpers
# ---------------------------------------------------------------------------

def empty_params(out, n_in, q, g, device="cuda"):
    Gr = n_in // g
    f = dict(dtype=torch.float32, device=device)
    return {"delta": torch.empty(out, Gr, **f), "zu": torch.empty(out, Gr, **f), "s": torch.empty(out, n_in, **f),
            "sr": torch.empty(out, **f), "alpha": torch.empty(out, Gr, q, **f), "zb": torch.empty(out, Gr, **f)}


def empty_grads(out, n_in, q, g, device="cuda"):
    Gr = n_in // g
    f = dict(dtype=torch.float32, device=device)
    return {"ddelta": torch.empty(out, Gr, **f), "dzu": torch.empty(out, Gr, **f),
            "ds": torch.empty(out, n_in, **f), "dsr": torch.empty(out, **f),
            "dalpha": torch.empty(out, Gr, q, **f), "dzb": torch.empty(out, Gr, **f)}


def weights_tensor(stored, device="cuda"):
    """Device tensor from a stored numpy weight array (fp32, or uint16 bf16 bits)."""
    import numpy as np
    if stored.dtype == np.uint16:
        return torch.from_numpy(stored.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(stored, np.float32)).to(device)


class HostStep:
    """One quantizer optimisation step on HOST buffers, through the C ABI.

    ``run`` copies the step's inputs (W, the six parameter tensors, the code
    words and dL/dW^) from host tensors -- pinned, for asynchronous copies --
    into device buffers owned by this object, runs ``uq_quantize_fwd`` and
    ``uq_quantize_bwd`` on the device, and copies the results (W^, the new
    code words and the six gradients) back into host tensors.  All work is
    queued on ``stream``; ``run`` returns without synchronising.
    """

    IN_KEYS = ("W",) + PARAM_NAMES + ("codes", "dL_dWhat")
    OUT_KEYS = ("W_hat", "codes") + GRAD_NAMES

    def __init__(self, out, n_in, q, g, w_dtype=torch.bfloat16, device="cuda", stream=None):
        self.out, self.n_in, self.q, self.g = out, n_in, q, g
        self.device = torch.device(device)
        self.stream = stream or torch.cuda.Stream(self.device)
        d = self.device
        self.dev = {"W": torch.empty(out, n_in, dtype=w_dtype, device=d),
                    "codes": torch.empty(out, n_in, dtype=torch.uint8, device=d),
                    "dL_dWhat": torch.empty(out, n_in, dtype=torch.float32, device=d),
                    "W_hat": torch.empty(out, n_in, dtype=torch.float32, device=d)}
        self.params = empty_params(out, n_in, q, g, d)
        self.grads = empty_grads(out, n_in, q, g, d)

    def empty_host(self, pinned=True):
        """Host tensors of the right shapes for ``run``'s inputs and outputs."""
        mk = lambda t: torch.empty(t.shape, dtype=t.dtype, pin_memory=pinned)
        ins = {"W": mk(self.dev["W"]), "codes": mk(self.dev["codes"]), "dL_dWhat": mk(self.dev["dL_dWhat"])}
        ins.update({k: mk(v) for k, v in self.params.items()})
        outs = {"W_hat": mk(self.dev["W_hat"]), "codes": mk(self.dev["codes"])}
        outs.update({k: mk(v) for k, v in self.grads.items()})
        return ins, outs

    def bytes_in(self, host_in):
        return sum(host_in[k].numel() * host_in[k].element_size() for k in self.IN_KEYS)

    def bytes_out(self, host_out):
        return sum(host_out[k].numel() * host_out[k].element_size() for k in self.OUT_KEYS)

    def run(self, host_in, host_out, step, p_period=2, map_mode=MAP_LOCAL_PERIODIC):
        dev = {**self.dev, **self.params}
        with torch.cuda.stream(self.stream):
            for k in self.IN_KEYS:
                dev[k].copy_(host_in[k], non_blocking=True)
            uq_quantize_fwd(self.dev["W"], self.q, self.g, self.params, self.dev["codes"], self.dev["W_hat"],
                            map_mode, step, p_period, stream=self.stream)
            uq_quantize_bwd(self.dev["W"], self.q, self.g, self.params, self.dev["codes"], self.dev["dL_dWhat"],
                            self.grads, stream=self.stream)
            host_out["W_hat"].copy_(self.dev["W_hat"], non_blocking=True)
            host_out["codes"].copy_(self.dev["codes"], non_blocking=True)
            for k in GRAD_NAMES:
                host_out[k].copy_(self.grads[k], non_blocking=True)


class HostPipeline:
    """Overlapped quantizer steps on HOST buffers, through the C ABI.

    ``submit`` queues one step: the host-to-device copies of its inputs on an
    upload stream, ``uq_quantize_fwd`` + ``uq_quantize_bwd`` on a compute
    stream and the device-to-host copies of its results on a download
    stream, ordered by CUDA events.  ``depth`` device buffer sets are used in
    turn, so a step's uploads overlap the previous steps' compute and
    downloads (the two copy directions run concurrently).  Steps submitted
    back to back must be independent -- e.g. different weight matrices of a
    model -- because a step's host inputs are read when its upload starts.
    Host tensors should be pinned; ``synchronize`` waits for every step.
    """

    def __init__(self, out, n_in, q, g, w_dtype=torch.bfloat16, device="cuda", depth=2):
        self.steps = [HostStep(out, n_in, q, g, w_dtype, device, stream=None) for _ in range(depth)]
        dev = torch.device(device)
        self.up = torch.cuda.Stream(dev)
        self.comp = torch.cuda.Stream(dev)
        self.down = torch.cuda.Stream(dev)
        self.ev = [{k: torch.cuda.Event() for k in ("up", "comp", "down")} for _ in range(depth)]
        self.n = 0

    def empty_host(self, pinned=True):
        return self.steps[0].empty_host(pinned)

    def bytes_in(self, host_in):
        return self.steps[0].bytes_in(host_in)

    def bytes_out(self, host_out):
        return self.steps[0].bytes_out(host_out)

    def submit(self, host_in, host_out, step, p_period=2, map_mode=MAP_LOCAL_PERIODIC):
        k = self.n % len(self.steps)
        hs, ev = self.steps[k], self.ev[k]
        dev = {**hs.dev, **hs.params}
        # inputs of this buffer set are free once the compute that read them is done
        self.up.wait_event(ev["comp"])
        with torch.cuda.stream(self.up):
            for name in HostStep.IN_KEYS:
                dev[name].copy_(host_in[name], non_blocking=True)
        ev["up"].record(self.up)
        # outputs of this buffer set are free once their download is done
        self.comp.wait_event(ev["up"])
        self.comp.wait_event(ev["down"])
        uq_quantize_fwd(hs.dev["W"], hs.q, hs.g, hs.params, hs.dev["codes"], hs.dev["W_hat"], map_mode, step,
                        p_period, stream=self.comp)
        uq_quantize_bwd(hs.dev["W"], hs.q, hs.g, hs.params, hs.dev["codes"], hs.dev["dL_dWhat"], hs.grads,
                        stream=self.comp)
        ev["comp"].record(self.comp)
        self.down.wait_event(ev["comp"])
        with torch.cuda.stream(self.down):
            host_out["W_hat"].copy_(hs.dev["W_hat"], non_blocking=True)
            host_out["codes"].copy_(hs.dev["codes"], non_blocking=True)
            for name in GRAD_NAMES:
                host_out[name].copy_(hs.grads[name], non_blocking=True)
        ev["down"].record(self.down)
        self.n += 1

    def synchronize(self):
        self.down.synchronize()


class Quantizer:
    """Pre-validated buffers of one weight matrix, for repeated steps.

    Checks every tensor once at construction (shapes, dtypes, device,
    contiguity, the same checks as the functions above) and keeps the C
    argument structures, so ``fwd``/``bwd``/``export`` are single C calls.
    That matters for small matrices, whose kernels are shorter than the
    per-call marshalling, and for capturing a whole step in a CUDA graph.
    ``stream`` (a torch.cuda.Stream or raw handle) defaults to the current
    stream at call time.
    """

    def __init__(self, W, q, g, params, codes, W_hat, dL_dWhat, grads=None):
        self.W, self.q, self.g = W, q, g
        self.out, self.n_in = _dims(W, g)
        self.wd = _wdtype(W)
        dev = W.device
        self.device = dev
        self.keep = (params, codes, W_hat, dL_dWhat, grads)       # keep the tensors alive
        self.p = _params(params, self.out, self.n_in, q, g, dev)
        self.codes = _check(codes, "codes", (self.out, self.n_in), torch.uint8, dev)
        self.what = _check(W_hat, "W_hat", (self.out, self.n_in), torch.float32, dev)
        self.G = _check(dL_dWhat, "dL_dWhat", (self.out, self.n_in), torch.float32, dev)
        Gr = self.n_in // g
        shapes = {"ddelta": (self.out, Gr), "dzu": (self.out, Gr), "ds": (self.out, self.n_in),
                  "dsr": (self.out,), "dalpha": (self.out, Gr, q), "dzb": (self.out, Gr)}
        # grads may be None when only the fused train_step is used (it writes no gradients)
        self.gr = None if grads is None else uq_grads(
            **{n: _check(grads[n], f"grads['{n}']", shapes[n], torch.float32, dev) for n in GRAD_NAMES})
        self.wptr = W.data_ptr()
        self.L = lib()

    def _st(self, stream):
        if self.device.index != torch.cuda.current_device():
            raise ValueError(f"this Quantizer's tensors are on {self.device} but the current device is "
                             f"cuda:{torch.cuda.current_device()} (call it under torch.cuda.device(...))")
        return _stream(stream, self.device)

    def fwd(self, step, p_period=2, map_mode=MAP_LOCAL_PERIODIC, stream=None):
        _raise(self.L.uq_quantize_fwd(self.wptr, self.wd, self.out, self.n_in, self.q, self.g, self.p, self.codes,
                                      map_mode, step, p_period, self.what, self._st(stream)))

    def bwd(self, stream=None):
        if self.gr is None:
            raise ValueError("this Quantizer was built without gradient buffers")
        _raise(self.L.uq_quantize_bwd(self.wptr, self.wd, self.out, self.n_in, self.q, self.g, self.p, self.codes,
                                      self.G, self.gr, self._st(stream)))

    def train_step(self, step, lr_F=LR_THETA_F, lr_B=LR_THETA_B, p_period=2, map_mode=MAP_LOCAL_PERIODIC,
                   stream=None):
        """Fused backward of ``step`` + SGD update + forward of ``step + 1`` (uq_train_step)."""
        _raise(self.L.uq_train_step(self.wptr, self.wd, self.out, self.n_in, self.q, self.g, self.p, self.codes,
                                    self.G, float(lr_F), float(lr_B), map_mode, step, p_period, self.what,
                                    self._st(stream)))

    def export(self, bitplanes, alpha_star, zb_star, mode=EXPORT_REUSE_CODES, stream=None):
        Gr = self.n_in // self.g
        _raise(self.L.uq_export_bcq(
            self.wptr, self.wd, self.out, self.n_in, self.q, self.g, self.p, self.codes, mode,
            _check(bitplanes, "bitplanes", (self.q, self.out, self.n_in // 32), torch.int32, self.device),
            _check(alpha_star, "alpha_star", (self.out, Gr, self.q), torch.float32, self.device),
            _check(zb_star, "zb_star", (self.out, Gr), torch.float32, self.device), self._st(stream)))
