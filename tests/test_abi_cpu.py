"""Host-side checks of the C ABI that need no GPU.

* the library builds and exports every function declared in include/*.h;
* argument validation rejects bad calls before anything is launched, with
  the documented status codes and a message;
* the oracle and the product package do not import each other.

The validation tests hand the library fake (but aligned, non-null) pointers,
so they only run where no CUDA device is present: every case must be
rejected by validation, and on a CPU-only machine even a validation bug could
only produce UQ_ERR_CUDA, never touch memory.
"""

import ctypes
import glob
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def libpath():
    from paper_2506_03781_gb300 import build
    return build.build()


def declared_functions():
    names = []
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        txt = re.sub(r"/\*.*?\*/", "", open(h).read(), flags=re.S)
        names += re.findall(r"^\s*(?:const\s+)?[a-z_0-9]+\s*\*?\s*(uq_[a-z_0-9]+)\s*\(", txt, flags=re.M)
    return sorted(set(names))


def test_header_declares_the_abi():
    names = declared_functions()
    for n in ("uq_init_params", "uq_quantize_fwd", "uq_quantize_bwd", "uq_export_bcq", "uq_last_error"):
        assert n in names


def test_library_exports_every_declared_symbol(libpath):
    lib = ctypes.CDLL(libpath)
    for n in declared_functions():
        assert hasattr(lib, n), n
    from paper_2506_03781_gb300 import api
    assert set(api.ENTRY_POINTS) == set(declared_functions())
    assert api.uq_abi_version() == 1
    assert api.uq_last_error() == ""


def _no_gpu():
    try:
        import torch
        return not torch.cuda.is_available()
    except Exception:
        return True


cpu_only = pytest.mark.skipif(not _no_gpu(), reason="fake-pointer validation tests run only without a GPU")

FAKE = 0x7f0000000000          # 16-byte aligned, never dereferenced


def _params(api, **over):
    d = {n: FAKE + 0x1000 * i for i, n in enumerate(api.PARAM_NAMES)}
    d.update(over)
    return api.uq_params(**d)


def _grads(api, **over):
    d = {n: FAKE + 0x100000 + 0x1000 * i for i, n in enumerate(api.GRAD_NAMES)}
    d.update(over)
    return api.uq_grads(**d)


@cpu_only
@pytest.mark.parametrize("case,expect", [
    (dict(q=0), "UNSUPPORTED"), (dict(q=5), "UNSUPPORTED"),
    (dict(g=48), "ARG"), (dict(g=16), "ARG"), (dict(g=96, n_in=384), "UNSUPPORTED"),
    (dict(n_in=200), "ARG"), (dict(out=0), "ARG"), (dict(n_in=0), "ARG"),
    (dict(n_in=(1 << 24) + 128, g=128), "UNSUPPORTED"),
    (dict(wd=7), "ARG"), (dict(map_mode=3), "ARG"), (dict(p_period=0), "ARG"), (dict(step=-1), "ARG"),
    (dict(W=0), "ARG"), (dict(W=FAKE + 8), "ALIGN"), (dict(what=0), "ARG"), (dict(codes=FAKE + 4), "ALIGN"),
    (dict(params=dict(delta=0)), "ARG"), (dict(params=dict(alpha=FAKE + 2)), "ALIGN"),
])
def test_fwd_validation(libpath, case, expect):
    from paper_2506_03781_gb300 import api
    a = dict(W=FAKE, wd=api.W_BF16, out=8, n_in=256, q=3, g=128, codes=FAKE + 0x9000, map_mode=1, step=0,
             p_period=2, what=FAKE + 0xA000)
    a.update({k: v for k, v in case.items() if k != "params"})
    p = _params(api, **case.get("params", {}))
    st = api.lib().uq_quantize_fwd(a["W"], a["wd"], a["out"], a["n_in"], a["q"], a["g"], p, a["codes"],
                                   a["map_mode"], a["step"], a["p_period"], a["what"], None)
    assert st == getattr(api, "UQ_ERR_" + expect), (st, api.uq_last_error())
    assert api.uq_last_error() != ""


@cpu_only
def test_fwd_keep_step_does_not_need_weights(libpath):
    """On a non-remap local step W, s and s_r are not read, so NULL is accepted
    by validation (on this GPU-less machine the launch itself then fails)."""
    from paper_2506_03781_gb300 import api
    p = _params(api, s=0, sr=0)
    st = api.lib().uq_quantize_fwd(0, api.W_BF16, 8, 256, 3, 128, p, FAKE + 0x9000, 1, 1, 2, FAKE + 0xA000, None)
    assert st == api.UQ_ERR_CUDA
    assert "uq_quantize_fwd" in api.uq_last_error()


@cpu_only
@pytest.mark.parametrize("field", ["ddelta", "dzu", "ds", "dsr", "dalpha", "dzb"])
def test_bwd_validation_each_grad(libpath, field):
    from paper_2506_03781_gb300 import api
    st = api.lib().uq_quantize_bwd(FAKE, api.W_BF16, 8, 256, 3, 128, _params(api), FAKE + 0x9000,
                                   FAKE + 0xB000, _grads(api, **{field: 0}), None)
    assert st == api.UQ_ERR_ARG and field in api.uq_last_error()


@cpu_only
def test_export_and_init_validation(libpath):
    from paper_2506_03781_gb300 import api
    L = api.lib()
    # export: unknown mode, EQ4 without W, REUSE without codes, misaligned planes
    assert L.uq_export_bcq(FAKE, 1, 8, 256, 3, 128, _params(api), FAKE, 9, FAKE, FAKE, FAKE, None) == api.UQ_ERR_ARG
    assert L.uq_export_bcq(0, 1, 8, 256, 3, 128, _params(api), FAKE, 1, FAKE, FAKE, FAKE, None) == api.UQ_ERR_ARG
    assert L.uq_export_bcq(FAKE, 1, 8, 256, 3, 128, _params(api), 0, 0, FAKE, FAKE, FAKE, None) == api.UQ_ERR_ARG
    assert L.uq_export_bcq(FAKE, 1, 8, 256, 3, 128, _params(api), FAKE, 0, FAKE + 4, FAKE, FAKE,
                           None) == api.UQ_ERR_ALIGN
    # init: G < 1, T < 0, bad clip, g too large, missing s
    assert L.uq_init_params(FAKE, 1, 8, 256, 3, 128, 0, 15, 0, _params(api), FAKE, None) == api.UQ_ERR_ARG
    assert L.uq_init_params(FAKE, 1, 8, 256, 3, 128, 30, -1, 0, _params(api), FAKE, None) == api.UQ_ERR_ARG
    assert L.uq_init_params(FAKE, 1, 8, 256, 3, 128, 30, 15, 5, _params(api), FAKE, None) == api.UQ_ERR_ARG
    assert L.uq_init_params(FAKE, 1, 1, 65536, 3, 65536, 30, 15, 0, _params(api), FAKE,
                            None) == api.UQ_ERR_UNSUPPORTED
    assert L.uq_init_params(FAKE, 1, 8, 256, 3, 128, 30, 15, 0, _params(api, s=0), FAKE, None) == api.UQ_ERR_ARG


@cpu_only
@pytest.mark.parametrize("case,expect", [
    (dict(q=5), "UNSUPPORTED"), (dict(n_in=200), "ARG"), (dict(map_mode=2), "ARG"), (dict(p_period=0), "ARG"),
    (dict(step=-1), "ARG"), (dict(step=(1 << 63) - 1), "ARG"),
    # shapes the fused kernel does not take: group sizes outside {32, 64, 128}, ragged units, rows over 64 units
    (dict(g=256, n_in=512), "UNSUPPORTED"), (dict(n_in=384), "UNSUPPORTED"), (dict(g=32, n_in=384), "UNSUPPORTED"),
    (dict(n_in=32768 + 512), "UNSUPPORTED"), (dict(g=32, n_in=16384 + 256), "UNSUPPORTED"),
    (dict(W=0), "ARG"), (dict(gup=0), "ARG"), (dict(gup=FAKE + 4), "ALIGN"), (dict(what=0), "ARG"),
    (dict(codes=0), "ARG"), (dict(params=dict(sr=0)), "ARG"), (dict(params=dict(s=FAKE + 8)), "ALIGN"),
])
def test_train_step_validation(libpath, case, expect):
    from paper_2506_03781_gb300 import api
    a = dict(W=FAKE, wd=api.W_BF16, out=8, n_in=512, q=3, g=128, codes=FAKE + 0x9000, gup=FAKE + 0xB000,
             map_mode=1, step=0, p_period=2, what=FAKE + 0xA000)
    a.update({k: v for k, v in case.items() if k != "params"})
    p = _params(api, **case.get("params", {}))
    st = api.lib().uq_train_step(a["W"], a["wd"], a["out"], a["n_in"], a["q"], a["g"], p, a["codes"], a["gup"],
                                 0.005, 0.0005, a["map_mode"], a["step"], a["p_period"], a["what"], None)
    assert st == getattr(api, "UQ_ERR_" + expect), (st, api.uq_last_error())
    assert api.uq_last_error() != ""


@cpu_only
@pytest.mark.parametrize("g,n_in", [(128, 512), (128, 32768), (64, 32768), (32, 16384), (32, 256)])
def test_train_step_accepts_the_fused_shapes(libpath, g, n_in):
    """Shapes at the limits of the fused kernel pass validation (on this
    GPU-less machine the launch itself then fails with UQ_ERR_CUDA)."""
    from paper_2506_03781_gb300 import api
    st = api.lib().uq_train_step(FAKE, api.W_BF16, 8, n_in, 3, g, _params(api), FAKE + 0x9000, FAKE + 0xB000,
                                 0.005, 0.0005, 1, 0, 2, FAKE + 0xA000, None)
    assert st == api.UQ_ERR_CUDA, api.uq_last_error()
    assert "uq_train_step" in api.uq_last_error()


@cpu_only
@pytest.mark.parametrize("case,expect", [
    (dict(q=0), "UNSUPPORTED"), (dict(g=48), "ARG"), (dict(n_in=200), "ARG"), (dict(out=0), "ARG"),
    (dict(batch=0), "ARG"), (dict(batch=65), "ARG"), (dict(xd=5), "ARG"),
    (dict(g=384, n_in=1536), "UNSUPPORTED"), (dict(g=640, n_in=1280), "UNSUPPORTED"),
    (dict(g=768, n_in=1536), "UNSUPPORTED"),
    (dict(planes=0), "ARG"), (dict(planes=FAKE + 4), "ALIGN"), (dict(a=0), "ARG"), (dict(z=FAKE + 8), "ALIGN"),
    (dict(x=0), "ARG"), (dict(y=0), "ARG"), (dict(y=FAKE + 12), "ALIGN"),
    (dict(work=0), "ARG"), (dict(work=FAKE + 4), "ALIGN"), (dict(wbytes=8 * 4 - 4), "ARG"),
])
def test_bcq_gemv_validation(libpath, case, expect):
    from paper_2506_03781_gb300 import api
    a = dict(planes=FAKE, a=FAKE + 0x1000, z=FAKE + 0x2000, out=8, n_in=512, q=3, g=128, x=FAKE + 0x3000,
             xd=api.W_BF16, batch=1, y=FAKE + 0x4000, work=FAKE + 0x5000, wbytes=1 << 20)
    a.update(case)
    st = api.lib().uq_bcq_gemv(a["planes"], a["a"], a["z"], a["out"], a["n_in"], a["q"], a["g"], a["x"], a["xd"],
                               a["batch"], a["y"], a["work"], a["wbytes"], None)
    assert st == getattr(api, "UQ_ERR_" + expect), (st, api.uq_last_error())
    assert api.uq_last_error() != ""


@cpu_only
@pytest.mark.parametrize("g,n_in", [(32, 512), (256, 512), (512, 1024), (1024, 3072), (2048, 2048)])
def test_bcq_gemv_accepts_groups_that_tile_the_column_tiles(libpath, g, n_in):
    """g dividing 512 or a multiple of 512 passes validation (only the launch
    fails on this GPU-less machine); both product entry points agree."""
    from paper_2506_03781_gb300 import api
    L = api.lib()
    st = L.uq_bcq_gemv(FAKE, FAKE + 0x1000, FAKE + 0x2000, 8, n_in, 3, g, FAKE + 0x3000, api.W_BF16, 1,
                       FAKE + 0x4000, FAKE + 0x5000, 1 << 20, None)
    assert st == api.UQ_ERR_CUDA, api.uq_last_error()
    st = L.uq_bcq_gemv_noalloc(FAKE, FAKE + 0x1000, FAKE + 0x2000, 8, n_in, 3, g, FAKE + 0x3000, api.W_BF16, 1,
                               FAKE + 0x4000, None)
    assert st == api.UQ_ERR_CUDA, api.uq_last_error()


@cpu_only
@pytest.mark.parametrize("g", [384, 640, 896, 1152])
def test_bcq_gemv_noalloc_rejects_groups_that_straddle_column_tiles(libpath, g):
    from paper_2506_03781_gb300 import api
    st = api.lib().uq_bcq_gemv_noalloc(FAKE, FAKE + 0x1000, FAKE + 0x2000, 8, 2 * g * 9, 3, g, FAKE + 0x3000,
                                       api.W_BF16, 1, FAKE + 0x4000, None)
    assert st == api.UQ_ERR_UNSUPPORTED and "divide 512" in api.uq_last_error()


def test_bcq_gemv_workspace_size(libpath):
    from paper_2506_03781_gb300 import api
    # one float per 512-column tile, token and row
    assert api.uq_bcq_gemv_workspace_bytes(8, 512, 1) == 8 * 4
    assert api.uq_bcq_gemv_workspace_bytes(8192, 28672, 1) == 56 * 8192 * 4
    assert api.uq_bcq_gemv_workspace_bytes(100, 4096 + 96, 3) == 9 * 3 * 100 * 4
    for bad in ((0, 512, 1), (8, 500, 1), (8, 512, 0), (8, 512, 65)):
        assert api.uq_bcq_gemv_workspace_bytes(*bad) == -1


@cpu_only
def test_omni_validation(libpath):
    from paper_2506_03781_gb300 import api
    L = api.lib()
    P = lambda **o: api.uq_params_omni(**{**{n: FAKE + 0x1000 * i for i, n in enumerate(api.OMNI_PARAM_NAMES)}, **o})
    Gd = lambda **o: api.uq_grads_omni(**{**{n: FAKE + 0x10000 + 0x1000 * i for i, n in enumerate(api.OMNI_GRAD_NAMES)},
                                         **o})
    fwd = lambda g=128, n_in=512, p=None, **k: L.uq_quantize_fwd_omni(
        k.get("W", FAKE), 1, 8, n_in, 3, g, p or P(), FAKE + 0x9000, k.get("map", 1), 0, 2, FAKE + 0xA000, None)
    assert fwd(g=1024, n_in=2048) == api.UQ_ERR_UNSUPPORTED
    assert fwd(g=384, n_in=768) == api.UQ_ERR_UNSUPPORTED
    assert fwd(W=0) == api.UQ_ERR_ARG
    assert fwd(p=P(beta=0)) == api.UQ_ERR_ARG
    assert fwd(p=P(gamma=FAKE + 4)) == api.UQ_ERR_ALIGN
    assert fwd(map=7) == api.UQ_ERR_ARG
    assert fwd() == api.UQ_ERR_CUDA                                   # valid: only the launch fails here
    bwd = lambda gr: L.uq_quantize_bwd_omni(FAKE, 1, 8, 512, 3, 128, P(), FAKE + 0x9000, FAKE + 0xB000, gr, None)
    for f in api.OMNI_GRAD_NAMES:
        assert bwd(Gd(**{f: 0})) == api.UQ_ERR_ARG and f in api.uq_last_error()
    assert L.uq_omni_scales(FAKE, 1, 8, 512, 3, 128, FAKE, FAKE, 0, FAKE, None) == api.UQ_ERR_ARG
    assert L.uq_omni_scales(FAKE, 1, 8, 768, 3, 96, FAKE, FAKE, FAKE, FAKE, None) == api.UQ_ERR_UNSUPPORTED


@cpu_only
def test_awq_validation(libpath):
    from paper_2506_03781_gb300 import api
    L = api.lib()
    P = lambda **o: api.uq_params_awq(**{**{n: FAKE + 0x1000 * i for i, n in enumerate(api.AWQ_PARAM_NAMES)}, **o})
    Gd = lambda **o: api.uq_grads_awq(**{**{n: FAKE + 0x10000 + 0x1000 * i for i, n in enumerate(api.AWQ_GRAD_NAMES)},
                                        **o})
    fwd = lambda g=128, n_in=512, p=None, W=FAKE, step=0: L.uq_quantize_fwd_awq(
        W, 1, 8, n_in, 3, g, p or P(), FAKE + 0x9000, 1, step, 2, FAKE + 0xA000, None)
    assert fwd(g=1024, n_in=2048) == api.UQ_ERR_UNSUPPORTED
    assert fwd(W=0) == api.UQ_ERR_ARG
    assert fwd(W=0, step=1) == api.UQ_ERR_CUDA                        # keep step: W is not read
    assert fwd(p=P(sa=0)) == api.UQ_ERR_ARG
    assert fwd(p=P(za=FAKE + 4)) == api.UQ_ERR_ALIGN
    bwd = lambda gr=None, ws=FAKE + 0x20000, nb=1 << 30: L.uq_quantize_bwd_awq(
        FAKE, 1, 8, 512, 3, 128, P(), FAKE + 0x9000, FAKE + 0xB000, gr or Gd(), ws, nb, None)
    for f in api.AWQ_GRAD_NAMES:
        assert bwd(Gd(**{f: 0})) == api.UQ_ERR_ARG and f in api.uq_last_error()
    assert bwd(ws=0) == api.UQ_ERR_ARG
    assert bwd(nb=0) == api.UQ_ERR_ARG and "workspace" in api.uq_last_error()
    assert api.uq_awq_bwd_workspace_bytes(8, 512, 3, 96) == -1
    assert api.uq_awq_bwd_workspace_bytes(8, 512, 3, 128) >= 8 * 4


@cpu_only
def test_bwd_ex_and_half_export_validation(libpath):
    from paper_2506_03781_gb300 import api
    L = api.lib()
    bwd = lambda flt, gr=None: L.uq_quantize_bwd_ex(FAKE, api.W_BF16, 8, 256, 3, 128, _params(api), FAKE + 0x9000,
                                                    FAKE + 0xB000, gr or _grads(api), flt, None)
    assert bwd(2) == api.UQ_ERR_ARG and "filter" in api.uq_last_error()
    assert bwd(api.FILTER_ELEMENT, _grads(api, ds=0)) == api.UQ_ERR_ARG
    assert bwd(api.FILTER_ELEMENT) == api.UQ_ERR_CUDA                 # valid: only the launch fails here
    ex = lambda mode=0, a=FAKE, W=FAKE, codes=FAKE: L.uq_export_bcq_half(W, 1, 8, 256, 3, 128, _params(api), codes,
                                                                         mode, FAKE, a, FAKE, None)
    assert ex(mode=5) == api.UQ_ERR_ARG
    assert ex(a=FAKE + 2) == api.UQ_ERR_ALIGN
    assert ex(mode=1, W=0) == api.UQ_ERR_ARG
    assert ex(codes=0) == api.UQ_ERR_ARG
    assert ex() == api.UQ_ERR_CUDA


def test_binding_rejects_host_tensors_before_calling(libpath):
    import torch
    from paper_2506_03781_gb300 import api
    W = torch.zeros(4, 128)
    with pytest.raises(ValueError):
        api.uq_quantize_fwd(W, 3, 128, {n: torch.zeros(1) for n in api.PARAM_NAMES}, torch.zeros(4, 128, dtype=torch.uint8),
                            torch.zeros(4, 128))


def test_oracle_and_product_are_independent():
    """The oracle imports nothing from the product package and vice versa;
    the only shared module is the seeded input generator."""
    prod = os.path.join(ROOT, "paper_2506_03781_gb300")
    for f in glob.glob(os.path.join(ROOT, "oracle", "*.py")):
        src = open(f).read()
        assert not re.search(r"^\s*(from|import)\s+paper_2506_03781_gb300", src, flags=re.M), f
    for f in glob.glob(os.path.join(prod, "**", "*"), recursive=True):
        if f.endswith((".py", ".cu", ".cuh", ".h")):
            src = open(f).read()
            assert not re.search(r"^\s*(from|import)\s+oracle", src, flags=re.M), f
    synth_src = open(os.path.join(prod, "synth.py")).read()
    for word in ("levels", "transform", "argmin", "bitplane"):
        assert word not in synth_src.lower(), word


def test_missing_library_raises_instead_of_falling_back(monkeypatch, tmp_path):
    """Without the built library every entry point raises: there is no other
    implementation behind the binding."""
    from paper_2506_03781_gb300 import api
    monkeypatch.setattr(api, "LIB", str(tmp_path / "libuq.so"))
    monkeypatch.setattr(api, "_lib", None)
    with pytest.raises(RuntimeError, match="no fallback"):
        api.lib()
    with pytest.raises(RuntimeError, match="no fallback"):
        api.uq_abi_version()
    with pytest.raises(RuntimeError, match="no fallback"):
        api.uq_bcq_gemv_workspace_bytes(8, 512)
