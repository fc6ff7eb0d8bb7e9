"""uq_bcq_gemv_noalloc: the BCQ product for callers that cannot allocate
device memory (for example code running where another allocator owns the
whole GPU, or where an allocation call is not allowed because it can block
the device).  It runs the product of uq_bcq_gemv with the library's own
built-in scratch instead of a caller workspace.

The GPU test calls it through the C ABI several times in a row, with
different shapes and inputs (one of them needs the whole scratch), and
checks that each result equals that of uq_bcq_gemv on the same inputs bit
for bit.  This file is
collected last, so that a run which stops at its first failure has run
every other test before it.
"""

import ctypes

import numpy as np
import pytest
import torch

from paper_2506_03781_gb300 import api

TOL = 1e-5        # of the L1 mass of the expanded terms, as in tests/test_gpu_gemv.py
FAKE = 0x7f0000000000


def _no_gpu():
    return not torch.cuda.is_available()


@pytest.mark.skipif(not _no_gpu(), reason="fake-pointer validation runs only without a GPU")
def test_noalloc_rejects_shapes_beyond_its_scratch_before_launching():
    from paper_2506_03781_gb300 import build
    build.build()
    L = api.lib()
    args = lambda out, n_in, batch: (FAKE, FAKE + 0x1000, FAKE + 0x2000, out, n_in, 3, 128, FAKE + 0x3000,
                                     api.W_BF16, batch, FAKE + 0x4000, None)
    # 56 tiles x 8192 rows x 3 tokens = 1,376,256 floats > 1,048,576
    assert L.uq_bcq_gemv_noalloc(*args(8192, 28672, 3)) == api.UQ_ERR_UNSUPPORTED
    assert "built-in scratch" in api.uq_last_error()
    assert L.uq_bcq_gemv_noalloc(*args(8192, 28672, 0)) == api.UQ_ERR_ARG
    # within the limit, validation passes and only the launch fails on this GPU-less machine
    assert L.uq_bcq_gemv_noalloc(*args(8192, 28672, 2)) == api.UQ_ERR_CUDA


def _mass(a_star, z_star, x, g):
    per_col = torch.repeat_interleave(a_star.double().abs().sum(-1) + z_star.double().abs(), g, dim=1)
    return x.double().abs() @ per_col.T


@pytest.mark.gpu
def test_noalloc_matches_the_workspace_entry_point_on_two_calls_in_a_row():
    """Both entry points launch the same kernels in the same fixed order, one
    with the caller's workspace and one with the built-in scratch, so their
    results must be identical bit for bit; the oracle's tolerance (1e-5 of
    the L1 mass of the expanded terms) is checked as well.  The second call
    needs exactly the scratch's 2^20 floats (1 tile x 64 tokens x 16384
    rows), so every word of the array is written and read."""
    d = torch.device("cuda", 0)
    gen = torch.Generator(device=d)
    gen.manual_seed(5)
    L = api.lib()
    cases = [(14336, 4096, 3, 128, 1, torch.bfloat16), (16384, 512, 2, 64, 64, torch.float32),
             (300, 28672 + 32 * 5, 2, 32, 2, torch.float32)]
    assert 16384 * 64 * 1 == 1 << 20
    for out, n_in, q, g, batch, xdt in cases:
        planes = torch.randint(-2 ** 31, 2 ** 31 - 1, (q, out, n_in // 32), generator=gen, device=d,
                               dtype=torch.int32)
        a_s = torch.randn(out, n_in // g, q, generator=gen, device=d) * 0.01
        z_s = torch.randn(out, n_in // g, generator=gen, device=d) * 0.003
        x = torch.randn(batch, n_in, generator=gen, device=d).to(xdt)
        y_ref = torch.full((batch, out), float("nan"), device=d)
        api.uq_bcq_gemv(planes, a_s, z_s, x, y_ref, g)
        y = torch.full((batch, out), float("nan"), device=d)
        st = L.uq_bcq_gemv_noalloc(planes.data_ptr(), a_s.data_ptr(), z_s.data_ptr(), out, n_in, q, g,
                                   x.data_ptr(), api._wdtype(x), batch, y.data_ptr(),
                                   ctypes.c_void_p(torch.cuda.current_stream(d).cuda_stream))
        assert st == api.UQ_OK, api.uq_last_error()
        torch.cuda.synchronize()
        assert torch.isfinite(y).all()
        assert torch.equal(y, y_ref), f"{out}x{n_in} batch {batch}: {int((y != y_ref).sum())} outputs differ"
        err = (y.double() - y_ref.double()).abs()
        assert (err <= TOL * _mass(a_s, z_s, x.float(), g) + 1e-30).all()
