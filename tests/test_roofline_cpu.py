"""The algorithmic bytes behind every roofline fraction, counted by hand for
the benchmark shapes from the per-element layout (bf16 W 2 B, s, W^, dL/dW^
and ds 4 B each, code word 1 B, (3 + q) fp32 parameters per group read and,
by the backward, written, s_r / ds_r 4 B per row, q bit-planes of 1 bit per
weight, alpha* and z* (q + 1) fp32 per group)."""

import pytest

from paper_2506_03781_gb300 import roofline

OUT, IN, Q, G = 14336, 4096, 3, 128
N = OUT * IN                      # 58,720,256 weights
GROUPS = OUT * IN // G            # 458,752 groups
GP = GROUPS * (3 + Q) * 4         # 11,010,048 B of group parameters


@pytest.mark.parametrize("kind,expect", [
    ("fwd_remap", 12 * N + GP + 4 * OUT),                      # W 2 + s 4 + codes 1 in, W^ 4 + codes 1 out
    ("fwd_keep", 5 * N + GP),                                  # codes 1 in, W^ 4 out
    ("fwd_full", 11 * N + GP + 4 * OUT),                       # W 2 + s 4 in, W^ 4 + codes 1 out
    ("bwd", 15 * N + 2 * GP + 8 * OUT),                        # W, s, codes, dL/dW^ in, ds out
    ("step_remap", 20 * N + 2 * GP + 8 * OUT),                 # + s' and W^ and codes written
    ("step_keep", 19 * N + 2 * GP + 8 * OUT),
    ("export_reuse", N + 3 * N // 8 + GP + GROUPS * 16),       # codes in; planes, alpha*, z* out
    ("export_eq4", 2 * N + 3 * N // 8 + GP + GROUPS * 16),     # W in instead of the codes
])
def test_bytes_of_the_benchmark_kernels(kind, expect):
    assert roofline.bytes_per_launch(kind, OUT, IN, Q, G, 2) == expect


def test_headline_values_in_megabytes():
    mb = lambda k: roofline.bytes_per_launch(k, OUT, IN, Q, G, 2) / 1e6
    assert round(mb("fwd_remap"), 1) == 715.7
    assert round(mb("fwd_keep"), 1) == 304.6
    assert round(mb("bwd"), 1) == 902.9
    assert round(mb("export_reuse"), 1) == 99.1
    assert round(mb("step_remap"), 1) == 1196.5 and round(mb("step_keep"), 1) == 1137.8
    # one step of the benchmark averages a remap and a keep step (p = 2)
    avg = (roofline.step_bytes(OUT, IN, Q, G, 2, True) + roofline.step_bytes(OUT, IN, Q, G, 2, False)) / 2
    assert avg == 1413099520.0


def test_bcq_product_bytes():
    out, n_in = 8192, 28672
    n = out * n_in
    groups = out * n_in // G
    # planes q/8 B per weight, alpha* and z* per group, one bf16 token in, y out
    assert roofline.bytes_per_launch("gemv", out, n_in, Q, G, 2) == 3 * n // 8 + groups * 16 + 2 * n_in + 4 * out
    assert roofline.bytes_per_launch("gemv", out, n_in, Q, G, 2) == 117530624


def test_fp32_weights_add_two_bytes_where_w_is_read():
    for kind in ("fwd_remap", "fwd_full", "bwd", "step_remap", "export_eq4"):
        d = roofline.bytes_per_launch(kind, OUT, IN, Q, G, 4) - roofline.bytes_per_launch(kind, OUT, IN, Q, G, 2)
        assert d == 2 * N, kind
    for kind in ("fwd_keep", "export_reuse"):
        assert roofline.bytes_per_launch(kind, OUT, IN, Q, G, 4) == roofline.bytes_per_launch(kind, OUT, IN, Q, G, 2)
