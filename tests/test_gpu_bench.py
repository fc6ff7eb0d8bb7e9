"""The benchmark's contract on the GPU: one short `bench.py` run prints one
JSON line whose keys, units and counts are the ones the line promises (the
metric and workload, the roofline object of the dominant kernel, the
end-to-end figure with its host<->device bytes, the launch count and the
clock record)."""

import json

import pytest

pytestmark = pytest.mark.gpu


def test_bench_prints_one_complete_line(capsys):
    import bench
    steps, warmup = 6, 3
    ret = bench.main(["--steps", str(steps), "--warmup", str(warmup), "--no-block", "--no-sweep",
                      "--no-cpu-baseline"])
    lines = [ln for ln in capsys.readouterr().out.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d == json.loads(json.dumps(ret))
    assert d["metric"] == bench.METRIC and d["unit"] == "weights/s" and d["higher_is_better"] is True
    assert d["n_gpus"] == 1 and d["steps"] == steps and d["warmup"] == warmup and d["scaling"] == "weak"
    assert d["config"]["workload"] == "mlp14336x4096_bf16" and d["config"]["shape"] == [14336, 4096]
    assert d["config"]["q"] == 3 and d["config"]["g"] == 128
    n = 14336 * 4096
    assert d["value"] == pytest.approx(n * steps / (d["ms_per_step"] * steps / 1e3), rel=1e-9)
    r = d["roofline"]
    assert r["bound"] == "hbm" and r["unit"] == "GB/s" and r["kernel"] == "bwd_stream_kernel"
    assert 0.2 < r["frac"] < 1.5 and r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    assert r["achieved"] == pytest.approx(r["algorithmic_bytes"] / (r["avg_ms"] / 1e3) / 1e9)
    assert "traffic" in r
    e = d["e2e"]
    assert e["value"] > 0 and e["unit"] == "weights/s"
    assert e["h2d_bytes_per_step"] > 10 * n and e["d2h_bytes_per_step"] > 9 * n
    assert d["gpu_launches"] == 2 * steps
    c = d["clocks"]
    assert c["samples"] >= 1 and c["sm_mhz"] and c["sm_max_mhz"]
    assert d["cpu_baseline"] is None
    for k in ("fwd_remap", "fwd_keep", "bwd"):
        assert d["kernels"][k]["avg_ms"] > 0
    assert set(d["bcq_gemv"]) == {"14336x4096", "8192x28672"}
    assert d["train_step"]["avg_ms"] > 0
