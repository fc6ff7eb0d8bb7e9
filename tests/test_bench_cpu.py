"""Host-side legs of the benchmark that need no GPU: the reference arm (the
CPU oracle timed on a bounded sample of the headline workload, one JSON line,
rank 0 only under torchrun) and the oracle timing of the other workloads."""

import os

import pytest
import torch.multiprocessing as mp

from tests.test_dist_cpu import _free_port


def test_reference_arm_line(capsys):
    """`bench.py --impl reference` times the CPU oracle on a bounded sample
    and prints one JSON line with the GPU arm's metric, unit and direction."""
    import json

    import bench
    bench.main(["--impl", "reference", "--steps", "2", "--warmup", "3"])
    lines = [ln for ln in capsys.readouterr().out.splitlines() if ln.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC
    assert d["unit"] == "weights/s" and d["higher_is_better"] is True
    assert d["steps"] == 2 and d["warmup"] == 3 and d["value"] > 0
    assert d["config"]["workload"] == "mlp14336x4096_bf16" and d["config"]["mapping"] == "local, p=2"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["value"] == d["value"]
    assert d["e2e"] == {"value": d["value"], "unit": "weights/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}


def _ref_worker(rank, world, port, results):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    import bench
    results[rank] = bench.main(["--impl", "reference", "--steps", "1", "--warmup", "3"]) is not None


@pytest.mark.timeout(180)
def test_reference_arm_rank0_only():
    """Under torchrun the reference arm runs on rank 0 alone; the others exit 0 without work."""
    world = 2
    port = _free_port()
    ctx = mp.get_context("spawn")
    results = ctx.Manager().dict()
    procs = [ctx.Process(target=_ref_worker, args=(r, world, port, results)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(150)
        assert p.exitcode == 0
    assert results[0] is True and results[1] is False



def test_oracle_timing_of_a_workload_covers_every_matrix():
    """The per-workload oracle baseline runs whole steps (fwd + bwd + export
    over a row sample of every matrix) until its budget has passed."""
    import bench
    from paper_2506_03781_gb300 import synth
    wl = synth.WORKLOADS["llama3_8b_block_bf16"]
    v, n, steps, el = bench.time_oracle_workload(wl, wl.q, 0.05, weights_per_matrix=8192)
    expect = sum(max(1, min(m.out, 8192 // m.n_in)) * m.n_in for m in wl.matrices)
    assert n == expect and steps >= 1 and el >= 0.05
    assert v == pytest.approx(n * steps / el)


def test_clock_record_from_nvidia_smi_lines():
    """The clock record of the bench line: median SM clock under load, the
    maximum, and every throttle reason seen Active in any sample (a run with
    hw_slowdown, hw_thermal_slowdown or sw_thermal_slowdown is rejected;
    sw_power_cap is kept and noted)."""
    import bench
    ok = "2026/12/02 10:00:00.100, 2070, 2070, 900.1, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active"
    cap = "2026/12/02 10:00:00.200, 1950, 2070, 1380.0, 0x0000000000000004, Not Active, Not Active, Not Active, Active"
    hot = "2026/12/02 10:00:00.300, 1500, 2070, 1390.0, 0x0000000000000040, Not Active, Active, Not Active, Not Active"
    r = bench.parse_clock_samples([ok, ok, cap, "garbage", "", "a, b, c, d, e, f, g, h, i"])
    assert r == {"sm_mhz": 2070.0, "sm_max_mhz": 2070.0, "reasons": ["sw_power_cap"], "samples": 3}
    r = bench.parse_clock_samples([ok, hot, cap])
    assert r["reasons"] == ["hw_thermal_slowdown", "sw_power_cap"] and r["sm_mhz"] == 1950.0
    assert bench.parse_clock_samples([]) == {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
    # the query the sampler issues has exactly the fields the parser reads
    assert bench.ClockSampler.FIELDS.count(",") == 7


def test_kernel_hash_ignores_comments_and_layout():
    """The backward's traffic record is keyed by a hash of its code with the
    comments and the layout removed: a comment or a re-indentation keeps the
    key, a change of code does not."""
    import bench
    src = "int a = 1; // one\n/* block\n comment */ int  b =\n 2;"
    assert bench.strip_comments(src) == "int a = 1; int b = 2;"
    assert bench.strip_comments("x /* y */ z // w") == "x z"
    assert bench.strip_comments("int a = 1;") != bench.strip_comments("int a = 2;")
    h = bench.kernel_hash()
    assert len(h) == 16 and h == bench.kernel_hash()
