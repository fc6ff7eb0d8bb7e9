"""Benchmark of the UniQuan_F quantizer step on GB300.

One step = the quantizer forward (Eq. 3, local and periodic mapping with
p = 2: remap on even steps, keep on odd steps) + its backward (App. C.1) over
the whole workload matrix, W resident in HBM.  Between steps the parameters
change as they would after an SGD update: a ring of parameter sets is
prepared before timing, each the previous one multiplied by 1 + eps N(0, 1)
(eps chosen so that ~0.03 % of the codes move per remap step, the paper's
per-step rate); the ring is generated outside the timed region.

Prints ONE JSON line (rank 0).  --impl reference times the CPU oracle on a
bounded sample of the same workload instead.  Under torchrun every rank runs
its own copy of the workload (rows are independent, no exchange step) and
the slowest rank's time is reported.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "quantizer fwd+bwd weights/sec and achieved HBM GB/s (% of GB300 peak) at q=3,g=128"
RING = 16                       # parameter sets prepared before timing
CLOCK_LEAD_S = 0.15             # untimed load before the timed steps while clocks are sampled
CLOCK_MIN_S = 0.5               # sampling runs at least this long (about 5 samples at 100 ms)
CLOCK_CHUNK = 16                # untimed steps between host checks of the elapsed time (even)


# ---------------------------------------------------------------------------
# distributed plumbing (host logic, tested with gloo on CPU)
# ---------------------------------------------------------------------------

def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def max_over_ranks(value: float, world: int, device=None) -> float:
    """Largest value over all ranks (the slowest rank's time)."""
    if world <= 1:
        return value
    import torch
    import torch.distributed as dist
    t = torch.tensor([value], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def weak_scaling_value(units_per_rank: int, steps: int, world: int, seconds: float) -> float:
    """Whole-job throughput: units all ranks processed / the slowest rank's time."""
    return units_per_rank * steps * world / seconds


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id: str | None):
        self.proc = None
        self.path = None
        self.gpu_id = gpu_id

    def start(self):
        self.t0 = time.time()
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            cmd = ["nvidia-smi", f"--query-gpu=timestamp,{self.FIELDS}", "--format=csv,noheader,nounits",
                   "-lms", "100"]
            if self.gpu_id:
                cmd += ["-i", self.gpu_id]
            self.proc = subprocess.Popen(cmd, stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            self.t0 = time.time()
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        time.sleep(max(0.0, CLOCK_MIN_S - (time.time() - self.t0)))
        self.proc.terminate()
        self.proc.wait()
        with open(self.path) as fh:
            lines = fh.readlines()
        os.unlink(self.path)
        return parse_clock_samples(lines)


def parse_clock_samples(lines):
    """Clock record from `nvidia-smi --query-gpu=timestamp,<ClockSampler.FIELDS>
    --format=csv,noheader,nounits` lines: median SM clock, the maximum SM
    clock, and every throttle reason (of hw_slowdown, hw_thermal_slowdown,
    sw_thermal_slowdown, sw_power_cap) seen Active in any sample.  Lines that
    do not parse are skipped."""
    sm, smax, reasons = [], [], set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for line in lines:
        parts = [p.strip() for p in line.split(",")]
        if len(parts) < 9:
            continue
        try:
            sm.append(float(parts[1]))
            smax.append(float(parts[2]))
        except ValueError:
            continue
        for n, v in zip(names, parts[5:9]):
            if v.lower() == "active":
                reasons.add(n)
    return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
            "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# helpers
# ---------------------------------------------------------------------------

def measured_peaks():
    try:
        return json.load(open(os.path.join(ROOT, "MEASURED_PEAKS.json")))
    except Exception:
        return None


def strip_comments(src):
    """C/C++ source without its comments and with runs of whitespace
    collapsed, so that edits to comments or layout keep the hash (string
    literals hold no comment markers in these files)."""
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    src = re.sub(r"//[^\n]*", " ", src)
    return " ".join(src.split())


def kernel_hash():
    """Hash of the code (comments and layout ignored) of the backward's source
    files: a recorded DRAM-traffic capture is used only for the code it was
    taken on."""
    h = hashlib.sha256()
    for f in ("uq_stream.cu", "uq_common.cuh", "uq_pipe.cuh"):
        h.update(strip_comments(open(os.path.join(ROOT, "paper_2506_03781_gb300", "csrc", f)).read()).encode())
    return h.hexdigest()[:16]


def recorded_traffic(workload, q):
    """DRAM bytes per backward launch from the committed ncu summary, if it was
    taken on the current kernel source (else None)."""
    path = os.path.join(ROOT, "profiles", "bwd_traffic.json")
    try:
        rec = json.load(open(path))
    except Exception:
        return None
    key = f"{workload}/q{q}"
    ent = rec.get(key)
    if not ent or ent.get("kernel_hash") != kernel_hash():
        return None
    return ent.get("dram_bytes_per_launch")


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count()


# ---------------------------------------------------------------------------
# CPU oracle timing (the cpu_baseline / --impl reference legs)
# ---------------------------------------------------------------------------

def oracle_sample_inputs(wl, q, rows, row0=0):
    """Oracle-initialised inputs of rows row0 .. row0 + rows of the workload."""
    import oracle as O
    from paper_2506_03781_gb300 import synth
    _, W = synth.workload_weights(wl, 0, slice(row0, row0 + rows))
    g = wl.g
    init = O.unified_init(W, q, g, G=2, T=2)
    P = {k: init[k] for k in ("delta", "zu", "s", "sr", "alpha", "zb")}
    P = synth.jitter(P, synth.perturb_factors(synth.param_shapes(rows, W.shape[1], g, q), wl.init_eps, 0))
    Gup = synth.upstream_grad(rows, W.shape[1], wl.grad_var, 0)
    return W, P, init["codes"], Gup


def parity_sample(wl, q, rows, Wd, P_dev, codes_dev, Gup_dev, dev, stream):
    """Parity counters of the timed kernels (part of the CPU-baseline leg).

    The oracle's inputs for the first `rows` rows (its own unified
    initialization, the seeded jitter and dL/dW^ of oracle_sample_inputs)
    replace those rows of copies of the benchmark's device buffers; the GPU
    then runs the timed calls over the WHOLE matrix in the timed launch
    configuration -- the forward of a remap step (t = 0) and its backward,
    the forward of a keep step (t = 1), and one fused step (t = 1, whose
    forward of t + 1 remaps) -- and the sampled rows are compared with the
    oracle: codes and W^ bit for bit (mismatches counted), gradients and
    updated parameters as the worst ratio of error to tolerance (1e-4 of the
    fp64 L1 mass; for the fused step lr times that plus two fp32 ulps)."""
    import torch
    import oracle as O
    from paper_2506_03781_gb300 import api
    g = wl.g
    W, P, codes0, Gup = oracle_sample_inputs(wl, q, rows)
    Pd = {k: v.clone() for k, v in P_dev.items()}
    for k in Pd:
        Pd[k][:rows].copy_(torch.from_numpy(np.ascontiguousarray(P[k])))
    cd = codes_dev.clone()
    cd[:rows].copy_(torch.from_numpy(codes0))
    Gd = Gup_dev.clone()
    Gd[:rows].copy_(torch.from_numpy(Gup))
    what = torch.empty_like(Gd)
    out, n_in = Gd.shape
    gr = api.empty_grads(out, n_in, q, g, dev)
    args = lambda Q: (W, Q["s"], Q["sr"], Q["delta"], Q["zu"], Q["alpha"], Q["zb"])
    host = lambda t: t[:rows].cpu().numpy()

    def grad_ratio(ref, mass):
        worst = 0.0
        for k in ("ddelta", "dzu", "dzb", "dalpha", "dsr"):
            err = np.abs(host(gr[k]).astype(np.float64) - ref[k])
            worst = max(worst, float((err / (1e-4 * mass[k] + 1e-30)).max()))
        ds = ref["ds"]
        err = np.abs(host(gr["ds"]).astype(np.float64) - ds)
        worst = max(worst, float((err / (1e-4 * np.maximum(np.abs(ds), 1e-6 * np.abs(ds).max()))).max()))
        return worst

    res = {"rows": rows, "weights": rows * n_in,
           "inputs": "the oracle's own init of the first rows (G=2, T=2), seeded jitter and dL/dW^; the GPU runs "
                     "the whole matrix in the timed launch configuration"}
    api.uq_quantize_fwd(Wd, q, g, Pd, cd, what, api.MAP_LOCAL_PERIODIC, 0, wl.p, stream=stream)
    api.uq_quantize_bwd(Wd, q, g, Pd, cd, Gd, gr, stream=stream)
    torch.cuda.synchronize()
    r_what, r_codes = O.quantize_fwd(*args(P), codes0, g, O.MAP_LOCAL_PERIODIC, 0, wl.p)
    ref = O.quantize_bwd(*args(P), r_codes, Gup, g)
    mass = O.bwd_l1_mass(*args(P), r_codes, Gup, g)
    res["fwd_remap"] = {"codes_mismatch": int((host(cd) != r_codes).sum()),
                        "what_mismatch": int((host(what) != r_what).sum()),
                        "codes_moved": int((r_codes != codes0).sum())}
    res["bwd"] = {"grad_worst_frac_of_tol": grad_ratio(ref, mass)}
    api.uq_quantize_fwd(Wd, q, g, Pd, cd, what, api.MAP_LOCAL_PERIODIC, 1, wl.p, stream=stream)
    torch.cuda.synchronize()
    k_what, _ = O.quantize_fwd(*args(P), r_codes, g, O.MAP_LOCAL_PERIODIC, 1, wl.p)
    res["fwd_keep"] = {"codes_mismatch": int((host(cd) != r_codes).sum()),
                       "what_mismatch": int((host(what) != k_what).sum())}
    api.uq_train_step(Wd, q, g, Pd, cd, Gd, what, 1, stream=stream)
    torch.cuda.synchronize()
    new, c2, w2 = O.train_step(*args(P), r_codes, Gup, g, 1)
    worst = 0.0
    gname = {"delta": "ddelta", "zu": "dzu", "s": "ds", "sr": "dsr", "alpha": "dalpha", "zb": "dzb"}
    for k in ("delta", "zu", "s", "sr", "alpha", "zb"):
        lr = O.LR_F if k in ("delta", "zu", "s", "sr") else O.LR_B
        gm = mass[gname[k]] if k != "s" else np.maximum(np.abs(ref["ds"]), 1e-6 * np.abs(ref["ds"]).max())
        tol = (lr * 1e-4 * gm + 2 * np.spacing(np.abs(new[k]).astype(np.float32))
               + np.spacing(np.abs(lr * ref[gname[k]]).astype(np.float32)))
        err = np.abs(host(Pd[k]).astype(np.float64) - new[k])
        worst = max(worst, float((err / tol).max()))
    res["train_step"] = {"codes_mismatch": int((host(cd) != c2).sum()), "param_worst_frac_of_tol": worst}
    del Pd, cd, Gd, what, gr
    torch.cuda.empty_cache()
    return res


def time_oracle_step(wl, q, rows, budget_s, row0=0, barrier=None):
    """Runs oracle steps (fwd at step t + bwd) until budget_s elapses; returns
    (weights per second, steps run, seconds).  With a barrier, the timed loop
    starts once every party has prepared its inputs."""
    import oracle as O
    W, P, codes, Gup = oracle_sample_inputs(wl, q, rows, row0)
    g = wl.g
    if barrier is not None:
        barrier.wait()
    t0 = time.perf_counter()
    n = 0
    while True:
        _, codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, g,
                                  O.MAP_LOCAL_PERIODIC, n, wl.p)
        O.quantize_bwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, Gup, g)
        n += 1
        el = time.perf_counter() - t0
        if el >= budget_s and n >= 2:
            break
    return W.size * n / el, n, el


def _oracle_shard(wl_name, q, row0, rows, budget_s, barrier, results):
    """One process of the row-parallel oracle timing (spawned; no CUDA)."""
    from paper_2506_03781_gb300 import synth
    wl = synth.WORKLOADS[wl_name]
    _, n, el = time_oracle_step(wl, q, rows, budget_s, row0, barrier)
    results.put((rows * wl.matrices[0].n_in * n, el))


def time_oracle_parallel(wl, q, rows, budget_s, workers):
    """The same oracle steps on `workers` row shards at once, one process
    each (rows are independent): every process prepares its shard, waits at
    a barrier, then runs budget_s seconds.  Returns (aggregate weights per
    second, the longest process's seconds).  Spawned processes, one numpy
    thread each."""
    import multiprocessing as mp
    ctx = mp.get_context("spawn")
    barrier, results = ctx.Barrier(workers), ctx.Queue()
    saved = {k: os.environ.get(k) for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS")}
    os.environ.update({k: "1" for k in saved})
    import queue
    procs, out = [], []
    try:
        procs = [ctx.Process(target=_oracle_shard, args=(wl.name, q, k * rows, rows, budget_s, barrier, results))
                 for k in range(workers)]
        for pr in procs:
            pr.start()
        deadline = time.perf_counter() + 10 * budget_s + 300
        while len(out) < workers and time.perf_counter() < deadline:
            try:
                out.append(results.get(timeout=5))
            except queue.Empty:
                if any(pr.exitcode not in (None, 0) for pr in procs):
                    break                               # a worker failed: no all-core figure
    finally:
        for k, v in saved.items():
            if v is None:
                os.environ.pop(k, None)
            else:
                os.environ[k] = v
        for pr in procs:
            pr.join(timeout=5)
            if pr.is_alive():
                pr.kill()                               # this call's own child process
                pr.join()
    if len(out) < workers:
        return None, None
    el = max(o[1] for o in out)
    return sum(o[0] for o in out) / el, el


# ---------------------------------------------------------------------------
# GPU run
# ---------------------------------------------------------------------------

def time_slabs(wl, q, steps, warmup, dev, seed=0, graph=True):
    """time_matrices with the matrices of one input width stored as row ranges
    of one slab (api.RowSlabs): per step one forward, one backward and one
    export per width instead of per matrix (the Llama-3-8B block: 2 widths,
    7 matrices)."""
    import torch
    from paper_2506_03781_gb300 import api, synth
    g = wl.g
    gen = torch.Generator(device=dev)
    gen.manual_seed(1000 * wl.seed + q + 7 * seed)
    slabs = api.RowSlabs({m.name: (m.out, m.n_in) for m in wl.matrices}, q, g,
                         torch.bfloat16 if wl.wdtype == "bf16" else torch.float32, dev, with_export=True)
    for idx, m in enumerate(wl.matrices):
        raw, _ = synth.workload_weights(wl, idx)
        slabs.view(m.name)["W"].copy_(api.weights_tensor(raw, dev))
    slabs.init_params(G=wl.G, T=wl.T)
    for d in slabs.slabs.values():
        for k in ("delta", "s", "sr", "alpha"):
            d["params"][k].mul_(1.0 + wl.init_eps * torch.randn(d["params"][k].shape, generator=gen, device=dev))
        d["dL_dWhat"].copy_(torch.randn(d["dL_dWhat"].shape, generator=gen, device=dev) * float(np.sqrt(wl.grad_var)))

    def step(t):
        slabs.fwd(t, wl.p)
        slabs.bwd()
        slabs.export()

    for t in range(warmup):
        step(t)
    torch.cuda.synchronize()
    graphs = None
    if graph:
        side = torch.cuda.Stream(dev)
        graphs = []
        for t in (0, 1):
            cg = torch.cuda.CUDAGraph()
            with torch.cuda.graph(cg, stream=side):
                step(t)
            graphs.append(cg)
        torch.cuda.synchronize()
    stream = torch.cuda.current_stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for t in range(steps):
        if graphs is not None:
            graphs[(warmup + t) % wl.p != 0].replay()
        else:
            step(warmup + t)
    e1.record(stream)
    torch.cuda.synchronize()
    n = sum(m.out * m.n_in for m in wl.matrices)
    del slabs, graphs
    torch.cuda.empty_cache()
    return e0.elapsed_time(e1) / steps, n, 3 * len({m.n_in for m in wl.matrices})


def time_matrices(wl, q, steps, warmup, dev, with_export=False, seed=0, graph=False):
    """Times `steps` optimisation steps over every matrix of a workload, all
    launches back to back on one stream: per matrix the forward (local
    mapping, p from the workload: remap and keep steps alternate) and the
    backward, plus the bit-plane export when `with_export`.  Parameters come
    from the GPU unified initialization, jittered once.  With `graph` the
    launches of a remap step and of a keep step are captured once as two CUDA
    graphs and replayed.  Returns (ms per step, total weights)."""
    import torch
    from paper_2506_03781_gb300 import api, synth
    g = wl.g
    gen = torch.Generator(device=dev)
    gen.manual_seed(1000 * wl.seed + q + 7 * seed)
    mats = []
    for idx, m in enumerate(wl.matrices):
        raw, _ = synth.workload_weights(wl, idx)
        Wd = api.weights_tensor(raw, dev)
        p = api.empty_params(m.out, m.n_in, q, g, dev)
        codes = torch.empty(m.out, m.n_in, dtype=torch.uint8, device=dev)
        api.uq_init_params(Wd, q, g, p, codes, G=wl.G, T=wl.T)
        for k in ("delta", "s", "sr", "alpha"):
            p[k].mul_(1.0 + wl.init_eps * torch.randn(p[k].shape, generator=gen, device=dev))
        G = torch.randn(m.out, m.n_in, generator=gen, device=dev) * float(np.sqrt(wl.grad_var))
        qz = api.Quantizer(Wd, q, g, p, codes, torch.empty(m.out, m.n_in, device=dev), G,
                           api.empty_grads(m.out, m.n_in, q, g, dev))
        ex = None
        if with_export:
            ex = (torch.empty(q, m.out, m.n_in // 32, dtype=torch.int32, device=dev),
                  torch.empty(m.out, m.n_in // g, q, device=dev), torch.empty(m.out, m.n_in // g, device=dev))
        mats.append((qz, ex))

    def step(t):
        for qz, ex in mats:
            qz.fwd(t, wl.p)
            qz.bwd()
            if ex is not None:
                qz.export(*ex)

    for t in range(warmup):
        step(t)
    torch.cuda.synchronize()
    graphs = None
    if graph:
        side = torch.cuda.Stream(dev)
        graphs = []
        for t in (0, 1):                        # a remap step, a keep step
            cg = torch.cuda.CUDAGraph()
            with torch.cuda.graph(cg, stream=side):
                step(t)
            graphs.append(cg)
        torch.cuda.synchronize()
    stream = torch.cuda.current_stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for t in range(steps):
        if graphs is not None:
            graphs[(warmup + t) % wl.p != 0].replay()
        else:
            step(warmup + t)
    e1.record(stream)
    torch.cuda.synchronize()
    n = sum(m.out * m.n_in for m in wl.matrices)
    del mats, graphs
    torch.cuda.empty_cache()
    return e0.elapsed_time(e1) / steps, n


def _train_step_run(Wd, q, g, P0, codes0, Gup, p, steps, stream, dev):
    """CUDA-event times of `steps` fused steps (after 3 warm-up calls) on
    copies of the parameters and codes, updated in place from call to call,
    and the share of the codes the next remapping step moves."""
    import torch
    from paper_2506_03781_gb300 import api
    P = {k: v.clone() for k, v in P0.items()}
    codes = codes0.clone()
    what = torch.empty(codes.shape, dtype=torch.float32, device=dev)
    qz = api.Quantizer(Wd, q, g, P, codes, what, Gup, api.empty_grads(codes.shape[0], codes.shape[1], q, g, dev))
    for t in range(3):
        qz.train_step(t, p_period=p, stream=stream)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(steps)]
    for t in range(steps):
        ev[t][0].record(stream)
        qz.train_step(3 + t, p_period=p, stream=stream)
        ev[t][1].record(stream)
    torch.cuda.synchronize()
    api.uq_check_device(stream)
    # share of the codes the next remapping step moves (untimed)
    t_next = 3 + steps
    if (t_next + 1) % p != 0:
        qz.train_step(t_next, p_period=p, stream=stream)
        t_next += 1
    before = codes.clone()
    qz.train_step(t_next, p_period=p, stream=stream)
    torch.cuda.synchronize()
    moved = float((codes != before).float().mean())
    ms = [a.elapsed_time(b) for a, b in ev]
    remap = [m for t, m in enumerate(ms) if (3 + t + 1) % p == 0]
    keep = [m for t, m in enumerate(ms) if (3 + t + 1) % p != 0]
    return {"avg_ms": statistics.mean(ms), "steps": steps,
            "remap": statistics.mean(remap) if remap else float("nan"),
            "keep": statistics.mean(keep) if keep else float("nan"),
            "codes_moved_per_remap_step": moved}


def time_train_step(Wd, q, g, P0, codes0, Gup, p, steps, stream, dev, rate=3e-4):
    """The fused step (uq_train_step) timed in two regimes of dL/dW^.

    SGD applies the same dL/dW^ at every step here.  The workload's draw,
    N(0, 1e-4), then moves Delta by a large fraction per step and a few per
    cent of the codes on every remapping step, far more than training does
    (Table 2: about 0.03 % per step).  The main timing therefore scales the
    draw so that a remapping step moves about `rate` of the codes (the
    scale is picked from powers of ten by two untimed steps each); the
    unscaled draw is timed too ("unscaled")."""
    import math
    import torch
    from paper_2506_03781_gb300 import api
    best, best_k = None, 1.0
    for k in (1.0, 0.1, 0.01, 1e-3, 1e-4, 1e-5):
        P = {n: v.clone() for n, v in P0.items()}
        codes = codes0.clone()
        what = torch.empty(codes.shape, dtype=torch.float32, device=dev)
        qz = api.Quantizer(Wd, q, g, P, codes, what, Gup * k, None)
        t = 0 if (0 + 1) % p == 0 else 1
        if t:
            qz.train_step(0, p_period=p, stream=stream)
        before = codes.clone()
        qz.train_step(t, p_period=p, stream=stream)
        torch.cuda.synchronize()
        moved = float((codes != before).float().mean())
        err = abs(math.log10(max(moved, 1e-9) / rate))
        if best is None or err < best:
            best, best_k = err, k
        del qz, P, codes, what
    res = _train_step_run(Wd, q, g, P0, codes0, Gup * best_k, p, steps, stream, dev)
    res["dL_dWhat"] = (f"the workload's N(0, 1e-4) draw times {best_k:g}, the power of ten whose remapping step moves "
                       f"closest to {rate:g} of the codes; the same draw every step")
    unscaled = _train_step_run(Wd, q, g, P0, codes0, Gup, p, steps, stream, dev)
    unscaled["dL_dWhat"] = "the workload's N(0, 1e-4) draw, the same every step"
    res["unscaled"] = unscaled
    return res


def time_gemv(q, g, dev, stream, peak, shapes=((14336, 4096), (8192, 28672)), reps=60):
    """CUDA-event time of the BCQ product from the exported format
    (uq_bcq_gemv, one bf16 token: the split kernel and the tile sum) per
    call, on random bit-planes, alpha*, z* of each shape; the calls cycle
    through enough copies of the inputs to exceed twice the L2, so every call
    reads them from HBM.  `reps` calls are replayed from one CUDA graph."""
    import math
    import torch
    from paper_2506_03781_gb300 import api, roofline
    res = {}
    gen = torch.Generator(device=dev)
    gen.manual_seed(77)
    for out, n_in in shapes:
        nbytes = roofline.bytes_per_launch("gemv", out, n_in, q, g, 2)
        copies = max(2, math.ceil(2 * 129e6 / nbytes))
        ring = []
        for _ in range(copies):
            planes = torch.randint(-2 ** 31, 2 ** 31 - 1, (q, out, n_in // 32), generator=gen, device=dev,
                                   dtype=torch.int32)
            a_s = torch.randn(out, n_in // g, q, generator=gen, device=dev) * 0.01
            z_s = torch.randn(out, n_in // g, generator=gen, device=dev) * 0.003
            x = torch.randn(1, n_in, generator=gen, device=dev).to(torch.bfloat16)
            ring.append((planes, a_s, z_s, x, torch.empty(1, out, device=dev)))
        ws = api.bcq_gemv_workspace(out, n_in, 1, dev)
        for i in range(3):
            api.uq_bcq_gemv(*ring[i % copies], g, workspace=ws, stream=stream)
        torch.cuda.synchronize()
        # the calls are captured once in a CUDA graph so that the replay measures
        # device time, not the per-call argument checking of the Python binding
        side = torch.cuda.Stream(dev)
        side.wait_stream(torch.cuda.current_stream(dev))
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=side):
            for i in range(reps):
                api.uq_bcq_gemv(*ring[i % copies], g, workspace=ws, stream=side)
        graph.replay()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        graph.replay()
        e1.record(stream)
        torch.cuda.synchronize()
        us = e0.elapsed_time(e1) * 1e3 / reps
        del graph
        res[f"{out}x{n_in}"] = {"us": us, "gbs": nbytes / us / 1e3, "frac": nbytes / us / 1e3 / peak,
                                "weights_per_s": out * n_in / (us * 1e-6), "algorithmic_bytes": nbytes,
                                "input_copies": copies}
        del ring
    torch.cuda.empty_cache()
    return res


def time_link(hp, hin, hout, reps=3):
    """The copy ceiling of the end-to-end number, measured in this process:
    the same pinned host buffers copied to the device alone, back alone, and
    both directions at once (CUDA events on the copy streams), in GB/s, and
    the weights/s those copies alone would allow."""
    import torch
    from paper_2506_03781_gb300 import api
    hs = hp.steps[0]
    dev = {**hs.dev, **hs.params}
    up_b, down_b = hp.bytes_in(hin), hp.bytes_out(hout)

    def h2d():
        with torch.cuda.stream(hp.up):
            for name in api.HostStep.IN_KEYS:
                dev[name].copy_(hin[name], non_blocking=True)

    def d2h():
        with torch.cuda.stream(hp.down):
            hout["W_hat"].copy_(hs.dev["W_hat"], non_blocking=True)
            hout["codes"].copy_(hs.dev["codes"], non_blocking=True)
            for name in api.GRAD_NAMES:
                hout[name].copy_(hs.grads[name], non_blocking=True)

    def timed(fns):
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(torch.cuda.current_stream())
        for st in (hp.up, hp.down):
            st.wait_event(e0)
        for _ in range(reps):
            for f in fns:
                f()
        for st in (hp.up, hp.down):
            torch.cuda.current_stream().wait_stream(st)
        e1.record(torch.cuda.current_stream())
        torch.cuda.synchronize()
        return e0.elapsed_time(e1) / 1e3 / reps

    t_up, t_down, t_both = timed([h2d]), timed([d2h]), timed([h2d, d2h])
    return {"h2d_gbs": up_b / t_up / 1e9, "d2h_gbs": down_b / t_down / 1e9,
            "duplex_ms_per_step": t_both * 1e3,
            "copy_ceiling_weights_per_s": hs.out * hs.n_in / t_both}


def time_block_step(dev, steps=20, warmup=4, samples=4, idx_steps=64):
    """Algorithm 1 on a Llama-3-8B-shaped block (seq 2048, bf16 block
    compute, the block workload's q and g): ms per optimisation step (block
    forward + backward in torch, then uq_train_step for the seven weights),
    the quantizer's share of it, the share of codes a remap step moves, and,
    over `idx_steps` further untimed steps, the index-change statistics of
    the paper's Table 2 (shares of weights whose level index moves by 0, 1,
    2, >2 in one step and over the whole run) and the loss of every step."""
    import time
    import torch
    from paper_2506_03781_gb300 import api, synth
    from paper_2506_03781_gb300.recon import NAMES, BlockReconstructor, index_change_shares
    wl = synth.WORKLOADS["llama3_8b_block_bf16"]
    shape = synth.BLOCKS["llama3_8b"]
    Wb = synth.block_weights(shape, wl.seed)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    rec = BlockReconstructor(shape, {n: Wb[n][0] for n in NAMES}, wl.q, wl.g, device=dev, G=wl.G, T=wl.T)
    torch.cuda.synchronize()
    init_s = time.perf_counter() - t0
    X, Xh = synth.block_inputs(shape, samples, wl.seed, perturb=0.01)
    Xd = [torch.from_numpy(x).to(dev) for x in X]
    Xhd = [torch.from_numpy(x).to(dev) for x in Xh]
    Y = rec.targets(Xd)
    losses = []
    for i in range(warmup):
        losses.append(rec.step(Y[i % samples], Xhd[i % samples]))
    torch.cuda.synchronize()
    stream = torch.cuda.current_stream(dev)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for i in range(steps):
        losses.append(rec.step(Y[i % samples], Xhd[i % samples]))
    e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / steps
    # the quantizer alone: the seven fused steps of one optimisation step
    q0, q1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    q0.record(stream)
    qgrads = {n: (torch.randn(rec.what_c[n].shape, device=dev) * 1e-7).to(torch.bfloat16) for n in NAMES} \
        if rec.bf16_io else None
    for i in range(steps):
        rec.quantizer_step(qgrads)
    q1.record(stream)
    torch.cuda.synchronize()
    qms = q0.elapsed_time(q1) / steps
    # codes moved by remap steps (the forward of t + 1 remaps when (t + 1) % p == 0)
    moved = []
    for i in range(4):
        before = {n: rec.codes[n].clone() for n in NAMES}
        remap = (rec.t + 1) % rec.p == 0
        rec.step(Y[i % samples], Xhd[i % samples])
        if remap:
            ch = sum(int((rec.codes[n] != before[n]).sum()) for n in NAMES)
            moved.append(ch / sum(rec.codes[n].numel() for n in NAMES))
    # Table 2 (index changes) and the reconstruction-error curve (Fig. 5b): idx_steps
    # further steps from here, the level index of every weight after each one
    r0 = torch.cat([r.view(-1) for r in rec.ranks().values()])
    prev, per_step, curve = r0, [], []
    for i in range(idx_steps):
        curve.append(rec.step(Y[i % samples], Xhd[i % samples]))
        r = torch.cat([r.view(-1) for r in rec.ranks().values()])
        per_step.append(index_change_shares(r, prev))
        prev = r
    index_change = {
        "bins": ["0", "1", "2", ">2"],
        "single_step_mean": [statistics.mean(s[k] for s in per_step) for k in range(4)],
        "single_step_max_moved": max(1.0 - s[0] for s in per_step),
        "all_steps": index_change_shares(prev, r0),
        "steps": idx_steps,
        "learning_rates": [rec.lr_F, rec.lr_B],
        "paper_llama3_8b": {"single_step": [0.9997, 0.0001, 0.0, 0.0001],
                            "all_steps_2560": [0.8930, 0.0837, 0.0136, 0.0097]},
    }
    api.uq_check_device(stream)
    n_w = sum(rec.codes[n].numel() for n in NAMES)
    res = {"block": shape.name, "seq": shape.seq, "q": wl.q, "g": wl.g, "weights": n_w, "steps": steps,
           "ms_per_step": ms, "quantizer_ms_per_step": qms, "quantizer_share": qms / ms,
           "codes_moved_per_remap_step": statistics.mean(moved) if moved else None,
           # mean loss of each epoch (one pass over the samples, from the first step on)
           "loss_per_epoch": [float(torch.stack(losses[k:k + samples]).mean())
                              for k in range(0, len(losses) - samples + 1, samples)],
           "init_s": init_s,
           "index_change": index_change,
           # loss of every step of the index-change run (the reconstruction-error curve)
           "loss_curve": [float(v) for v in torch.stack(curve)] if curve else [],
           "paper_step_s_a100_derived": 0.25}
    del rec, Y, Xd, Xhd
    torch.cuda.empty_cache()
    return res


def time_variants(dev, stream, peak, q=3, g=128, out=14336, n_in=4096, reps=20):
    """CUDA-event times of the OmniQuant- and AWQ-unified quantizer kernels
    (forward remap and keep steps, backward) on a matrix of the headline
    shape with random parameters and inputs (every call moves far more than
    the L2 holds)."""
    import torch
    from paper_2506_03781_gb300 import api, roofline
    gen = torch.Generator(device=dev)
    gen.manual_seed(99)
    Wd = (torch.randn(out, n_in, generator=gen, device=dev) * 0.02).to(torch.bfloat16)
    Gr = n_in // g
    codes = torch.randint(0, 1 << q, (out, n_in), generator=gen, device=dev, dtype=torch.uint8)
    what = torch.empty(out, n_in, device=dev)
    Gup = torch.randn(out, n_in, generator=gen, device=dev) * 0.01
    lv = torch.tensor([2.0 ** (q - 2 - j) for j in range(q)], device=dev)
    alpha = (lv * (1 + 0.05 * torch.randn(out, Gr, q, generator=gen, device=dev))).contiguous()
    zb = ((1 << q) - 1) / 2 + 0.1 * torch.randn(out, Gr, generator=gen, device=dev)
    omni = {"beta": 0.9 + 0.1 * torch.rand(out, Gr, generator=gen, device=dev),
            "gamma": 0.9 + 0.1 * torch.rand(out, Gr, generator=gen, device=dev), "alpha": alpha, "zb": zb}
    og = {"dbeta": torch.empty(out, Gr, device=dev), "dgamma": torch.empty(out, Gr, device=dev),
          "dalpha": torch.empty(out, Gr, q, device=dev), "dzb": torch.empty(out, Gr, device=dev)}
    awq = {"sa": 0.5 + torch.rand(n_in, generator=gen, device=dev), "delta": torch.full((out, Gr), 0.01, device=dev),
           "za": torch.full((out, Gr), 3.5, device=dev), "alpha": alpha, "zb": zb}
    ag = {"dsa": torch.empty(n_in, device=dev), "ddelta": torch.empty(out, Gr, device=dev),
          "dza": torch.empty(out, Gr, device=dev), "dalpha": torch.empty(out, Gr, q, device=dev),
          "dzb": torch.empty(out, Gr, device=dev)}
    ws = torch.empty(max(api.uq_awq_bwd_workspace_bytes(out, n_in, q, g) // 4, 4), device=dev)
    calls = {
        "omni_fwd_remap": lambda: api.uq_quantize_fwd_omni(Wd, q, g, omni, codes, what, api.MAP_LOCAL_PERIODIC, 0, 2,
                                                            stream=stream),
        "omni_fwd_keep": lambda: api.uq_quantize_fwd_omni(Wd, q, g, omni, codes, what, api.MAP_LOCAL_PERIODIC, 1, 2,
                                                           stream=stream),
        "omni_bwd": lambda: api.uq_quantize_bwd_omni(Wd, q, g, omni, codes, Gup, og, stream=stream),
        "awq_fwd_remap": lambda: api.uq_quantize_fwd_awq(Wd, q, g, awq, codes, what, api.MAP_LOCAL_PERIODIC, 0, 2,
                                                          stream=stream),
        "awq_fwd_keep": lambda: api.uq_quantize_fwd_awq(Wd, q, g, awq, codes, what, api.MAP_LOCAL_PERIODIC, 1, 2,
                                                         stream=stream),
        "awq_bwd": lambda: api.uq_quantize_bwd_awq(Wd, q, g, awq, codes, Gup, ag, workspace=ws, stream=stream),
    }
    res = {}
    for name, fn in calls.items():
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        nbytes = roofline.bytes_per_launch(name, out, n_in, q, g, 2)
        res[name] = {"avg_ms": ms, "gbs": nbytes / ms / 1e6, "frac": nbytes / ms / 1e6 / peak}
    del Wd, codes, what, Gup, ws
    torch.cuda.empty_cache()
    return res


def run_gpu(args):
    import torch
    from paper_2506_03781_gb300 import api, roofline, synth

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    wl = synth.WORKLOADS[args.workload]
    m = wl.matrices[0]
    q, g = args.q, wl.g
    out, n_in = m.out, m.n_in
    N = out * n_in

    raw, _ = synth.workload_weights(wl, 0)
    Wd = api.weights_tensor(raw, dev)
    wbytes = Wd.element_size()
    p0 = api.empty_params(out, n_in, q, g, dev)
    codes = torch.empty(out, n_in, dtype=torch.uint8, device=dev)
    api.uq_init_params(Wd, q, g, p0, codes, G=wl.G, T=wl.T)

    # parameter ring: set_0 = init * (1 + init_eps N), set_t = set_{t-1} * (1 + step_eps N)
    gen = torch.Generator(device=dev)
    gen.manual_seed(1000 * wl.seed + q)
    jit = ("delta", "s", "sr", "alpha")

    def jitter(p, eps):
        outp = dict(p)
        for k in jit:
            outp[k] = p[k] * (1.0 + eps * torch.randn(p[k].shape, generator=gen, device=dev))
        return outp

    ring = [jitter(p0, wl.init_eps)]
    for _ in range(1, min(RING, args.warmup + args.steps)):
        ring.append(jitter(ring[-1], wl.step_eps))
    Gup = torch.randn(out, n_in, generator=gen, device=dev) * float(np.sqrt(wl.grad_var))
    what = torch.empty(out, n_in, dtype=torch.float32, device=dev)
    grads = api.empty_grads(out, n_in, q, g, dev)
    stream = torch.cuda.current_stream(dev)

    def step(t, ev=None):
        P = ring[t % len(ring)]
        if ev is not None:
            ev[0].record(stream)
        api.uq_quantize_fwd(Wd, q, g, P, codes, what, api.MAP_LOCAL_PERIODIC, t, wl.p, stream=stream)
        if ev is not None:
            ev[1].record(stream)
        api.uq_quantize_bwd(Wd, q, g, P, codes, Gup, grads, stream=stream)
        if ev is not None:
            ev[2].record(stream)

    for t in range(args.warmup):
        step(t)
    torch.cuda.synchronize()

    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    gpu_id = None
    try:
        gpu_id = str(torch.cuda.get_device_properties(dev).uuid)
        gpu_id = gpu_id if gpu_id.startswith("GPU-") else "GPU-" + gpu_id
    except Exception:
        gpu_id = None
    def load_for(seconds, t0):
        # the same step loop, untimed, in chunks of an even number of steps
        # (so the remap/keep alternation of the timed steps is unchanged)
        n, t_start = 0, time.perf_counter()
        while time.perf_counter() - t_start < seconds:
            for i in range(CLOCK_CHUNK):
                step(t0 + n + i)
            torch.cuda.synchronize()
            n += CLOCK_CHUNK
        return n

    # Clocks are sampled every 100 ms while the GPU runs the step loop: the
    # sampler starts before an untimed lead-in, and an untimed tail after the
    # closing barrier keeps the load on until it has run CLOCK_MIN_S, so that
    # every sample is taken under the load of the timed steps.
    clk = ClockSampler(gpu_id)
    clk.start()
    lead = load_for(CLOCK_LEAD_S, args.warmup)
    t_first = args.warmup + lead
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for t in range(args.steps):
        step(t_first + t, evs[t])
    end.record(stream)
    torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    load_for(CLOCK_MIN_S - (time.time() - clk.t0), t_first + args.steps)
    clocks = clk.stop()
    clocks["sampled_over"] = "an untimed lead-in of the same step loop, the timed steps and an untimed tail"
    ms = start.elapsed_time(end)
    ms_max = max_over_ranks(ms, world, dev)
    secs = ms_max / 1e3
    value = weak_scaling_value(N, args.steps, world, secs)

    fwd_ms = [e[0].elapsed_time(e[1]) for e in evs]
    bwd_ms = [e[1].elapsed_time(e[2]) for e in evs]
    bwd_bytes = roofline.bytes_per_launch("bwd", out, n_in, q, g, wbytes)
    steps_idx = [t_first + t for t in range(args.steps)]
    step_bytes = sum(roofline.step_bytes(out, n_in, q, g, wbytes, t % wl.p == 0) for t in steps_idx)
    peaks = measured_peaks()
    peak = peaks["hbm_gbs"] if peaks else 6800.0
    bwd_avg_s = statistics.mean(bwd_ms) / 1e3
    achieved = bwd_bytes / bwd_avg_s / 1e9
    fwd_remap = [f for f, t in zip(fwd_ms, steps_idx) if t % wl.p == 0]
    fwd_keep = [f for f, t in zip(fwd_ms, steps_idx) if t % wl.p != 0]

    # export timed separately (one launch after the steps)
    planes = torch.empty(q, out, n_in // 32, dtype=torch.int32, device=dev)
    a_s = torch.empty(out, n_in // g, q, dtype=torch.float32, device=dev)
    z_s = torch.empty(out, n_in // g, dtype=torch.float32, device=dev)
    P_last = ring[(args.warmup + args.steps - 1) % len(ring)]
    ex = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    for _ in range(3):
        api.uq_export_bcq(Wd, q, g, P_last, codes, planes, a_s, z_s, api.EXPORT_REUSE_CODES, stream=stream)
    ex[0].record(stream)
    for _ in range(10):
        api.uq_export_bcq(Wd, q, g, P_last, codes, planes, a_s, z_s, api.EXPORT_REUSE_CODES, stream=stream)
    ex[1].record(stream)
    torch.cuda.synchronize()
    exp_ms = ex[0].elapsed_time(ex[1]) / 10
    exp_bytes = roofline.bytes_per_launch("export_reuse", out, n_in, q, g, wbytes)

    # fused optimisation step (backward of t + SGD update + forward of t + 1)
    # on its own copy of the parameters, updated in place step after step
    train = time_train_step(Wd, q, g, ring[0], codes, Gup, wl.p, min(args.steps, 100), stream, dev)
    train_bytes = {k: roofline.bytes_per_launch(k, out, n_in, q, g, wbytes) for k in ("step_remap", "step_keep")}
    for tr in (train, train["unscaled"]):
        for k in ("remap", "keep"):
            ms_k = tr[k]
            tr[k] = {"avg_ms": ms_k, "gbs": train_bytes["step_" + k] / 1e6 / ms_k,
                     "frac": train_bytes["step_" + k] / 1e6 / ms_k / peak}
    train["weights_per_s"] = N / (train["avg_ms"] / 1e3)
    train["algorithmic_bytes_avg"] = (train_bytes["step_remap"] + train_bytes["step_keep"]) / 2

    # deployment: the BCQ product from the exported format (one bf16 token)
    gemv = time_gemv(q, g, dev, stream, peak)

    # UniQuan with OmniQuant's and AWQ's maps (App. E) on the same shape
    variants = time_variants(dev, stream, peak, q, g, out, n_in)

    # Algorithm 1 on a Llama-3-8B-shaped block (the quantizer inside the loop)
    block = None if args.no_block else time_block_step(dev)

    # end-to-end through the public host-buffer API: every step uploads its
    # inputs from pinned host memory, runs fwd+bwd and downloads its results;
    # consecutive steps (independent, like successive weight matrices)
    # overlap their uploads, compute and downloads.
    hp = api.HostPipeline(out, n_in, q, g, Wd.dtype, dev, depth=2)
    hin, hout = hp.empty_host(pinned=True)
    hin["W"].copy_(Wd.cpu())
    for k in api.PARAM_NAMES:
        hin[k].copy_(ring[0][k].cpu())
    hin["codes"].copy_(codes.cpu())
    hin["dL_dWhat"].copy_(Gup.cpu())
    e2e_steps = max(3, min(args.steps, 20))
    for t in range(3):
        hp.submit(hin, hout, t, wl.p)
    torch.cuda.synchronize()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(hp.up)
    for t in range(e2e_steps):
        hp.submit(hin, hout, t, wl.p)
    e1.record(hp.down)
    torch.cuda.synchronize()
    e2e_ms = e0.elapsed_time(e1)
    e2e_ms = max_over_ranks(e2e_ms, world, dev)
    e2e_value = weak_scaling_value(N, e2e_steps, world, e2e_ms / 1e3)
    link = time_link(hp, hin, hout)

    # bit-width sweep of the same matrix (the workload is specified for q in {2, 3, 4})
    sweep = {}
    if not args.no_sweep:
        for qq in wl.qs:
            if qq == q:
                sweep[f"q{qq}"] = {"weights_per_s": value / world, "ms_per_step": ms_max / args.steps}
                continue
            ms_q, n_q = time_matrices(wl, qq, min(args.steps, 50), 3, dev)
            sweep[f"q{qq}"] = {"weights_per_s": n_q / (ms_q / 1e3), "ms_per_step": ms_q}

    result = None
    if rank == 0:
        cpu = cpu_all = parity = None
        if world == 1 and not args.no_cpu_baseline:
            rows = 96
            v, n, el = time_oracle_step(wl, q, rows, args.cpu_budget)
            cpu = {"value": v, "unit": "weights/s", "cores": 1, "kind": "oracle",
                   "sample": f"first {rows} rows of {out}x{n_in} ({rows * n_in} weights), {n} oracle steps "
                             f"(local remap/keep alternating + backward) in {el:.1f} s, numpy single thread"}
            parity = parity_sample(wl, q, rows, Wd, ring[0], codes, Gup, dev, stream)
            workers = max(1, min(cpu_cores(), out // rows))
            vp, elp = time_oracle_parallel(wl, q, rows, args.cpu_budget, workers)
            if vp is not None:
                cpu_all = {"value": vp, "unit": "weights/s", "cores": workers, "kind": "oracle",
                           "sample": f"{workers} processes, each on its own {rows}-row shard of {out}x{n_in}, the "
                                     f"same oracle steps for {elp:.1f} s (row-parallel, one numpy thread each)"}
        result = {
            "metric": METRIC,
            "value": value,
            "unit": "weights/s",
            "n_gpus": world,
            "steps": args.steps,
            "warmup": args.warmup,
            "ms_per_step": ms_max / args.steps,
            "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": None,
            "dtype": "f32 (bf16 W)",
            "data": "synthetic (seeded Student-t(4) weights with outlier columns; no model weights)",
            "config": {"workload": wl.name, "shape": [out, n_in], "q": q, "g": g, "mapping": "local, p=2",
                       "weights_per_step": N, "ring_of_parameter_sets": len(ring),
                       "l2": "inputs larger than L2 (about 1.5 GB moved per step vs 129 MB L2)",
                       "step_bytes_avg": step_bytes / args.steps,
                       "hbm_gbs_step": step_bytes / secs / 1e9 * world},
            "roofline": {"bound": "hbm", "kernel": "bwd_stream_kernel", "achieved": achieved, "peak": peak,
                         "unit": "GB/s", "frac": achieved / peak,
                         "traffic": recorded_traffic(wl.name, q),
                         "algorithmic_bytes": bwd_bytes, "avg_ms": bwd_avg_s * 1e3,
                         "peak_source": "MEASURED_PEAKS.json hbm_gbs" if peaks else "fallback"},
            "kernels": {
                "fwd_remap": {"avg_ms": statistics.mean(fwd_remap) if fwd_remap else None,
                              "gbs": (roofline.bytes_per_launch("fwd_remap", out, n_in, q, g, wbytes) / 1e6
                                      / statistics.mean(fwd_remap)) if fwd_remap else None},
                "fwd_keep": {"avg_ms": statistics.mean(fwd_keep) if fwd_keep else None,
                             "gbs": (roofline.bytes_per_launch("fwd_keep", out, n_in, q, g, wbytes) / 1e6
                                     / statistics.mean(fwd_keep)) if fwd_keep else None},
                "bwd": {"avg_ms": bwd_avg_s * 1e3, "gbs": achieved},
                "export_reuse": {"ms": exp_ms, "gbs": exp_bytes / 1e6 / exp_ms},
            },
            "e2e": {"value": e2e_value, "unit": "weights/s",
                    "h2d_bytes_per_step": hp.bytes_in(hin), "d2h_bytes_per_step": hp.bytes_out(hout),
                    "steps": e2e_steps, "ms_per_step": e2e_ms / e2e_steps, "link": link,
                    "api": "paper_2506_03781_gb300.api.HostPipeline (pinned host buffers, uploads/compute/"
                           "downloads of consecutive steps overlapped)"},
            "train_step": train,
            "bcq_gemv": gemv,
            "block_step": block,
            "unified_variants": variants,
            "q_sweep": sweep,
            "gpu_launches": 2 * args.steps,
            "clocks": clocks,
            "cpu_baseline": cpu,
            "cpu_baseline_all_cores": cpu_all,
            "parity": parity,
        }
        print(json.dumps(result))
    if world > 1:
        torch.distributed.destroy_process_group()
    return result


def time_oracle_workload(wl, q, budget_s, weights_per_matrix=131072):
    """The CPU oracle as it stands (numpy, one thread) on a bounded sample of
    every matrix of a workload: the first rows of each matrix (about
    `weights_per_matrix` weights), oracle-initialised and jittered like the
    GPU inputs.  One step = per matrix the forward (local mapping at step t),
    the backward and the bit-plane export (Theorem 1, reused codes).  Runs
    whole steps until budget_s has passed.  Returns (weights per second,
    weights per step, steps, seconds)."""
    import oracle as O
    from paper_2506_03781_gb300 import synth
    g = wl.g
    mats = []
    for idx, m in enumerate(wl.matrices):
        rows = max(1, min(m.out, weights_per_matrix // m.n_in))
        _, W = synth.workload_weights(wl, idx, slice(0, rows))
        init = O.unified_init(W, q, g, G=2, T=2)
        P = {k: init[k] for k in ("delta", "zu", "s", "sr", "alpha", "zb")}
        P = synth.jitter(P, synth.perturb_factors(synth.param_shapes(rows, m.n_in, g, q), wl.init_eps, idx))
        mats.append([W, P, init["codes"], synth.upstream_grad(rows, m.n_in, wl.grad_var, idx)])
    n = sum(mm[0].size for mm in mats)
    t0 = time.perf_counter()
    steps = 0
    while True:
        for mm in mats:
            W, P, codes, Gup = mm
            _, codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, g,
                                      O.MAP_LOCAL_PERIODIC, steps, wl.p)
            O.quantize_bwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, Gup, g)
            O.export_bcq(W, P["delta"], P["zu"], P["alpha"], P["zb"], codes, g)
            mm[2] = codes
        steps += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            return n * steps / el, n, steps, el


def run_workloads(args):
    """Times the other workloads: the Llama-3-8B block (seven matrices, q = 2,
    g = 64, fwd + bwd + export as one launch sequence on one stream) and the
    Llama-2-70B MLP matrices (q = 3, g = 128, fwd + bwd + export).  One JSON
    line per workload."""
    import torch
    from paper_2506_03781_gb300 import synth
    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    lines = []
    names = ("llama3_8b_block_bf16", "llama2_70b_mlp_bf16", "attn4k_bf16", "mat1k_f32")
    for name in names:
        wl = synth.WORKLOADS[name]
        cpu = None
        if not args.no_cpu_baseline:
            v, n_s, k, el = time_oracle_workload(wl, wl.q, args.cpu_budget / len(names))
            cpu = {"value": v, "unit": "weights/s", "cores": 1, "kind": "oracle",
                   "sample": f"the first rows of each of the {len(wl.matrices)} matrices ({n_s} weights), {k} "
                             f"oracle steps of fwd + bwd + bit-plane export in {el:.1f} s, numpy single thread"}
        for graph in (False, True):
            ms, n = time_matrices(wl, wl.q, args.steps, args.warmup, dev, with_export=True, graph=graph)
            line = {"workload": name, "q": wl.q, "g": wl.g, "weights": n, "steps": args.steps,
                    "cuda_graph": graph, "ms_per_step": ms, "weights_per_s": n / (ms / 1e3),
                    "step": "per matrix: fwd (local mapping, remap/keep alternating) + bwd + bit-plane export",
                    "cpu_baseline": cpu}
            print(json.dumps(line))
            lines.append(line)
        if len({m.n_in for m in wl.matrices}) < len(wl.matrices):
            ms, n, launches = time_slabs(wl, wl.q, args.steps, args.warmup, dev)
            line = {"workload": name, "q": wl.q, "g": wl.g, "weights": n, "steps": args.steps,
                    "cuda_graph": True, "ms_per_step": ms, "weights_per_s": n / (ms / 1e3),
                    "step": f"grouped: the matrices of each input width as one row slab, fwd + bwd + bit-plane "
                            f"export per width ({launches} calls per step)",
                    "cpu_baseline": cpu}
            print(json.dumps(line))
            lines.append(line)
    return lines


def run_reference(args):
    """The CPU oracle as it stands, on a bounded sample of the same workload:
    every step is one oracle forward (local mapping at step t, so remap and
    keep steps alternate as on the GPU) and one backward over the first 64
    rows of the matrix.  Inputs are prepared once, before the warm-up."""
    rank, world, _ = dist_env()
    if rank != 0:
        return None
    import oracle as O
    from paper_2506_03781_gb300 import synth
    wl = synth.WORKLOADS[args.workload]
    m = wl.matrices[0]
    rows = 64
    W, P, codes, Gup = oracle_sample_inputs(wl, args.q, rows)
    g = wl.g

    def step(t, codes):
        _, codes = O.quantize_fwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, g,
                                  O.MAP_LOCAL_PERIODIC, t, wl.p)
        O.quantize_bwd(W, P["s"], P["sr"], P["delta"], P["zu"], P["alpha"], P["zb"], codes, Gup, g)
        return codes

    for t in range(args.warmup):
        codes = step(t, codes)
    t0 = time.perf_counter()
    for t in range(args.warmup, args.warmup + args.steps):
        codes = step(t, codes)
    el = time.perf_counter() - t0
    value = W.size * args.steps / el
    sample = (f"first {rows} rows of {m.out}x{m.n_in} per step ({W.size} weights), one oracle fwd "
              f"(local mapping, p={wl.p}) + bwd, numpy single thread")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "weights/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": el / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32/f64 (oracle)",
            "data": "synthetic", "config": {"workload": wl.name, "shape": [m.out, m.n_in], "q": args.q, "g": g,
                                            "mapping": f"local, p={wl.p}"},
            "cpu_baseline": {"value": value, "unit": "weights/s", "cores": 1, "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": "weights/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line))
    return line


KERNELS = ("bwd", "fwd_remap", "fwd_keep", "export", "step", "omni_bwd", "awq_bwd", "gemv")


def run_kernel(args):
    """Profiling driver: one kernel of the path on one problem, for ncu.

    Allocates a single problem of the headline shape (14336 x 4096 bf16,
    about 1.5 GB on the device; 8192 x 28672 planes for the BCQ product),
    launches the named call `--launches` times after one warm-up launch on
    one stream and prints one JSON line with the CUDA-event time per launch.
    The launch list of a capture is therefore short and known: launch 0 is
    the warm-up, launches 1.. are the measured ones (for `step` every call
    alternates a remapping and a keeping forward of t + 1).
    """
    import torch
    from paper_2506_03781_gb300 import api, roofline, synth

    dev = torch.device("cuda", 0)
    torch.cuda.set_device(dev)
    stream = torch.cuda.current_stream(dev)
    wl = synth.WORKLOADS["mlp14336x4096_bf16"]
    m = wl.matrices[0]
    q, g = args.q, wl.g
    out, n_in = m.out, m.n_in
    gen = torch.Generator(device=dev)
    gen.manual_seed(1000 * wl.seed + q)
    name = args.kernel
    if name == "gemv":
        out, n_in = 8192, 28672
        planes = torch.randint(-2 ** 31, 2 ** 31 - 1, (q, out, n_in // 32), generator=gen, device=dev,
                               dtype=torch.int32)
        a_s = torch.randn(out, n_in // g, q, generator=gen, device=dev) * 0.01
        z_s = torch.randn(out, n_in // g, generator=gen, device=dev) * 0.003
        x = torch.randn(1, n_in, generator=gen, device=dev).to(torch.bfloat16)
        y = torch.empty(1, out, device=dev)
        ws = api.bcq_gemv_workspace(out, n_in, 1, dev)
        call = lambda i: api.uq_bcq_gemv(planes, a_s, z_s, x, y, g, workspace=ws, stream=stream)
        nbytes = roofline.bytes_per_launch("gemv", out, n_in, q, g, 2)
    elif name in ("omni_bwd", "awq_bwd"):
        Wd = (torch.randn(out, n_in, generator=gen, device=dev) * 0.02).to(torch.bfloat16)
        Gr = n_in // g
        codes = torch.randint(0, 1 << q, (out, n_in), generator=gen, device=dev, dtype=torch.uint8)
        Gup = torch.randn(out, n_in, generator=gen, device=dev) * 0.01
        lv = torch.tensor([2.0 ** (q - 2 - j) for j in range(q)], device=dev)
        alpha = (lv * (1 + 0.05 * torch.randn(out, Gr, q, generator=gen, device=dev))).contiguous()
        zb = ((1 << q) - 1) / 2 + 0.1 * torch.randn(out, Gr, generator=gen, device=dev)
        if name == "omni_bwd":
            P = {"beta": 0.9 + 0.1 * torch.rand(out, Gr, generator=gen, device=dev),
                 "gamma": 0.9 + 0.1 * torch.rand(out, Gr, generator=gen, device=dev), "alpha": alpha, "zb": zb}
            gr = {"dbeta": torch.empty(out, Gr, device=dev), "dgamma": torch.empty(out, Gr, device=dev),
                  "dalpha": torch.empty(out, Gr, q, device=dev), "dzb": torch.empty(out, Gr, device=dev)}
            call = lambda i: api.uq_quantize_bwd_omni(Wd, q, g, P, codes, Gup, gr, stream=stream)
        else:
            P = {"sa": 0.5 + torch.rand(n_in, generator=gen, device=dev),
                 "delta": torch.full((out, Gr), 0.01, device=dev), "za": torch.full((out, Gr), 3.5, device=dev),
                 "alpha": alpha, "zb": zb}
            gr = {"dsa": torch.empty(n_in, device=dev), "ddelta": torch.empty(out, Gr, device=dev),
                  "dza": torch.empty(out, Gr, device=dev), "dalpha": torch.empty(out, Gr, q, device=dev),
                  "dzb": torch.empty(out, Gr, device=dev)}
            ws = torch.empty(max(api.uq_awq_bwd_workspace_bytes(out, n_in, q, g) // 4, 4), device=dev)
            call = lambda i: api.uq_quantize_bwd_awq(Wd, q, g, P, codes, Gup, gr, workspace=ws, stream=stream)
        nbytes = roofline.bytes_per_launch(name, out, n_in, q, g, 2)
    else:
        raw, _ = synth.workload_weights(wl, 0)
        Wd = api.weights_tensor(raw, dev)
        P = api.empty_params(out, n_in, q, g, dev)
        codes = torch.empty(out, n_in, dtype=torch.uint8, device=dev)
        api.uq_init_params(Wd, q, g, P, codes, G=wl.G, T=wl.T)
        for k in ("delta", "s", "sr", "alpha"):
            P[k].mul_(1.0 + wl.init_eps * torch.randn(P[k].shape, generator=gen, device=dev))
        Gup = torch.randn(out, n_in, generator=gen, device=dev) * float(np.sqrt(wl.grad_var) * args.grad_scale)
        what = torch.empty(out, n_in, dtype=torch.float32, device=dev)
        qz = api.Quantizer(Wd, q, g, P, codes, what, Gup, api.empty_grads(out, n_in, q, g, dev))
        if name == "bwd":
            call = lambda i: qz.bwd(stream=stream)
        elif name == "fwd_remap":
            call = lambda i: qz.fwd(0, wl.p, stream=stream)
        elif name == "fwd_keep":
            call = lambda i: qz.fwd(1, wl.p, stream=stream)
        elif name == "step":
            call = lambda i: qz.train_step(i, p_period=wl.p, stream=stream)
        else:
            ex = (torch.empty(q, out, n_in // 32, dtype=torch.int32, device=dev),
                  torch.empty(out, n_in // g, q, device=dev), torch.empty(out, n_in // g, device=dev))
            call = lambda i: qz.export(*ex, stream=stream)
        kind = {"export": "export_reuse", "step": "step_keep"}.get(name, name)
        nbytes = roofline.bytes_per_launch(kind, out, n_in, q, g, 2)
    torch.cuda.synchronize()
    call(0)
    torch.cuda.synchronize()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)) for _ in range(args.launches)]
    for i in range(args.launches):
        ev[i][0].record(stream)
        call(1 + i)
        ev[i][1].record(stream)
    torch.cuda.synchronize()
    api.uq_check_device(stream)
    us = [a.elapsed_time(b) * 1e3 for a, b in ev]
    res = {"kernel": name, "shape": [out, n_in], "q": q, "g": g, "launches": args.launches, "us": us,
           "algorithmic_bytes": nbytes, "kernel_hash": kernel_hash()}
    print(json.dumps(res))
    return res


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="gb300", choices=["gb300", "reference"])
    ap.add_argument("--workload", default="mlp14336x4096_bf16")
    ap.add_argument("--q", type=int, default=3)
    ap.add_argument("--cpu-budget", type=float, default=12.0, help="seconds of oracle CPU work")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-sweep", action="store_true", help="skip the q sweep of the headline matrix")
    ap.add_argument("--no-block", action="store_true", help="skip the block reconstruction loop timing")
    ap.add_argument("--workloads", action="store_true", help="time the other workloads instead")
    ap.add_argument("--kernel", choices=KERNELS, help="profiling driver: one kernel on one problem (for ncu)")
    ap.add_argument("--launches", type=int, default=2, help="measured launches of --kernel after one warm-up")
    ap.add_argument("--grad-scale", type=float, default=1.0, help="--kernel: factor on the N(0, 1e-4) dL/dW^ draw")
    args = ap.parse_args(argv)
    args.warmup = max(3, args.warmup)          # at least 3 untimed warm-up steps
    if args.impl == "reference":
        return run_reference(args)
    if args.kernel:
        return run_kernel(args)
    if args.workloads:
        return run_workloads(args)
    return run_gpu(args)


if __name__ == "__main__":
    main()
