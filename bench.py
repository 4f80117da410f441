"""Benchmark of the batched timeline composer on GB300.

Workload: the GPT-175B Megatron-shaped step (96 ranks, TP8 PP6 DP2, 16 micro-batches
1F1B, ~1.1M ops) composed for 1024 what-if scenarios per GPU.  One step = the whole
hot path over that batch: CC estimation for every collective x scenario, the first
composition, the overlap test and the second (slowdown-adjusted) composition.

metric: node x scenario timeline updates per second (each compose pass updates
every op in every scenario, so one step is 2 * V * S updates), plus the achieved
HBM bandwidth of the compose kernel against the measured GB300 copy peak.

Usage: python bench.py [--gpus N] [--steps K] [--warmup W] [--impl echo|reference]
Under torchrun each rank composes its own slice of 1024 scenarios of one batch of
1024 * N (weak scaling, no collective on the data path); the step time is the
max over ranks.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "node×scenario timeline updates/sec and achieved HBM GB/s vs GB300 peak"
UNIT = "updates/s"
WORKLOAD = "gpt175b"
# DRAM bytes per node-scenario of the composition kernels from the committed ncu
# capture (a data file beside its summary), valid for the kernel source it names
PROFILE_DATA = os.path.join(ROOT, "profiles", "traffic_per_node_scenario.json")


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), \
        int(os.environ.get("LOCAL_RANK", "0"))


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index=None):
        self.index = index
        self.proc = None
        self.path = os.path.join(tempfile.gettempdir(), f"echo_bench_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            os.makedirs(os.path.dirname(self.path), exist_ok=True)
            cmd = ["nvidia-smi", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits", "-lms", "100"]
            if self.index is not None:
                cmd[1:1] = ["-i", str(self.index)]
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(cmd, stdout=self.f, stderr=subprocess.DEVNULL)
        except Exception as ex:  # pragma: no cover
            log("clock sampling unavailable:", ex)
            self.proc = None

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:  # pragma: no cover
            self.proc.kill()
        self.f.close()
        sm, mx, reasons, power = [], [], set(), []
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            p = [x.strip() for x in line.split(",")]
            if len(p) < 9:
                continue
            try:
                sm.append(float(p[1]))
                mx.append(float(p[2]))
                power.append(float(p[3]))
            except ValueError:
                continue
            for nm, val in zip(names, p[5:9]):
                if val.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm), "power_w_max": max(power) if power else None}


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def source_hash(name):
    """sha256[:16] of a kernel source file of the library, comments and whitespace
    left out (so that a change to the comments alone keeps a capture current)."""
    import re
    with open(os.path.join(ROOT, "paper_2412_12487_gb300", "csrc", name), encoding="utf-8") as f:
        src = f.read()
    src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
    src = re.sub(r"//[^\n]*", " ", src)
    src = " ".join(src.split())
    return hashlib.sha256(src.encode()).hexdigest()[:16]


def profiled_traffic(workload, kernel, launch_units):
    """DRAM bytes per launch of `kernel` on `workload` from the committed ncu data
    (per node-scenario, scaled to ``launch_units`` node-scenarios), if it was taken
    on the kernel's current source."""
    try:
        with open(PROFILE_DATA) as f:
            d = json.load(f)["workloads"][workload]["kernels"][kernel]
        if d["source_sha256_16"] != source_hash(d["source"]):
            return None
        return float(d["dram_bytes_per_node_scenario"]) * launch_units
    except (OSError, ValueError, KeyError, TypeError):
        return None


_HOST_BUFFERS = []


def pinned_host_array(shape, dtype=np.int64):
    """A page-locked host array for the duration matrix.  It is mapped with
    transparent huge pages requested (fewer address translations for the copy
    engine, whose throughput otherwise drops on fragmented host memory) and then
    registered with CUDA; torch's pinned allocator is the fallback."""
    import mmap
    import torch
    nbytes = int(np.prod(shape)) * np.dtype(dtype).itemsize
    try:
        buf = mmap.mmap(-1, nbytes, flags=mmap.MAP_PRIVATE | mmap.MAP_ANONYMOUS)
        if hasattr(mmap, "MADV_HUGEPAGE"):
            buf.madvise(mmap.MADV_HUGEPAGE)
        arr = np.frombuffer(buf, dtype=dtype).reshape(shape)
        rc = torch.cuda.cudart().cudaHostRegister(arr.ctypes.data, nbytes, 0)
        if getattr(rc, "value", rc) != 0:
            raise RuntimeError(f"cudaHostRegister: {rc}")
        _HOST_BUFFERS.append((buf, arr))
        return torch.from_numpy(arr)
    except Exception as ex:  # pragma: no cover - depends on the host
        log("huge-page host buffer unavailable, using torch's pinned allocator:", ex)
        return torch.from_numpy(np.empty(0, dtype)).new_empty(shape).pin_memory()


def build_inputs(rank, world, n_scen=None, pinned=True, workload=WORKLOAD):
    """The graph and this rank's slice of a batch of n_scen * world scenarios."""
    import torch
    from paper_2412_12487_gb300 import sharding as SH
    from paper_2412_12487_gb300 import workloads as W
    c = W.config(workload)
    c = W.GPTConfig(**{**c.__dict__, "n_scen": n_scen or c.n_scen})
    t0 = time.time()
    g = W.build_gpt_graph(c)
    s0, s1 = SH.shard_bounds(c.n_scen * world, world, rank)
    sc = SH.slice_scenarios(W.scenario_params(c, c.n_scen * world), s0, s1)
    V, S = g.n_ops, sc.n_scen
    dur_t = pinned_host_array((V, S)) if pinned else torch.empty((V, S), dtype=torch.int64)
    W.durations(g, sc.peak_flop_per_ns, out=dur_t.numpy())
    log(f"[rank {rank}] inputs: V={V} S={S} dur={V * S * 8 / 1e9:.2f} GB ({time.time() - t0:.1f}s)")
    return c, g, sc, dur_t


def algorithmic_bytes(g, info, S):
    """Bytes each kernel of one step must move (reuse of values written in the same
    pass is not counted):
      compose           first composition: every compute/memcpy duration read, the
                        finishes that a later step reads written (all of them for the
                        dataflow composer), the graph arrays, the CC table;
      compose_adjusted  final composition: durations read and every finish written,
                        plus the validator's rows of the candidates;
      overlap           validator: each candidate's finish and duration read, its
                        next duration written, the comm rows its cursors visit."""
    from paper_2412_12487_gb300 import workloads as W
    v_cd = int(((g.kind == W.KIND_COMPUTE) | (g.kind == W.KIND_MEMCPY)).sum())
    v_comm = g.n_ops - v_cd
    graph = 8 * (g.n_ops + 1) + 4 * g.n_edges + 4 * g.n_ops
    cc = 16 * info["n_signatures"] * S
    n_cand, n_kept, n_ce = info["n_overlap_candidates"], info["n_kept_finishes"], info["n_validator_comm_entries"]
    return {"compose": S * (8 * v_cd + 8 * n_kept) + graph + cc,
            "compose_adjusted": S * (16 * v_cd + 8 * v_comm + 8 * n_cand) + graph + cc,
            "overlap": S * (24 * n_cand + 16 * n_ce)}


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except Exception:  # pragma: no cover
        pass
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu part")):
                return line.split(":", 1)[1].strip()
    except OSError:  # pragma: no cover
        pass
    return "unknown"


def run_echo(args):
    import torch
    import torch.distributed as dist
    from paper_2412_12487_gb300 import Echo
    from paper_2412_12487_gb300 import sharding as SH

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    c, g, sc, dur_t = build_inputs(rank, world, args.scenarios, workload=args.workload)
    V, S = g.n_ops, sc.n_scen
    # a stream of its own: the events below and every library launch share it
    stream = torch.cuda.Stream(local)
    torch.cuda.set_stream(stream)
    e = Echo(local, stream)
    t0 = time.time()
    e.load_graph(g)
    e.load_scenarios(sc, dur=dur_t)
    info = e.info()
    log(f"[rank {rank}] loaded in {time.time() - t0:.1f}s: {info}")

    def step():
        e.estimate_collectives()
        e.compose(refine_passes=1)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize()

    clocks = Clocks(local if world == 1 else None)
    # device-resident timing
    e.set_profiling(True)
    e.read_profile()
    barrier()
    clocks.start()
    ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        step()
    ev1.record(stream)
    barrier()
    clk = clocks.stop()
    prof = e.read_profile()
    e.set_profiling(False)
    ms = ev0.elapsed_time(ev1) / args.steps
    # end to end through the public API, every step: that step's durations copied in
    # from pinned host memory, the makespans read out.  Two contexts on two streams take
    # alternate steps from two host threads (the library releases the GIL in every
    # call), so one step's upload overlaps the other's compute, as a serving loop would.
    import threading
    # every synthetic duration fits 32 bits, so the upload takes int32 (half the bytes)
    dur32 = pinned_host_array((V, S), np.int32)
    dur32.numpy()[:] = dur_t.numpy()
    assert int(dur_t.numpy().max()) < 2**31
    stream2 = torch.cuda.Stream(local)
    e2 = Echo(local, stream2)
    e2.load_graph(g)
    pipes = [(e, stream), (e2, stream2)]
    mk_host = [torch.empty(S, dtype=torch.int64, pin_memory=True) for _ in pipes]

    def e2e_steps_on(k, n):
        ctx = pipes[k][0]
        for _ in range(n):
            ctx.load_scenarios(sc, dur=dur32)
            ctx.estimate_collectives()
            ctx.compose(refine_passes=1)
            ctx.read_makespan(out=mk_host[k].numpy())

    def run_pipelined(n):
        ts = [threading.Thread(target=e2e_steps_on, args=(k, n // 2 + (1 if k < n % 2 else 0))) for k in range(2)]
        for t_ in ts:
            t_.start()
        for t_ in ts:
            t_.join()

    run_pipelined(4)
    e2e_steps = 2 * max(2, min(args.steps, 10) // 2)
    barrier()
    ev0.record(stream)
    stream2.wait_event(ev0)
    run_pipelined(e2e_steps)
    ev1.record(stream)
    ev2 = torch.cuda.Event(enable_timing=True)
    ev2.record(stream2)
    barrier()
    e2e_ms = max(ev0.elapsed_time(ev1), ev0.elapsed_time(ev2)) / e2e_steps
    e2.close()

    ms, e2e_ms = SH.max_over_ranks([ms, e2e_ms], device=torch.device("cuda", local))
    units = 2 * V * S  # two compose passes per step
    value = units * world / (ms / 1e3)
    e2e_value = units * world / (e2e_ms / 1e3)

    launches = sum(n for k, (n, _) in prof.items() if k != "dur_copy")  # kernels only
    peak, peak_kind = measured_peaks()
    alg = algorithmic_bytes(g, info, S)
    composer = "dataflow" if info["sigma"] == 32 else "levelled"
    kernels = {}
    for k, (n, t_) in prof.items():
        ent = {"launches": n, "ms_per_launch": t_ / max(n, 1)}
        if k in alg and n:
            ach = alg[k] / (t_ / n / 1e3) / 1e9
            ent.update({"alg_bytes_per_launch": alg[k], "achieved_gbs": ach, "frac": ach / peak})
        kernels[k] = ent
    # the dominant kernel of the step (largest total time) carries the roofline
    dom = max((k for k in alg if k in prof), key=lambda k: prof[k][1], default=None)
    traffic = None
    if dom:
        traffic = profiled_traffic(args.workload, dom, V * S)
    roof = {"kernel": dom, "bound": "hbm", "achieved": kernels[dom]["achieved_gbs"] if dom else None,
            "peak": peak, "peak_source": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)",
            "unit": "GB/s", "frac": kernels[dom]["frac"] if dom else None, "traffic": traffic,
            "alg_bytes_per_launch": alg.get(dom)}
    step_bytes = sum(alg[k] * prof[k][0] for k in alg if k in prof) / max(args.steps, 1)
    out = None
    if rank == 0:
        cpu = cpu_baseline(g, c, args) if world == 1 and args.cpu_sample > 0 else None
        h2d = V * S * 4 + 6 * S * 8 + sc.slowdown.size * 8  # int32 durations, fp64 parameters
        out = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": {"workload": f"{c.name} x {S} scenarios per GPU", "ops": V, "edges": g.n_edges,
                       "levels": info["n_levels"], "scenarios_per_gpu": S, "refine_passes": 1,
                       "sigma": info["sigma"], "composer": composer,
                       "updates_per_step": units,
                       "l2": f"no flush: the {V * S * 8 / 1e9:.1f} GB duration matrix and the "
                             f"finish matrices each exceed the 129 MB L2"},
            "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": S * 8,
                    "ms_per_step": e2e_ms,
                    "pipelining": "2 contexts on 2 streams take alternate steps (one's upload under the "
                                  "other's compute)",
                    "inputs": "durations as int32 (every value fits), composed in int64"},
            "gpu_launches": launches,
            "kernels": kernels,
            "roofline": roof,
            "step_alg_gbs": step_bytes / (ms / 1e3) / 1e9,
            "clocks": clk,
            "cpu_baseline": cpu,
        }
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    e.close()
    return out


def cpu_baseline(g, c, args):
    """The CPU oracle as it stands on the host cores, on bounded samples of the same
    workload (the batch's first scenarios): scenario-parallel on every core (the
    reported value), and single-threaded beside it.  One sample step = CC estimate,
    two compositions and the overlap test, as on the GPU."""
    import oracle
    from paper_2412_12487_gb300 import workloads as W
    cores = os.cpu_count() or 1
    base = W.scenario_params(c)
    n1 = min(max(1, args.cpu_sample), c.n_scen)
    sub = W.select_scenarios(base, g, list(range(n1)))
    t0 = time.time()
    oracle.compose(g, sub, refine_passes=1, threads=1, want_cc=False, want_overlap=False, want_times=False)
    dt1 = time.time() - t0
    nm = min(cores * max(1, args.cpu_sample // 2), c.n_scen)
    sub = W.select_scenarios(base, g, list(range(nm)))
    t0 = time.time()
    oracle.compose(g, sub, refine_passes=1, threads=cores, want_cc=False, want_overlap=False, want_times=False)
    dtm = time.time() - t0
    model = cpu_model()
    return {"value": 2 * g.n_ops * nm / dtm, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": f"{nm} of the {c.n_scen} scenarios of {c.name} ({g.n_ops} ops), one scenario per "
                      f"thread on {cores} threads: CC estimate + 2 compositions + overlap test, {dtm:.1f} s",
            "seconds": dtm, "cpu_model": model,
            "single_core": {"value": 2 * g.n_ops * n1 / dt1, "unit": UNIT, "cores": 1,
                            "sample": f"{n1} scenarios, single-threaded, {dt1:.1f} s"}}


CCQ_WORKLOAD = "cc-queries"


def cc_query_fp64_ops(q):
    """fp64 adds, multiplies and divides of each query's estimate, branch by branch
    as the closed forms of Sec. 5.3 evaluate them (ring: per-step size and time,
    steps times step, setup, reduction; tree: chunk size, beta, gamma, the four
    terms of Eq. 5; AUTO: both; send/recv: one chunk transfer times eta)."""
    from paper_2412_12487_gb300 import workloads as W
    n = q.cc_type.shape[0]
    add, mul, div = np.zeros(n), np.zeros(n), np.zeros(n)
    live = (q.n_ranks > 1) & (q.nbytes > 0)
    t, a, inter = q.cc_type, q.cc_algo, q.n_nodes > 1
    ring_ar = live & (t == W.CC_ALLREDUCE) & (a != W.ALGO_TREE)
    tree_ar = live & (t == W.CC_ALLREDUCE) & (a != W.ALGO_RING)
    for m, (ad, mu, dv) in ((live & (t == W.CC_SENDRECV), (2, 1, 2)), (live & (t == W.CC_ALLGATHER), (2, 2, 2)),
                            (live & (t == W.CC_REDUCESCATTER), (3, 3, 2)), (ring_ar, (3, 3, 2))):
        add[m] += ad
        mul[m] += mu
        div[m] += dv
    add[tree_ar] += 5 + inter[tree_ar]
    mul[tree_ar] += 6
    div[tree_ar] += 2 + inter[tree_ar]
    return float(add.sum()), float(mul.sum()), float(div.sum())


def run_cc_queries(args):
    """The standalone CC-estimator sweep (1M queries of Sec. 5.3's closed forms):
    queries/s of the estimator kernel (device time) and through the C ABI call
    (host arrays in, host results out), with the oracle's rate on a sample.  Its
    roofline is the fp64 rate of this device for the sweep's mix of adds,
    multiplies and divides (measured in the same run), beside the HBM bound of its
    82 bytes per query."""
    import torch
    import oracle
    from paper_2412_12487_gb300 import Echo, echo as E
    from paper_2412_12487_gb300 import workloads as W
    n = args.scenarios or 1_000_000
    q = W.make_cc_queries(n)
    stream = torch.cuda.Stream(0)
    torch.cuda.set_stream(stream)
    with Echo(0, stream) as e:
        for _ in range(args.warmup):
            e.cc_query(q)
        e.set_profiling(True)
        e.read_profile()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for _ in range(args.steps):
            out = e.cc_query(q)
        torch.cuda.synchronize()
        call_ms = (time.perf_counter() - t0) / args.steps * 1e3
        prof = e.read_profile()
    k_n, k_ms = prof.get("cc_query", (0, 0.0))
    kern_ms = k_ms / max(k_n, 1)
    rates = E.measure_fp64(0)
    n_add, n_mul, n_div = cc_query_fp64_ops(q)
    bound_s = n_add / rates["dadd"] + n_mul / rates["dmul"] + n_div / rates["ddiv"]
    ops = n_add + n_mul + n_div
    peak_hbm, peak_kind = measured_peaks()
    bytes_q = 1 + 1 + 8 + 4 + 4 + 6 * 8 + 8 + 8  # type, algo, size, N, M, parameters, log2 M in; estimate out
    oracle.build()
    m = min(n, 20000)
    t0 = time.perf_counter()
    ref = np.array([oracle.cc_ns(int(q.cc_type[i]), int(q.cc_algo[i]), int(q.nbytes[i]), int(q.n_ranks[i]),
                                 int(q.n_nodes[i]), -(-int(q.n_ranks[i]) // int(q.n_nodes[i])),
                                 float(np.log2(q.n_nodes[i])), float(q.alpha_ns[i]), float(q.bw_intra[i]),
                                 float(q.lat_intra[i]), float(q.bw_inter[i]), float(q.lat_inter[i]),
                                 float(q.delta[i])) for i in range(m)])
    cpu_s = time.perf_counter() - t0
    rel = float(np.max(np.abs(out[:m] - ref) / np.maximum(np.abs(ref), 1e-300)))
    return {"metric": "CC-estimator queries/s", "value": n / (kern_ms / 1e3), "unit": "queries/s",
            "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": kern_ms,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": f"{n} CC-estimator queries (Sec. 5.3)"},
            "e2e": {"value": n / (call_ms / 1e3), "unit": "queries/s", "ms_per_step": call_ms,
                    "h2d_bytes_per_step": n * (1 + 1 + 8 + 4 + 4 + 6 * 8), "d2h_bytes_per_step": n * 8},
            "gpu_launches": k_n,
            "roofline": {"kernel": "cc_query", "bound": "alu", "unit": "Gop/s",
                         "achieved": ops / (kern_ms / 1e3) / 1e9, "peak": ops / bound_s / 1e9,
                         "frac": bound_s / (kern_ms / 1e3), "traffic": None,
                         "peak_source": "fp64 add/mul/div rates measured in this run (echo_measure_fp64), "
                                        "weighted by the sweep's operation mix",
                         "fp64_ops_per_query": ops / n, "fp64_rates_per_s": rates},
            "roofline_hbm": {"bound": "hbm", "unit": "GB/s", "achieved": n * bytes_q / (kern_ms / 1e3) / 1e9,
                             "peak": peak_hbm, "frac": n * bytes_q / (kern_ms / 1e3) / 1e9 / peak_hbm,
                             "peak_source": f"{peak_kind} copy bandwidth", "bytes_per_query": bytes_q},
            "max_rel_diff_vs_oracle_sample": rel,
            "cpu_baseline": {"value": m / cpu_s, "unit": "queries/s", "cores": 1, "kind": "oracle",
                             "cpu_model": cpu_model(),
                             "sample": f"first {m} queries, one at a time through the oracle's C function"}}


def run_reference(args):
    """Reference arm: the CPU oracle (a plain event-driven simulator written from
    the paper) timed on the host cores on the same workload, each step one scenario
    per core composed in parallel (a bounded sample of the batch)."""
    rank, world, _ = dist_env()
    if rank != 0:
        return None
    import oracle
    from paper_2412_12487_gb300 import workloads as W
    c = W.config(args.workload)
    g = W.build_gpt_graph(c)
    base = W.scenario_params(c)
    cores = os.cpu_count() or 1
    oracle.build()

    def step(i):
        sub = W.select_scenarios(base, g, [(i * cores + k) % base.n_scen for k in range(cores)])
        t0 = time.time()
        oracle.compose(g, sub, refine_passes=1, threads=cores, want_cc=False, want_overlap=False, want_times=False)
        return time.time() - t0

    for i in range(args.warmup):
        step(i)
    dt = sum(step(args.warmup + i) for i in range(args.steps)) / args.steps
    v = 2 * g.n_ops * cores / dt
    return {"impl": "reference", "metric": METRIC, "value": v, "unit": UNIT, "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "int64", "data": "synthetic",
            "config": {"workload": f"{c.name} x {cores} scenarios per step, one per core (bounded sample of "
                                   f"the {c.n_scen}-scenario batch)", "ops": g.n_ops},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "cpu_model": cpu_model(),
                             "sample": f"{cores} scenarios per step, one per thread"},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="echo", choices=["echo", "reference"])
    ap.add_argument("--cpu-sample", type=int, default=8,
                    help="scenarios of the CPU-oracle baseline sample (0 = skip)")
    ap.add_argument("--workload", default=WORKLOAD,
                    help="workload name (default: the GPT-175B step); others for profiling and comparison")
    ap.add_argument("--scenarios", type=int, default=None,
                    help="scenarios per GPU (default: the workload's 1024); smaller values "
                         "make small cases for profiling")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "echo":
        log("note: warmup raised to 3")
        args.warmup = 3
    if args.impl == "reference":
        out = run_reference(args)
    elif args.workload == CCQ_WORKLOAD:
        import __graft_entry__
        __graft_entry__.build()
        out = run_cc_queries(args)
    else:
        import __graft_entry__
        __graft_entry__.build()
        out = run_echo(args)
    if out is not None:
        print(json.dumps(out), flush=True)


if __name__ == "__main__":
    main()
