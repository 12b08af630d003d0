#!/usr/bin/env python
"""Fork-decode attention benchmark (one JSON line on rank 0).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--impl ours|reference]

A step is one complete fork-decode call (prefix stage + suffix stage + merge)
for every fork of the workload: one decode token per fork, one attention layer.
Metric: tokens/s = forks per step / seconds per step.  The default workload is
the largest one, the ragged multi-trace batch: 8 independent reasoning traces
with prefixes uniform in [4096, 32768] tokens, each forked into 4-16 branches
with suffixes uniform in [32, 1024], Hq=64, Hkv=8, head dim 128, page 16,
shuffled pages (708 MB of unique KV with its seed); ``--workload`` picks the
others.

Timing: W untimed warm-up steps, then K steps between CUDA events on the
launching stream, bracketed by a barrier and a device synchronise.  Inputs
rotate over enough resident replicas that every step's KV is evicted from L2
before it is read again (the union of replicas is >= 3x L2).  Steps replay
CUDA graphs of 16 library calls.  Each kernel's average launch time comes from
graphs of its stage alone (specgen_fork_attn_run_partials / _run_merge) run
back to back over the same replicas after the timed region, timed with events
on the same stream.

With N > 1 (torchrun) every rank runs its own replica of the workload: fork
decode shards by independent traces with no exchange, so scaling is weak and
no collective is used.  ``--impl reference`` times the fp64 CPU oracle instead.
"""

from __future__ import annotations

import argparse
import json
import math
import os
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
DEFAULT_WORKLOAD = "ragged_t8"


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=2000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--op", choices=["attend", "decode_step", "pack", "prefill", "cascade"],
                    default="attend",
                    help="attend: one fork-decode attention call per step (the headline); "
                         "decode_step: append one K/V row per fork, then attend over the grown "
                         "suffixes, one plan for all steps; pack: move every trace's prefix "
                         "pages into one buffer and back (remote prefix cache); prefill: "
                         "causal prefill of a --chunk-token prompt chunk per fork; cascade: "
                         "decode over nested prefixes (fork events at 4096 and 8192 tokens, "
                         "8 forks each), timed beside the same forks as flat traces")
    ap.add_argument("--chunk", type=int, default=64, help="prefill chunk tokens per fork")
    ap.add_argument("--kv-layout", choices=["rows", "tiled"], default="tiled",
                    help="K/V pool layout: 8x8 core-matrix tiles (default; one bulk copy per "
                         "page and head, the faster layout on the default workload) or "
                         "token-major rows; latent (MLA) pools are always rows")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-secondary", action="store_true",
                    help="skip the other configurations' summary lines (`secondary`)")
    ap.add_argument("--cpu-sample-seconds", type=float, default=20.0)
    return ap.parse_args()


ARGS = parse_args()
if ARGS.impl == "reference" or os.environ.get("SPECGEN_ORACLE_CHILD"):
    # the oracle runs single-threaded so that `cores` is exact
    for var in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS"):
        os.environ[var] = "1"

sys.path.insert(0, ROOT)
import numpy as np  # noqa: E402

METRIC = "fork-decode attention tokens/s"


def log(*a):
    print(*a, file=sys.stderr, flush=True)


def dist_env():
    return (int(os.environ.get("RANK", 0)), int(os.environ.get("LOCAL_RANK", 0)),
            int(os.environ.get("WORLD_SIZE", 1)))


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            d = json.load(fh)
        return float(d["hbm_gbs"]), float(d["bf16_tflops"]), float(d["bf16_tflops_sustained"]), \
            "measured"
    except Exception:
        return 6800.0, 1900.0, 1700.0, "fallback"


# --------------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples of SM clock and throttle reasons while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines: list[str] = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def _query_once(self):
        try:
            out = subprocess.run(["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                                  "--format=csv,noheader,nounits"], capture_output=True,
                                 text=True, timeout=20).stdout
            return [l for l in out.splitlines() if l.strip()]
        except Exception:
            return []

    def stop(self):
        if self.proc is not None:
            self.proc.terminate()
            try:
                out, _ = self.proc.communicate(timeout=10)
            except Exception:
                self.proc.kill()
                out = ""
            self.lines = [l for l in (out or "").splitlines() if l.strip()]
        extra = self._query_once()
        samples = self.lines or extra
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in samples:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = float(parts[2])
            except ValueError:
                continue
            for name, val in zip(names, parts[5:9]):
                if val.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": float(np.median(sm)) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# --------------------------------------------------------------------------- CPU oracle
def oracle_sample(workload: str, seconds: float, first_fork: int = 0):
    """Time the fp64 oracle (as it stands) on whole forks until ~`seconds` pass."""
    import oracle
    from paper_2606_17518_gb300 import workloads as wl
    w = wl.make_workload(workload)
    forks = 0
    t0 = time.perf_counter()
    while True:
        f = (first_fork + forks) % w["total_forks"]
        oracle.fork_attn_decode_rows(w, [(f, h) for h in range(w["hq"])])
        forks += 1
        if time.perf_counter() - t0 >= seconds or forks >= 10000:
            break
    dt = time.perf_counter() - t0
    return forks, dt


def cpu_model() -> str:
    """The host CPU as /proc/cpuinfo names it (model name, else the Arm part number)."""
    try:
        info = open("/proc/cpuinfo").read()
    except OSError:
        return "unknown"
    for key in ("model name", "Model Name"):
        for line in info.splitlines():
            if line.split(":")[0].strip() == key:
                return line.split(":", 1)[1].strip()
    fields = {}
    for line in info.splitlines():
        if ":" in line:
            k, v = (x.strip() for x in line.split(":", 1))
            fields.setdefault(k, v)
    parts = [f"{k} {fields[k]}" for k in ("CPU implementer", "CPU part", "CPU variant")
             if k in fields]
    return "Arm, " + ", ".join(parts) if parts else "unknown"


def _oracle_children(workload: str, seconds: float, n: int):
    """`n` single-threaded oracle processes at once, each from its own first fork."""
    env = dict(os.environ, SPECGEN_ORACLE_CHILD="1", OMP_NUM_THREADS="1",
               OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    procs = []
    for i in range(n):
        code = ("import json,sys; sys.argv=['bench.py','--impl','reference']; import bench; "
                f"f,dt=bench.oracle_sample({workload!r},{seconds},{i}); "
                "print(json.dumps([f,dt]))")
        procs.append(subprocess.Popen([sys.executable, "-c", code], cwd=ROOT, env=env,
                                      stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                      text=True))
    out = []
    for pr in procs:
        stdout, _ = pr.communicate(timeout=600)
        out.append(json.loads(stdout.strip().splitlines()[-1]))
    return out


def cpu_baseline(workload: str, seconds: float):
    [(forks, dt)] = _oracle_children(workload, seconds, 1)
    return {"value": forks / dt, "unit": "tokens/s", "cores": 1, "kind": "oracle",
            "cpu": cpu_model(),
            "sample": f"{forks} whole forks (all heads) of {workload}, fp64 numpy, "
                      f"{dt:.1f} s on 1 host thread"}


def cpu_baseline_all_cores(workload: str, seconds: float, unique_bytes: int):
    """The same oracle on every host core at once (one single-threaded process per
    core, up to 16, over different forks); tokens/s = the sum of their rates."""
    n = min(16, os.cpu_count() or 1)
    if unique_bytes > (1 << 30):  # every process holds its own copy of the workload
        return None
    res = _oracle_children(workload, seconds, n)
    forks = sum(f for f, _ in res)
    return {"value": sum(f / dt for f, dt in res), "unit": "tokens/s", "cores": n,
            "kind": "oracle", "cpu": cpu_model(),
            "sample": f"{forks} whole forks of {workload} over {n} single-threaded processes, "
                      f"{max(dt for _, dt in res):.1f} s each at most"}


# --------------------------------------------------------------------------- reference arm
def run_reference():
    rank, _, world = dist_env()
    if rank != 0:
        return
    import oracle
    from paper_2606_17518_gb300 import workloads as wl
    w = wl.make_workload(ARGS.workload)
    F, hq = w["total_forks"], w["hq"]
    # a step is a bounded sample: one eighth of a fork's query heads (a token is
    # one fork's every head), cycling over forks and head blocks, so that a
    # run of thousands of steps still ends within minutes
    hb = hq // 8 if hq % 8 == 0 else 1
    blocks = [(f, h0) for f in range(F) for h0 in range(0, hq, hb)]

    def step(i):
        f, h0 = blocks[i % len(blocks)]
        oracle.fork_attn_decode_rows(w, [(f, h) for h in range(h0, h0 + hb)])

    for i in range(ARGS.warmup):
        step(i)
    t0 = time.perf_counter()
    for i in range(ARGS.steps):
        step(i)
    dt = time.perf_counter() - t0
    value = ARGS.steps * hb / hq / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": ARGS.gpus, "steps": ARGS.steps, "warmup": ARGS.warmup,
        "ms_per_step": dt / ARGS.steps * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": ARGS.workload, "step": f"{hb} of a fork's {hq} query heads "
                   "per step (a token is one fork's every head), cycling over forks"},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": 1, "kind": "oracle",
                         "sample": f"{ARGS.steps} blocks of {hb} query heads of "
                                   f"{ARGS.workload}, fp64 numpy, 1 host thread"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# --------------------------------------------------------------------------- GPU arm
# source files of each kernel (a stage of concurrent kernels is named "a+b")
KERNEL_SOURCES = {"fork_tc": "fork_tc", "fork_suffix": "suffix_stage", "mla_tc": "mla_tc",
                  "split_decode": "split_decode", "lse_merge": "lse_merge"}


def kernel_source_sha(name: str) -> str:
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2606_17518_gb300", "csrc")
    stems = [KERNEL_SOURCES.get(k, k) for k in name.split("+")]
    for fn in sorted(os.listdir(csrc)):
        if any(fn.startswith(st) for st in stems) or fn in ("common.cuh", "plan.h", "tc_common.cuh"):
            with open(os.path.join(csrc, fn), "rb") as fh:
                h.update(fh.read())
    return h.hexdigest()[:16]


def recorded_profile(kernel: str, workload: str):
    """The committed ncu record of a kernel on a workload (DRAM bytes and
    tensor-pipe activity per launch), if the kernel's sources are unchanged
    since it was taken; else None."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    try:
        with open(path) as fh:
            d = json.load(fh)
        rec = d[kernel][workload]
        if rec.get("source_sha") != kernel_source_sha(kernel):
            return None
        return rec
    except Exception:
        return None


def recorded_traffic(kernel: str, workload: str):
    """DRAM bytes per launch from the committed ncu summary, if still current."""
    rec = recorded_profile(kernel, workload)
    return float(rec["dram_bytes_per_launch"]) if rec else None


def run_ours():
    import ctypes as C

    import torch

    import __graft_entry__
    from paper_2606_17518_gb300 import _lib, workloads as wl
    from paper_2606_17518_gb300.fork_attn import ForkDecode

    rank, local_rank, world = dist_env()
    __graft_entry__.build()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)

    def barrier():
        if world > 1:
            import torch.distributed as dist
            dist.barrier()

    w = wl.make_workload(ARGS.workload)
    nbytes = wl.algorithmic_bytes(w)
    flops = wl.algorithmic_flops(w)
    F = w["total_forks"]
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 126 * 2 ** 20))
    replicas = max(1, math.ceil(3 * l2 / nbytes["total"]))
    log(f"[bench] {ARGS.workload}: {nbytes['total'] / 1e6:.1f} MB unique, L2 {l2 / 2**20:.0f} MiB,"
        f" {replicas} replicas")
    stream = torch.cuda.Stream(dev)
    sp = stream.cuda_stream
    layout = ARGS.kv_layout if w["v_pages"] is not None else "rows"
    kv_layout = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    reps = [ForkDecode(w, device=dev, kv_layout=kv_layout) for _ in range(replicas)]
    with torch.cuda.stream(stream):
        for r in reps:
            r.plan(sp)
    torch.cuda.synchronize(dev)
    args = [r.args() for r in reps]
    plans = [r.plan_info for r in reps]

    # Timed steps replay CUDA graphs.  Each graph holds `per_graph` consecutive
    # steps (one library call each, on rotating replicas) so that host launch
    # overhead never starves the GPU.  K is covered exactly: full graphs plus
    # one remainder graph.  Per-kernel times come from graphs of one stage
    # alone (specgen_fork_attn_run_partials / _run_merge, back to back on the
    # same stream and replicas), timed with events after the timed region.
    K, W = ARGS.steps, ARGS.warmup
    per_graph = max(1, min(16, K))
    lib = _lib.load()
    arg_refs = [C.byref(a) for a in args]
    plan_refs = [C.byref(p) for p in plans]
    sp_c = C.c_void_p(sp)
    for i in range(2):  # first calls configure the kernels outside any capture
        st = lib.specgen_fork_attn_run(arg_refs[i % replicas], plan_refs[i % replicas], sp_c)
        assert st == 0, _lib.status_string(st)
    torch.cuda.synchronize(dev)

    def make_graph(first_step, n_steps, call=lib.specgen_fork_attn_run):
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for k in range(n_steps):
                r = (first_step + k) % replicas
                st = call(arg_refs[r], plan_refs[r], sp_c)
                if st != 0:
                    break
        if st != 0:
            raise RuntimeError(_lib.status_string(st))
        return graph, None

    n_full, rem = divmod(K, per_graph)
    n_distinct = max(1, min(n_full, 8))
    full_graphs = [make_graph(g * per_graph, per_graph) for g in range(n_distinct)] if n_full else []
    rem_graph = make_graph(0, rem) if rem else None
    schedule = [full_graphs[i % n_distinct] for i in range(n_full)] + ([rem_graph] if rem else [])
    for i in range(max(1, (W + per_graph - 1) // per_graph)):
        schedule[i % len(schedule)][0].replay()
    torch.cuda.synchronize(dev)
    start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local_rank)
    barrier()
    torch.cuda.synchronize(dev)
    clocks.start()
    # an event after every graph as well: per-graph step times give the median
    # and the best step next to the mean
    marks = [torch.cuda.Event(enable_timing=True) for _ in schedule]
    with torch.cuda.stream(stream):
        start.record(stream)
        for (graph, _), mk in zip(schedule, marks):
            graph.replay()
            mk.record(stream)
        end.record(stream)
    torch.cuda.synchronize(dev)
    barrier()
    clk = clocks.stop()
    total_ms = start.elapsed_time(end)
    graph_steps = [per_graph] * n_full + ([rem] if rem else [])
    prev, per_step_us = start, []
    for mk, n in zip(marks, graph_steps):
        per_step_us.append(prev.elapsed_time(mk) * 1e3 / n)
        prev = mk
    # per-kernel times: each stage alone, back to back, over the same replicas
    def stage_ms(call):
        g_list = [make_graph(g * per_graph, per_graph, call)[0]
                  for g in range(max(1, min(8, K // per_graph)))]
        for g in g_list:
            g.replay()
        torch.cuda.synchronize(dev)
        t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        n_rep = max(1, min(64, (K + per_graph * len(g_list) - 1) // (per_graph * len(g_list))))
        with torch.cuda.stream(stream):
            t0.record(stream)
            for _ in range(n_rep):
                for g in g_list:
                    g.replay()
            t1.record(stream)
        torch.cuda.synchronize(dev)
        return t0.elapsed_time(t1) / (n_rep * len(g_list) * per_graph)

    tc_name = "mla_tc" if w["v_pages"] is None else "fork_tc"
    # the partial-attention kernels of a step: the prefix kernel and, beside it
    # on the SMs it leaves free, the suffix stage (they run concurrently, so
    # they are timed together as one stage), or the split-K kernel
    part_kernels = ([tc_name] if plans[0].n_tc_ctas > 0 else []) + \
        (["fork_suffix"] if plans[0].n_sfx_ctas > 0 else []) + \
        (["split_decode"] if plans[0].n_split_items > 0 else [])
    partials_ms = stage_ms(lib.specgen_fork_attn_run_partials)
    merge_ms = stage_ms(lib.specgen_fork_attn_run_merge)
    suffix_stage = measure_suffix_stage(w, reps, kv_layout, stream, dev, per_graph, nbytes)
    suffix_steady = (measure_suffix_steady(stream, dev, kv_layout)
                     if w["v_pages"] is not None else None)
    kernel_names = ["+".join(part_kernels), "lse_merge"]
    kernel_ms = [partials_ms, merge_ms]
    launches = len(part_kernels) + 1
    n_slots = per_graph * max(1, min(8, K // per_graph))
    status = reps[0].status(sp)
    if status != 0:
        raise RuntimeError(f"workspace status {_lib.status_string(status)}")

    if world > 1:
        import torch.distributed as dist
        t = torch.tensor([total_ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    ms_per_step = total_ms / K
    value = world * F / (ms_per_step * 1e-3)

    # ---- end to end through the public API: host buffers, copies in the timed region
    e2e = measure_e2e(w, reps, stream, dev, K=min(K, 500), W=min(W, 5))

    dom = int(np.argmax(kernel_ms)) if kernel_ms else 0
    hbm, tf_burst, tf_sus, peak_src = measured_peaks()
    # algorithmic bytes of the dominant launch: what that kernel must read/write once
    dom_name = kernel_names[dom] if kernel_names else None
    if dom_name != "lse_merge":
        # the kernel that reads the KV: unique prefix + every suffix + Q
        dom_bytes = nbytes["prefix"] + nbytes["suffix"] + nbytes["q"]
    else:
        dom_bytes = nbytes["total"]
    achieved = dom_bytes / (kernel_ms[dom] * 1e-3) / 1e9 if kernel_ms else None
    traffic = recorded_traffic(kernel_names[dom], f"{ARGS.workload}:{layout}")
    if dom_name.startswith("mla_tc"):
        # latent attention is a dense contraction (the 128 heads of a fork share
        # every latent key): bound by the bf16 tensor pipe, timed inside a long
        # loop of steps, so against the sustained bf16 peak
        tflops = flops["total"] / (kernel_ms[dom] * 1e-3) / 1e12
        roofline = {"bound": "tensor", "kernel": dom_name, "achieved": tflops, "peak": tf_sus,
                    "unit": "TFLOP/s", "frac": tflops / tf_sus, "traffic": traffic,
                    "peak_source": peak_src + " (bf16, sustained)",
                    "algorithmic_flops_per_launch": flops["total"],
                    "hbm_achieved_gbs": achieved}
    else:
        roofline = {"bound": "hbm", "kernel": dom_name, "achieved": achieved, "peak": hbm,
                    "unit": "GB/s", "frac": achieved / hbm if achieved else None,
                    "traffic": traffic, "peak_source": peak_src,
                    "algorithmic_bytes_per_launch": dom_bytes}

    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": W, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {
            "workload": ARGS.workload, "traces": w["num_traces"], "forks": F,
            "prefix_tokens": int(np.sum(w["prefix_lens"])),
            "suffix_tokens": int(np.sum(w["suffix_lens"])), "hq": w["hq"], "hkv": w["hkv"],
            "head_dim": [w["dqk"], w["dv"]], "page_size": w["page_size"], "kv_layout": layout,
            "unique_bytes": nbytes["total"], "flops": flops["total"],
            "l2": f"inputs rotate over {replicas} resident replicas (>= 3x L2)",
            "timing": f"CUDA graphs of {per_graph} steps; per-kernel times from graphs of "
                      f"one stage alone ({n_slots} distinct steps, replayed back to back after "
                      f"the timed region)",
            "parallelism": f"replicas x{world}",
        },
        "gpu_launches": K * launches,
        "kernels": {n: {"ms_per_launch": t, "share": t / max(1e-12, sum(kernel_ms))}
                    for n, t in zip(kernel_names, kernel_ms)},
        "step_us": {"mean": ms_per_step * 1e3, "median": float(np.median(per_step_us)),
                    "best": float(np.min(per_step_us)), "graphs": len(per_step_us)},
        "achieved_gbs_whole_step": nbytes["total"] / (ms_per_step * 1e-3) / 1e9,
        # the metric's other two parts: the dominant kernel's algorithmic GB/s
        # against the nominal 8 TB/s of HBM3e, and the prefix read amplification
        # (DRAM bytes of the recorded ncu capture, less the suffix, Q and output
        # bytes, over the unique prefix bytes; null without a current record)
        "hbm_vs_8tbs": (achieved / 8000.0) if achieved else None,
        "prefix_read_amplification": (
            (traffic - nbytes["suffix"] - nbytes["q"] - nbytes["out"]) / nbytes["prefix"]
            if traffic is not None and nbytes["prefix"] > 0 else None),
        # the suffix stage alone (diagnostic plan with empty prefixes), and the
        # suffix-stage kernel's streaming rate on a call large enough to amortise
        # its fixed per-call latency
        "suffix_stage": suffix_stage,
        "suffix_stage_steady": suffix_steady,
        # tensor-pipe activity of the dominant kernel from the recorded ncu capture
        "tensor_pipe_pct": (recorded_profile(kernel_names[dom], f"{ARGS.workload}:{layout}")
                            or {}).get("tensor_pipe_pct"),
        "roofline": roofline,
        "clocks": {k: clk[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")},
        "e2e": e2e,
    }
    if rank == 0 and world == 1 and not ARGS.no_cpu_baseline:
        try:
            line["cpu_baseline"] = cpu_baseline(ARGS.workload, ARGS.cpu_sample_seconds)
            line["cpu_baseline_all_cores"] = cpu_baseline_all_cores(
                ARGS.workload, ARGS.cpu_sample_seconds / 2, nbytes["total"])
        except Exception as exc:  # reported, never silently dropped
            line["cpu_baseline"] = {"error": repr(exc)[:200]}
    if rank == 0 and world == 1 and not ARGS.no_secondary:
        line["secondary"] = secondary_workloads(K, W)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


# the other configurations of the benchmark: c2 (8k prefix, 8 forks), c3 (32k
# prefix, 16 forks) and c5 (latent KV)
SECONDARY = ("fork_p8k_f8", "long_p32k_f16", "mla_p16k_f8")


def secondary_workloads(K, W):
    """The other configurations, each measured by this script in a child process
    of its own (`--workload NAME`, same steps and warm-up, no CPU baseline) after
    the main measurement, and summarised here: their rates, per-kernel times,
    rooflines and end-to-end rates, so that one default run records every
    configuration.  A child that fails is reported with its error."""
    out = {}
    for name in SECONDARY:
        if name == ARGS.workload:
            continue
        cmd = [sys.executable, os.path.abspath(__file__), "--workload", name, "--no-cpu-baseline",
               "--no-secondary", "--steps", str(K), "--warmup", str(W)]
        try:
            r = subprocess.run(cmd, capture_output=True, text=True, timeout=600, cwd=ROOT)
            if r.returncode != 0:
                raise RuntimeError(f"exit {r.returncode}: {r.stderr.strip()[-160:]}")
            d = json.loads(r.stdout.strip().splitlines()[-1])
            out[name] = {k: d.get(k) for k in ("value", "unit", "ms_per_step", "kernels",
                                                "roofline", "tensor_pipe_pct", "clocks")}
            out[name]["e2e"] = (d.get("e2e") or {}).get("value")
            out[name]["config"] = d.get("config")
        except Exception as exc:  # reported, never silently dropped
            out[name] = {"error": repr(exc)[:240]}
    return out


def measure_suffix_stage(w, reps, kv_layout, stream, dev, per_graph, nbytes):
    """The suffix stage alone: the same forks, queries and suffix pages with empty
    prefixes, so that the partial-attention kernels read only the suffix KV (a
    diagnostic plan: the suffix-stage kernel alone on every SM, where the plan
    splits; the step itself runs the prefix and suffix stages together).
    GB/s = (suffix KV + Q bytes) / the kernel's time, against the nominal 8 TB/s
    and the measured copy bandwidth."""
    import ctypes as C

    import torch

    from paper_2606_17518_gb300 import _lib
    if nbytes["suffix"] <= 0 or "segment_rows" in w:
        return None
    import copy
    lib = _lib.load()
    fds = []
    for r in reps:
        fd = copy.copy(r)  # the replica's device tensors, its own lengths and workspace
        fd.w = dict(r.w)
        fd.w["prefix_lens"] = np.zeros_like(r.w["prefix_lens"])
        fd.workspace, fd.ws_bytes = None, 0
        fd.set_suffix_lens(fd.w["suffix_lens"], update_device=False)
        with torch.cuda.stream(stream):
            fd.plan(stream.cuda_stream)
        fds.append(fd)
    torch.cuda.synchronize(dev)
    keep = [fd.args() for fd in fds]  # the structs outlive the graph capture
    arg_refs = [C.byref(a) for a in keep]
    plan_refs = [C.byref(fd.plan_info) for fd in fds]
    sp_c = C.c_void_p(stream.cuda_stream)
    st = lib.specgen_fork_attn_run_partials(arg_refs[0], plan_refs[0], sp_c)
    assert st == 0, _lib.status_string(st)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for k in range(per_graph):
            st = lib.specgen_fork_attn_run_partials(arg_refs[k % len(fds)], plan_refs[k % len(fds)],
                                                    sp_c)
            assert st == 0, _lib.status_string(st)
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize(dev)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n_rep = 32
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(n_rep):
            graph.replay()
        t1.record(stream)
    torch.cuda.synchronize(dev)
    ms = t0.elapsed_time(t1) / (n_rep * per_graph)
    hbm, _, _, _ = measured_peaks()
    gbs = (nbytes["suffix"] + nbytes["q"]) / (ms * 1e-3) / 1e9
    return {"kernel_us": ms * 1e3, "bytes_per_launch": nbytes["suffix"] + nbytes["q"],
            "gbs": gbs, "vs_8tbs": gbs / 8000.0, "vs_measured": gbs / hbm,
            "plan": "same forks, queries and suffix pages; empty prefixes"}


def measure_suffix_steady(stream, dev, kv_layout):
    """The suffix-stage kernel alone on a suffix-only call large enough that its
    fixed per-call latency (start, ramp, tail: a few microseconds) is amortised:
    64 forks of one trace with 2048-token suffixes and no prefix (538 MB of KV,
    Hq=64, Hkv=8, head dim 128, page 16).  Its GB/s is the kernel's streaming
    rate, against the nominal 8 TB/s and the measured copy bandwidth."""
    import ctypes as C

    import torch

    from paper_2606_17518_gb300 import _lib, workloads as wl
    from paper_2606_17518_gb300.fork_attn import ForkDecode
    spec = wl.DIAGNOSTIC["suffix_only_f64_s2048"]
    w = wl.make_workload(spec)
    fd = ForkDecode(w, device=dev, kv_layout=kv_layout)
    sp = stream.cuda_stream
    with torch.cuda.stream(stream):
        fd.plan(sp)
    torch.cuda.synchronize(dev)
    if fd.plan_info.n_sfx_ctas == 0:
        return None
    lib = _lib.load()
    args = fd.args()
    ref = (C.byref(args), C.byref(fd.plan_info), C.c_void_p(sp))
    st = lib.specgen_fork_attn_run_partials(*ref)
    assert st == 0, _lib.status_string(st)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph, stream=stream):
        for _ in range(8):
            st = lib.specgen_fork_attn_run_partials(*ref)
            assert st == 0, _lib.status_string(st)
    for _ in range(3):
        graph.replay()
    torch.cuda.synchronize(dev)
    t0, t1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    n_rep = 8
    with torch.cuda.stream(stream):
        t0.record(stream)
        for _ in range(n_rep):
            graph.replay()
        t1.record(stream)
    torch.cuda.synchronize(dev)
    ms = t0.elapsed_time(t1) / (n_rep * 8)
    nb = wl.algorithmic_bytes(w)
    nbytes = nb["suffix"] + nb["q"]
    hbm, _, _, _ = measured_peaks()
    gbs = nbytes / (ms * 1e-3) / 1e9
    status = fd.status(sp)
    del fd
    torch.cuda.empty_cache()
    if status != 0:
        raise RuntimeError(f"workspace status {status}")
    return {"kernel_us": ms * 1e3, "bytes_per_launch": nbytes, "gbs": gbs, "vs_8tbs": gbs / 8000.0,
            "vs_measured": gbs / hbm, "workload": spec.name,
            "plan": "64 forks x 2048 suffix tokens, no prefix: the suffix-stage kernel alone"}


def measure_e2e(w, reps, stream, dev, K, W):
    """tokens/s through specgen_fork_attn_decode_staged_inline with host-resident inputs.

    Every step is one library call that plans on the host, copies that step's
    queries, block tables and plan from pinned host memory (in one copy while
    the GPU is still busy with earlier steps; inputs first and plan after the
    planning when it is idle), runs the attention, and reads O and LSE back
    into pinned host memory.  The KV pools
    are the serving cache and stay resident.  A step's inputs travel as one
    packed buffer (Q, then the four table arrays, each at a 256-byte boundary,
    then room for the plan region) and its outputs as another (O, then LSE).
    The call writes the plan into the pinned input buffer, so the loop keeps a
    ring of them (at least 16, a multiple of the replicas) in two halves, and
    before it starts a half it waits for an event recorded after the last call
    that used that half: a buffer is reused only once the call that last read
    it has finished, and the host runs up to one and a half halves ahead of the
    GPU (one event call per half, none per step).
    """
    import ctypes as C

    import torch

    from paper_2606_17518_gb300 import _lib
    replicas = len(reps)
    sp = stream.cuda_stream
    align = lambda n: (n + 255) // 256 * 256
    n_host = 2 * replicas * max(1, -(-8 // replicas))
    half = n_host // 2

    def pack(tensors, extra=0):
        """One device buffer holding copies of `tensors` (256-byte aligned views,
        then `extra` bytes); returns (device bytes, bytes used, views)."""
        offs, n = [], 0
        for t in tensors:
            offs.append(n)
            n = align(n + t.numel() * t.element_size())
        dbuf = torch.zeros(n + extra, dtype=torch.uint8, device=dev)
        views = []
        for t, o in zip(tensors, offs):
            v = dbuf[o:o + t.numel() * t.element_size()].view(t.dtype).view(t.shape)
            v.copy_(t)
            views.append(v)
        return dbuf, n, views

    staged = []
    for r in reps:
        region = int(r.plan_info.ws_plan_off + r.plan_info.plan_bytes)
        din, in_bytes, (r.q, r.prefix_table, r.prefix_off, r.suffix_table, r.suffix_off) = pack(
            [r.q, r.prefix_table, r.prefix_off, r.suffix_table, r.suffix_off], region + 4096)
        dout, _, (r.out, r.lse) = pack([r.out, r.lse])
        staged.append((din, in_bytes, dout, r.args()))
    hosts = []
    for j in range(n_host):
        din = staged[j % replicas][0]
        hin = torch.empty(din.numel(), dtype=torch.uint8).pin_memory()
        hin.copy_(din)
        hout = torch.empty(staged[j % replicas][2].numel(), dtype=torch.uint8).pin_memory()
        hosts.append((hin, hout))
    torch.cuda.synchronize(dev)
    in_bytes0 = staged[0][1]
    region0 = int(reps[0].plan_info.ws_plan_off + reps[0].plan_info.plan_bytes)
    bi = align(in_bytes0) + region0
    bo = staged[0][2].numel()

    lib = _lib.load()
    call = lib.specgen_fork_attn_decode_staged_inline
    calls = []
    for j in range(n_host):
        r = reps[j % replicas]
        din, in_bytes, dout, args = staged[j % replicas]
        hin, hout = hosts[j]
        calls.append((C.byref(args), C.byref(r.lens), C.c_void_p(hin.data_ptr()),
                      C.c_void_p(din.data_ptr()), C.c_size_t(in_bytes), C.c_size_t(din.numel()),
                      C.c_void_p(dout.data_ptr()), C.c_void_p(hout.data_ptr()),
                      C.c_size_t(dout.numel()), C.c_void_p(sp)))
    done = [None, None]  # per half: an event after the last call that used it

    def step(i):
        j = i % n_host
        h = j // half
        if j % half == 0 and done[h] is not None:
            done[h].synchronize()  # every call that last used this half is done
        st = call(*calls[j])
        if st != 0:
            raise RuntimeError(_lib.status_string(st))
        if j % half == half - 1:
            ev = torch.cuda.Event()
            ev.record(stream)
            done[h] = ev

    for i in range(W):
        step(i)
    torch.cuda.synchronize(dev)
    t0 = time.perf_counter()
    for i in range(K):
        step(i)
    torch.cuda.synchronize(dev)
    dt = time.perf_counter() - t0
    for r, (din, in_bytes, _, _) in zip(reps, staged):
        st = _lib.specgen_workspace_status(din[align(in_bytes):], sp)
        if st != 0:
            raise RuntimeError(f"status {_lib.status_string(st)}")
        # the per-step plan left every replica planned and consistent
        r.plan_info = None
        r.plan(sp)
    torch.cuda.synchronize(dev)
    return {"value": w["total_forks"] * K / dt, "unit": "tokens/s", "h2d_bytes_per_step": bi,
            "d2h_bytes_per_step": bo, "steps": K,
            "api": "specgen_fork_attn_decode_staged_inline"}


def run_decode_steps():
    """--op decode_step: K serving steps of append + attention with growing suffixes.

    One plan is made for the lengths after the last step; the kernels cut the
    suffix items to the current lengths in a device array, which every step's
    append advances (writing the next lengths into a second array; the two
    swap).  Each step (copy of the step's Q and new K/V rows from pinned host
    memory, specgen_append_kv with pages from a device free list, attention,
    copy of O and LSE back to pinned memory) is captured in CUDA graphs of 16
    steps; the K timed steps replay
    them between CUDA events on the stream.  Per-kernel times: graphs of the
    attention stages alone at the final lengths, and a graph of appends into a
    second copy of the state.
    """
    import ctypes as C

    import torch

    import __graft_entry__
    from paper_2606_17518_gb300 import _lib, workloads as wl
    from paper_2606_17518_gb300.fork_attn import ForkDecode

    rank, local_rank, world = dist_env()
    __graft_entry__.build()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    per_graph = 16
    K = ARGS.steps
    W = -(-max(3, ARGS.warmup) // per_graph) * per_graph  # whole graphs of warm-up steps
    n = K + W
    w = wl.make_workload(ARGS.workload)
    layout = ARGS.kv_layout if w["v_pages"] is not None else "rows"
    kvl = _lib.KV_TILED if layout == "tiled" else _lib.KV_ROWS
    stream = torch.cuda.Stream(dev)
    sp = stream.cuda_stream
    B = w["page_size"]

    def prepare(steps):
        st = wl.make_decode_state(w, steps)
        fd = ForkDecode(st, device=dev, kv_layout=kvl)
        fd.use_device_lens = True
        lens0 = st["suffix_lens"].astype(np.int32).copy()
        fd.set_suffix_lens(lens0 + steps, update_device=False)
        fd.suffix_lens_dev.copy_(torch.from_numpy(lens0))
        with torch.cuda.stream(stream):
            fd.plan(sp)
        offs, lens, used = [], lens0.copy(), 0
        for _ in range(steps):
            offs.append(used)
            used += int(np.sum(lens % B == 0))
            lens = lens + 1
        free = torch.from_numpy(st["free_pages"]).to(dev)
        return st, fd, offs, free

    st, fd, offs, free = prepare(n)
    n_free = len(st["free_pages"])
    # a step's inputs (Q, then the new K and V rows) travel as one packed buffer
    # and its outputs (O, then LSE) as another: one copy each way per step,
    # each part at a 256-byte boundary; the library reads views of them
    align = lambda x: (x + 255) // 256 * 256
    i16 = lambda a: np.ascontiguousarray(a).view(np.int16).reshape(-1)
    parts_in = [i16(st["q"]), i16(st["k_new"][0])] + \
        ([] if st["v_new"] is None else [i16(st["v_new"][0])])
    off_in, nb_in = [], 0
    for a in parts_in:
        off_in.append(nb_in)
        nb_in = align(nb_in + a.size * 2)
    h_in = torch.zeros((n, nb_in // 2), dtype=torch.int16).pin_memory()
    for s_ in range(n):
        h_in[s_, 0:parts_in[0].size] = torch.from_numpy(parts_in[0])
        h_in[s_, off_in[1] // 2:off_in[1] // 2 + parts_in[1].size] = torch.from_numpy(i16(st["k_new"][s_]))
        if st["v_new"] is not None:
            h_in[s_, off_in[2] // 2:off_in[2] // 2 + parts_in[2].size] = \
                torch.from_numpy(i16(st["v_new"][s_]))
    d_in = torch.empty(nb_in // 2, dtype=torch.int16, device=dev)
    view_in = lambda k, shape: d_in[off_in[k] // 2:off_in[k] // 2 + int(np.prod(shape))].view(
        torch.bfloat16).view(shape)
    fd.q = view_in(0, tuple(st["q"].shape))
    d_k = view_in(1, tuple(st["k_new"].shape[1:]))
    d_v = None if st["v_new"] is None else view_in(2, tuple(st["v_new"].shape[1:]))
    o_bytes = fd.out.numel() * 2
    nb_out = align(o_bytes) + fd.lse.numel() * 4
    d_out = torch.empty(nb_out, dtype=torch.uint8, device=dev)
    fd.out = d_out[:o_bytes].view(torch.bfloat16).view(fd.out.shape)
    fd.lse = d_out[align(o_bytes):].view(torch.float32).view(fd.lse.shape)
    h_out = torch.empty(nb_out, dtype=torch.uint8).pin_memory()
    with torch.cuda.stream(stream):
        fd.run(sp)  # first launches configure the kernels outside any capture
    torch.cuda.synchronize(dev)

    def step(s):
        d_in.copy_(h_in[s], non_blocking=True)
        # the append writes the advanced device lengths (into the other of two
        # arrays), which this step's attention and the next append read
        fd.append_kv(d_k, d_v, free[offs[s]:], n_free - offs[s], sp, advance=True)
        fd.run(sp)
        h_out.copy_(d_out, non_blocking=True)

    graphs = []
    for g0 in range(0, n, per_graph):
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            for s in range(g0, min(n, g0 + per_graph)):
                step(s)
        graphs.append((g0, graph))
    warm = [g for g in graphs if g[0] < W]
    timed = [g for g in graphs if g[0] >= W]
    for _, g in warm:
        g.replay()
    torch.cuda.synchronize(dev)
    ev = lambda: torch.cuda.Event(enable_timing=True)
    start, end = ev(), ev()
    clocks = ClockSampler(local_rank)
    clocks.start()
    with torch.cuda.stream(stream):
        start.record(stream)
        for _, g in timed:
            g.replay()
        end.record(stream)
    torch.cuda.synchronize(dev)
    clk = clocks.stop()
    status = fd.status(sp)
    if status != 0:
        raise RuntimeError(f"workspace status {_lib.status_string(status)}")
    total_ms = start.elapsed_time(end)
    if world > 1:
        import torch.distributed as dist
        t = torch.tensor([total_ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        total_ms = float(t.item())
    F = w["total_forks"]
    ms_per_step = total_ms / K

    def graph_ms(fn, reps=16):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(reps):
                fn(i)
        g.replay()
        torch.cuda.synchronize(dev)
        a, b = ev(), ev()
        with torch.cuda.stream(stream):
            a.record(stream)
            g.replay()
            b.record(stream)
        torch.cuda.synchronize(dev)
        return a.elapsed_time(b) / reps

    # attention stages alone at the final lengths
    args, plan = fd.args(), fd.plan_info
    n_part_kernels = sum(int(x > 0) for x in (plan.n_tc_ctas, plan.n_sfx_ctas,
                                               plan.n_split_items))
    lib = _lib.load()
    part_ms = graph_ms(lambda i: lib.specgen_fork_attn_run_partials(C.byref(args), C.byref(plan),
                                                                     C.c_void_p(sp)))
    merge_ms = graph_ms(lambda i: lib.specgen_fork_attn_run_merge(C.byref(args), C.byref(plan),
                                                                   C.c_void_p(sp)))
    # appends alone, into a second copy of the state (16 steps of room, replayed once more)
    st_a, fd_a, offs_a, free_a = prepare(2 * per_graph)
    kn = torch.from_numpy(st_a["k_new"].view(np.int16)).to(dev).view(torch.bfloat16)
    vn = (None if st_a["v_new"] is None else
          torch.from_numpy(st_a["v_new"].view(np.int16)).to(dev).view(torch.bfloat16))
    nf_a = len(st_a["free_pages"])
    app_ms = graph_ms(lambda i: fd_a.append_kv(kn[i], None if vn is None else vn[i],
                                               free_a[offs_a[i]:], nf_a - offs_a[i], sp))
    w_end = dict(st, suffix_lens=st["suffix_lens"] + n)
    nbytes = wl.algorithmic_bytes(w_end)
    att_bytes = nbytes["prefix"] + nbytes["suffix"] + nbytes["q"]
    hbm, _, tf_sus, peak_src = measured_peaks()
    achieved = att_bytes / (part_ms * 1e-3) / 1e9
    attn = "mla_tc" if w["v_pages"] is None else "fork_tc"
    if attn == "mla_tc":  # dense contraction: against the sustained bf16 tensor peak
        tflops = wl.algorithmic_flops(w_end)["total"] / (part_ms * 1e-3) / 1e12
        roof = {"bound": "tensor", "kernel": attn, "achieved": tflops, "peak": tf_sus,
                "unit": "TFLOP/s", "frac": tflops / tf_sus, "traffic": None,
                "peak_source": peak_src + " (bf16, sustained)",
                "algorithmic_flops_per_launch": wl.algorithmic_flops(w_end)["total"]}
    else:
        roof = {"bound": "hbm", "kernel": attn, "achieved": achieved, "peak": hbm,
                "unit": "GB/s", "frac": achieved / hbm, "traffic": None,
                "peak_source": peak_src, "algorithmic_bytes_per_launch": att_bytes}
    kern = {"append_kv": app_ms, attn: part_ms, "lse_merge": merge_ms}
    line = {
        "metric": "fork-decode step tokens/s (append + attention, growing suffixes)",
        "value": world * F / (ms_per_step * 1e-3), "unit": "tokens/s", "n_gpus": world,
        "steps": K, "warmup": W, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": ARGS.workload, "op": "decode_step", "forks": F,
                   "suffix_growth": n, "kv_layout": layout,
                   "timing": "one plan for all steps (device suffix lengths); CUDA graphs of "
                             "16 steps incl. per-step H2D/D2H copies; per-kernel times from "
                             "graphs of each kernel alone",
                   "l2": "one resident state (KV stays resident across steps, as in serving)"},
        "gpu_launches": K * (2 + n_part_kernels),  # append, partial kernels, merge
        "kernels": {k: {"ms_per_launch": v, "share": v / sum(kern.values())}
                    for k, v in kern.items()},
        "roofline": roof,
        "clocks": {k: clk[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")},
        "e2e": {"value": world * F / (ms_per_step * 1e-3), "unit": "tokens/s",
                "h2d_bytes_per_step": int(nb_in),
                "d2h_bytes_per_step": int(nb_out),
                "note": "every timed step includes its own host copies"},
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_pack():
    """--op pack: every trace's prefix pages packed into one buffer and unpacked
    back under the same table (a round trip of the remote prefix cache's device
    side), on rotating replicas (>= 3x L2), CUDA graphs of 16 steps."""
    import ctypes as C

    import torch

    import __graft_entry__
    from paper_2606_17518_gb300 import _lib, workloads as wl

    rank, local_rank, world = dist_env()
    __graft_entry__.build()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    K, W = ARGS.steps, max(3, ARGS.warmup)
    w = wl.make_workload(ARGS.workload)
    stream = torch.cuda.Stream(dev)
    sp = stream.cuda_stream
    table = torch.from_numpy(w["prefix_table"]).to(dev)
    n = len(w["prefix_table"])
    to_dev = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int16)).to(dev)
    probe = _lib.make_pool_desc(hkv=w["hkv"], head_dim_qk=w["dqk"], head_dim_v=w["dv"],
                                page_size=w["page_size"], num_pages=w["num_pages"],
                                k_pages=0x100, v_pages=None if w["v_pages"] is None else 0x100)
    nbytes = _lib.specgen_packed_bytes(probe, n)
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 126 * 2 ** 20))
    replicas = max(1, math.ceil(3 * l2 / (2 * nbytes)))
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    reps = []
    for _ in range(replicas):
        k = to_dev(w["k_pages"])
        v = None if w["v_pages"] is None else to_dev(w["v_pages"])
        buf = torch.empty(nbytes // 2, dtype=torch.int16, device=dev)
        desc = _lib.make_pool_desc(hkv=w["hkv"], head_dim_qk=w["dqk"], head_dim_v=w["dv"],
                                   page_size=w["page_size"], num_pages=w["num_pages"],
                                   k_pages=k, v_pages=v, status=status)
        reps.append((k, v, buf, desc))
    lib = _lib.load()
    tab = C.c_void_p(table.data_ptr())
    pack = lambda r: lib.specgen_pack_pages(C.byref(reps[r][3]), tab, n,
                                            C.c_void_p(reps[r][2].data_ptr()), C.c_void_p(sp))
    unpack = lambda r: lib.specgen_unpack_pages(C.byref(reps[r][3]), tab, n,
                                                C.c_void_p(reps[r][2].data_ptr()), C.c_void_p(sp))
    per_graph = 16

    def graph_of(fns):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(per_graph):
                for fn in fns:
                    st = fn(i % replicas)
                    if st != 0:
                        raise RuntimeError(_lib.status_string(st))
        return g

    with torch.cuda.stream(stream):
        pack(0)
        unpack(0)
    torch.cuda.synchronize(dev)
    g_step, g_pack, g_unpack = graph_of([pack, unpack]), graph_of([pack]), graph_of([unpack])
    ev = lambda: torch.cuda.Event(enable_timing=True)

    def timed(g, steps):
        reps_n = max(1, -(-steps // per_graph))
        a, b = ev(), ev()
        with torch.cuda.stream(stream):
            a.record(stream)
            for _ in range(reps_n):
                g.replay()
            b.record(stream)
        torch.cuda.synchronize(dev)
        return a.elapsed_time(b) / (reps_n * per_graph)

    timed(g_step, W)
    clocks = ClockSampler(local_rank)
    clocks.start()
    ms_per_step = timed(g_step, K)
    clk = clocks.stop()
    pack_ms, unpack_ms = timed(g_pack, K), timed(g_unpack, K)
    if int(status.item()) != 0:
        raise RuntimeError("pack/unpack reported a bad page id")
    hbm, _, _, peak_src = measured_peaks()
    tokens = int(np.sum(w["prefix_lens"]))
    achieved = 2 * nbytes / (pack_ms * 1e-3) / 1e9
    line = {
        "metric": "prefix KV pack+unpack tokens/s", "value": world * tokens / (ms_per_step * 1e-3),
        "unit": "tokens/s", "n_gpus": world, "steps": per_graph * max(1, -(-K // per_graph)),
        "warmup": W, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": ARGS.workload, "op": "pack", "pages": n, "prefix_tokens": tokens,
                   "packed_bytes": nbytes,
                   "l2": f"rotating over {replicas} replicas (>= 3x L2)",
                   "timing": "CUDA graphs of 16 steps; per-kernel times from graphs of "
                             "each direction alone"},
        "gpu_launches": 2 * per_graph * max(1, -(-K // per_graph)),
        "kernels": {"pack_pages": {"ms_per_launch": pack_ms},
                    "unpack_pages": {"ms_per_launch": unpack_ms}},
        "roofline": {"bound": "hbm", "kernel": "pack_pages", "achieved": achieved, "peak": hbm,
                     "unit": "GB/s", "frac": achieved / hbm, "traffic": None,
                     "peak_source": peak_src, "algorithmic_bytes_per_launch": 2 * nbytes},
        "clocks": {k: clk[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")},
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_prefill():
    """--op prefill: every fork prefills its last --chunk suffix tokens (one query
    row per token, causal), plan made once, CUDA graphs of 16 runs on rotating
    replicas (>= 3x L2).  Value: prefilled tokens per second."""
    import ctypes as C

    import torch

    import __graft_entry__
    from paper_2606_17518_gb300 import _lib, workloads as wl
    from paper_2606_17518_gb300.fork_attn import ForkPrefill

    rank, local_rank, world = dist_env()
    __graft_entry__.build()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    K, W = ARGS.steps, max(3, ARGS.warmup)
    pf = wl.make_prefill(wl.make_workload(ARGS.workload), ARGS.chunk)
    nbytes = wl.algorithmic_bytes(pf)["total"]
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 126 * 2 ** 20))
    replicas = max(1, math.ceil(3 * l2 / nbytes))
    stream = torch.cuda.Stream(dev)
    sp = stream.cuda_stream
    reps = [ForkPrefill(pf, device=dev) for _ in range(replicas)]
    with torch.cuda.stream(stream):
        for r in reps:
            r.plan(sp)
            r.run(sp)
    torch.cuda.synchronize(dev)
    lib = _lib.load()
    args = [r.args() for r in reps]
    plans = [r.plan_info for r in reps]
    per_graph = 16

    def graph_of(call):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(per_graph):
                st = call(C.byref(args[i % replicas]), C.byref(plans[i % replicas]),
                          C.c_void_p(sp))
                if st != 0:
                    raise RuntimeError(_lib.status_string(st))
        return g

    ev = lambda: torch.cuda.Event(enable_timing=True)

    def timed(g, steps):
        n_rep = max(1, -(-steps // per_graph))
        a, b = ev(), ev()
        with torch.cuda.stream(stream):
            a.record(stream)
            for _ in range(n_rep):
                g.replay()
            b.record(stream)
        torch.cuda.synchronize(dev)
        return a.elapsed_time(b) / (n_rep * per_graph)

    g_run = graph_of(lib.specgen_fork_attn_run)
    timed(g_run, W)
    clocks = ClockSampler(local_rank)
    clocks.start()
    ms_per_step = timed(g_run, K)
    clk = clocks.stop()
    part_ms = timed(graph_of(lib.specgen_fork_attn_run_partials), K)
    merge_ms = timed(graph_of(lib.specgen_fork_attn_run_merge), K)
    if reps[0].status(sp) != 0:
        raise RuntimeError("prefill reported an error")
    rows = pf["rows"]
    # algorithmic flops: every query row against its own key count
    fo = pf["fork_offsets"]
    keys = 0
    for t in range(pf["num_traces"]):
        for f in range(fo[t], fo[t + 1]):
            c = int(pf["chunk_lens"][f])
            before = int(pf["suffix_lens"][f]) - c
            keys += c * int(pf["prefix_lens"][t]) + sum(before + j + 1 for j in range(c))
    flops = 2 * keys * pf["hq"] * (pf["dqk"] + pf["dv"])
    _, _, tf_sus, peak_src = measured_peaks()
    attn = "mla_tc" if pf["v_pages"] is None else "fork_tc"
    tflops = flops / (part_ms * 1e-3) / 1e12
    line = {
        "metric": "fork prefill tokens/s", "value": world * rows / (ms_per_step * 1e-3),
        "unit": "tokens/s", "n_gpus": world, "steps": per_graph * max(1, -(-K // per_graph)),
        "warmup": W, "ms_per_step": ms_per_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": ARGS.workload, "op": "prefill", "chunk": ARGS.chunk,
                   "query_rows": rows, "flops": flops, "unique_bytes": nbytes,
                   "l2": f"rotating over {replicas} replicas (>= 3x L2)",
                   "timing": "CUDA graphs of 16 runs; per-kernel times from graphs of each "
                             "stage alone"},
        "gpu_launches": 2 * per_graph * max(1, -(-K // per_graph)),
        "kernels": {attn: {"ms_per_launch": part_ms}, "lse_merge": {"ms_per_launch": merge_ms}},
        "roofline": {"bound": "tensor", "kernel": attn, "achieved": tflops, "peak": tf_sus,
                     "unit": "TFLOP/s", "frac": tflops / tf_sus, "traffic": None,
                     "peak_source": peak_src + " (bf16, sustained)",
                     "algorithmic_flops_per_launch": flops},
        "clocks": {k: clk[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")},
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def run_cascade():
    """--op cascade: decode over nested shared prefixes (a reasoning trace forked
    at 4096 and at 8192 tokens, 8 forks each, GQA 64/8, head dim 128): the
    shared segments are read once for every fork they serve.  The same forks
    planned as flat traces (each fork event re-reading its whole prefix) are
    timed beside it for comparison.  Plain CUDA graphs of 16 calls on rotating
    replicas (>= 3x L2)."""
    import ctypes as C

    import torch

    import __graft_entry__
    from paper_2606_17518_gb300 import _lib, workloads as wl
    from paper_2606_17518_gb300.fork_attn import ForkDecode

    rank, local_rank, world = dist_env()
    __graft_entry__.build()
    if not torch.cuda.is_available():
        raise SystemExit("bench.py needs a CUDA GPU")
    torch.cuda.set_device(local_rank)
    dev = torch.device("cuda", local_rank)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=dev)
    K, W = ARGS.steps, max(3, ARGS.warmup)
    wc = wl.make_cascade((4096, 8192), (8, 8))
    F = wc["total_forks"]
    stream = torch.cuda.Stream(dev)
    sp = stream.cuda_stream
    props = torch.cuda.get_device_properties(dev)
    l2 = int(getattr(props, "L2_cache_size", 126 * 2 ** 20))
    per_graph = 16
    lib = _lib.load()
    ev = lambda: torch.cuda.Event(enable_timing=True)

    def measure(w, unique):
        replicas = max(1, math.ceil(3 * l2 / unique))
        reps = [ForkDecode(w, device=dev) for _ in range(replicas)]
        with torch.cuda.stream(stream):
            for r in reps:
                r.plan(sp)
                r.run(sp)
        torch.cuda.synchronize(dev)
        args = [r.args() for r in reps]
        plans = [r.plan_info for r in reps]

        def graph_of(call):
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                for i in range(per_graph):
                    st = call(C.byref(args[i % replicas]), C.byref(plans[i % replicas]),
                              C.c_void_p(sp))
                    if st != 0:
                        raise RuntimeError(_lib.status_string(st))
            return g

        def timed(g, steps):
            n_rep = max(1, -(-steps // per_graph))
            a, b = ev(), ev()
            with torch.cuda.stream(stream):
                a.record(stream)
                for _ in range(n_rep):
                    g.replay()
                b.record(stream)
            torch.cuda.synchronize(dev)
            return a.elapsed_time(b) / (n_rep * per_graph)

        g = graph_of(lib.specgen_fork_attn_run)
        timed(g, W)
        clocks = ClockSampler(local_rank)
        clocks.start()
        step = timed(g, K)
        clk = clocks.stop()
        part = timed(graph_of(lib.specgen_fork_attn_run_partials), K)
        merge = timed(graph_of(lib.specgen_fork_attn_run_merge), K)
        if reps[0].status(sp) != 0:
            raise RuntimeError("cascade decode reported an error")
        return step, part, merge, clk

    page_bytes = wc["hkv"] * wc["page_size"] * (wc["dqk"] + wc["dv"]) * 2
    seg_bytes = int(np.sum(wc["prefix_lens"])) // wc["page_size"] * page_bytes
    flat_bytes = int(np.sum(wc["flat"]["prefix_lens"])) // wc["page_size"] * page_bytes
    sfx_bytes = int(np.sum(-(-wc["suffix_lens"] // wc["page_size"]))) * page_bytes
    q_bytes = wc["q"].size * 2
    alg = seg_bytes + sfx_bytes + q_bytes
    step, part, merge, clk = measure(wc, alg)
    f_step, f_part, _, _ = measure(wc["flat"], flat_bytes + sfx_bytes + q_bytes)
    hbm, _, _, peak_src = measured_peaks()
    achieved = alg / (part * 1e-3) / 1e9
    line = {
        "metric": "fork-decode attention tokens/s (nested prefixes)",
        "value": world * F / (step * 1e-3), "unit": "tokens/s", "n_gpus": world,
        "steps": per_graph * max(1, -(-K // per_graph)), "warmup": W, "ms_per_step": step,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": "cascade_p4k_p8k_f8x2", "op": "cascade",
                   "fork_points": [4096, 8192], "forks": [8, 8],
                   "algorithmic_bytes": alg, "flat_prefix_bytes": flat_bytes,
                   "flat_ms_per_step": f_step, "flat_kernel_ms": f_part,
                   "speedup_vs_flat": f_step / step,
                   "timing": "CUDA graphs of 16 calls; per-kernel times from graphs of each "
                             "stage alone"},
        "gpu_launches": 2 * per_graph * max(1, -(-K // per_graph)),
        "kernels": {"fork_tc": {"ms_per_launch": part}, "lse_merge": {"ms_per_launch": merge}},
        "roofline": {"bound": "hbm", "kernel": "fork_tc", "achieved": achieved, "peak": hbm,
                     "unit": "GB/s", "frac": achieved / hbm, "traffic": None,
                     "peak_source": peak_src, "algorithmic_bytes_per_launch": alg},
        "clocks": {k: clk[k] for k in ("sm_mhz", "sm_max_mhz", "reasons")},
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def main():
    if os.environ.get("SPECGEN_ORACLE_CHILD"):
        return
    if ARGS.impl == "reference":
        run_reference()
    elif ARGS.op == "decode_step":
        run_decode_steps()
    elif ARGS.op == "pack":
        run_pack()
    elif ARGS.op == "prefill":
        run_prefill()
    elif ARGS.op == "cascade":
        run_cascade()
    else:
        run_ours()


if __name__ == "__main__":
    main()
