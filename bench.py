#!/usr/bin/env python3
"""Benchmark of the permutation-group Allreduce on GB300.

One JSON line on stdout (rank 0).  A "step" is one Allreduce of the headline workload:
P = 24 virtual ranks x 64 MiB fp32 (16,777,216 elements per rank), bandwidth-optimal
schedule (S = 10), fused mode, inputs resident in HBM (3 GiB per step moved, far above
the 129 MB L2, so no flush is needed).  `value` = algorithmic bytes (every input read
once, every output written once: 2 * P * n * 4 bytes) / time, in GB/s, summed over
replicas when run on N GPUs (each GPU runs its own P virtual ranks: replicas only).

Also reported, on the same line:
  e2e           the same metric through gar_allreduce_host (pinned host buffers, the
                host<->device copies inside the timed region);
  roofline      the fused kernel's achieved GB/s vs the measured HBM copy bandwidth;
  cpu_baseline  the CPU oracle timed on a bounded sample of the workload;
  rows          the other hot-path rows: step-faithful mode, the P=127 bf16 step
                sweep, the P=8 sweep, the batched 425-byte Allreduces (reductions/s).

--impl reference times the CPU oracle (the method's plain simulation) on the same
metric instead.
"""

from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

HEADLINE = "p24_64mib_f32"
CLOCK_WINDOW_S = 1.0
METRIC = "Allreduce GB/s and % of HBM roofline at 1 GB300 vs P and steps; small-msg reductions/s"


def _dist_env():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            pk = json.load(f)
        return float(pk["hbm_gbs"]), "measured"
    except Exception:
        return 6800.0, "fallback"


def _cpu_info():
    cores = os.cpu_count() or 1
    model = ""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name"):
                model = line.split(":", 1)[1].strip()
                break
    except Exception:
        pass
    return cores, model


# ---------------------------------------------------------------------------
# Clock sampling during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join(ROOT, "_build", f"clocks_{os.getpid()}.csv")

    def __enter__(self):
        os.makedirs(os.path.dirname(self.path), exist_ok=True)
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.fh, stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()
            self.fh.close()

    def summary(self):
        if self.proc is None or not os.path.exists(self.path):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx = float(parts[2])
                except ValueError:
                    continue
                for nm, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(nm)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": mx,
                "reasons": sorted(reasons), "samples": len(sm)}


# ---------------------------------------------------------------------------
# Timing helpers
# ---------------------------------------------------------------------------

def _graph_us(gar, plan, ptrs, mode, calls=20, reps=5):
    """Microseconds per call of `calls` Allreduce calls captured in one CUDA graph and
    replayed (the way to issue many small Allreduces: no per-call host work); median of
    `reps` replays, after one warm-up replay."""
    import statistics
    import torch
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.stream(side):
        with torch.cuda.graph(graph, stream=side):
            for _ in range(calls):
                gar.gar_allreduce(plan, ptrs, mode, side)
    torch.cuda.current_stream().wait_stream(side)
    graph.replay()
    torch.cuda.synchronize()
    ts = []
    for _ in range(reps):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record()
        graph.replay()
        b.record()
        torch.cuda.synchronize()
        ts.append(a.elapsed_time(b) * 1e3 / calls)
    return statistics.median(ts)


def max_over_ranks(ms: float, dist, device) -> float:
    """The slowest rank's time (ms); identity without a process group."""
    if dist is None:
        return ms
    import torch
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_gbs(bytes_per_replica: int, world: int, ms: float) -> float:
    """Whole-job throughput: every replica's bytes over the slowest replica's time."""
    return bytes_per_replica * world / (ms * 1e-3) / 1e9


def _time_loop(fn, steps, warmup, stream, flush=None):
    """Runs fn() warmup times, then times `steps` calls with CUDA events on `stream`
    (synchronised on both sides).  With `flush`, L2 is flushed before every call and
    only the call itself is timed (per-call events).  Returns ms per call."""
    import torch
    for _ in range(warmup):
        if flush is not None:
            flush()
        fn()
    torch.cuda.synchronize()
    if flush is None:
        start = torch.cuda.Event(enable_timing=True)
        end = torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for _ in range(steps):
            fn()
        end.record(stream)
        torch.cuda.synchronize()
        return start.elapsed_time(end) / steps
    tot = 0.0
    for _ in range(steps):
        flush()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record(stream)
        fn()
        e.record(stream)
        torch.cuda.synchronize()
        tot += s.elapsed_time(e)
    return tot / steps


class L2Flusher:
    """Evicts L2 (129 MB on GB300) by reading a 512 MiB buffer into a scalar.  A read
    leaves only clean lines in L2, so nothing is written back inside the timed call that
    follows; the dirty lines of the previous call are written back during the flush."""

    def __init__(self, nbytes=512 << 20):
        import torch
        # float32 reduces in place of its own type: no widening copy (which would write)
        self.buf = torch.zeros(nbytes // 4, dtype=torch.float32, device="cuda")

    def __call__(self):
        self.buf.sum()


# ---------------------------------------------------------------------------
# Workloads
# ---------------------------------------------------------------------------

def _alg_bytes(P, n, dtype):
    return 2 * P * n * {"f32": 4, "bf16": 2, "i32": 4}[dtype]


def _step_dram_bytes(gar, plan, P, n, dtype):
    """DRAM bytes one step-faithful Allreduce moves under the kernels' access pattern:
    per block op and rank, the partner read, the own reads and the writes."""
    ops, _partners = gar.gar_plan_step_ops(plan)
    es = {"f32": 4, "bf16": 2, "i32": 4}[dtype]
    acc = 4
    q, rem = divmod(n, P)
    sizes = [q + (1 if b < rem else 0) for b in range(P)]
    tot = 0
    for (_l, recv_place, dst, recv_buf, o0b, o0o, o1b, o1o) in ops:
        for x in range(P):
            b = (x - dst) % P
            sz = sizes[b]
            if recv_place >= 0:
                tot += sz * (es if recv_buf == 1 else acc)
            for (ob, oo) in ((o0b, o0o), (o1b, o1o)):
                if ob:
                    tot += sz * (es if ob == 1 else acc)
                    if oo:
                        tot += sz * (es if oo == 1 else acc)
    return tot


def _l(P):
    L = 0
    while (1 << L) < P:
        L += 1
    return L


def run_ours(args):
    import torch
    import gar_inputs
    from paper_2004_09362_gb300 import build as gbuild
    gbuild.build()
    from paper_2004_09362_gb300 import gar

    ws, rank, local = _dist_env()
    torch.cuda.set_device(local)
    dist = None
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    stream = torch.cuda.current_stream()
    hbm_peak, peak_kind = _peaks()
    headline = (args.workload == HEADLINE and args.S in (None, 10) and args.mode == "fused"
                and args.op == "sum")

    if args.workload == "batched_425B":
        cfgb = gar_inputs.BATCHED
        flat, layout = gar_inputs.batched_inputs(cfgb["count"], cfgb["Ps"], cfgb["n"], "f32",
                                                 cfgb["dist"], cfgb["seed"] + rank, device="cuda")
        out_t = torch.empty_like(flat)
        plans = [gar.gar_plan_create(Pb, cfgb["n"], "f32", args.op, gar.GAR_STEPS_LO)
                 for Pb in cfgb["Ps"]]
        idx = {Pb: k for k, Pb in enumerate(cfgb["Ps"])}
        desc = gar.make_batch_desc([idx[Pb] for (Pb, _o) in layout],
                                   [flat.data_ptr() + o * 4 for (_Pb, o) in layout],
                                   [out_t.data_ptr() + o * 4 for (_Pb, o) in layout])
        bytes_step = 2 * flat.numel() * 4
        launches_per_step = 1
        kernel_desc = f"batched {cfgb['count']} x P in {cfgb['Ps']} x {cfgb['n']} f32 {args.op}"
        config = {"workload": "batched_425B", "count": cfgb["count"], "Ps": list(cfgb["Ps"]),
                  "n_per_rank": cfgb["n"], "schedule": "latency-optimal", "op": args.op,
                  "mode": "batched", "parallelism": f"replicas x{ws}",
                  "l2": "361 MB moved per step > 129 MB L2"}
        dtype = "f32"

        def step():
            gar.gar_allreduce_batched(plans, desc, cfgb["count"], stream)
        plan = None
    else:
        wl = gar_inputs.WORKLOADS[args.workload]
        P, n = wl.P, wl.n
        S = args.S if args.S is not None else 2 * _l(P)
        dtype = wl.dtype
        inp = gar_inputs.rank_inputs(P, n, wl.dtype, wl.dist, wl.seed + rank, device="cuda")
        plan = gar.gar_plan_create(P, n, wl.dtype, args.op, S)
        if args.mode in ("step", "persistent"):
            gar.ensure_workspace(plan)
        gar.gar_plan_prepare(plan, args.mode)
        ptrs = gar.rank_pointers(inp)
        info = plan.info()
        launches_per_step = 1 if args.mode in ("fused", "persistent") else info["n_launches"]
        if args.mode == "fused":
            bytes_step = _alg_bytes(P, n, wl.dtype)
        else:
            bytes_step = _step_dram_bytes(gar, plan, P, n, wl.dtype)
        kernel_desc = (f"{args.mode} P{P} S{S} {wl.dtype} {args.op}"
                       + (f" W{info['fused_width']} regs{info['fused_regs']}" if args.mode == "fused" else ""))
        sched = ("bandwidth-optimal" if S == 2 * _l(P) else "latency-optimal" if S == _l(P)
                 else "fold" if S > 2 * _l(P) else "intermediate")
        config = {"workload": args.workload, "P": P, "n_per_rank": n,
                  "bytes_per_rank": n * (2 if wl.dtype == "bf16" else 4), "steps_S": S,
                  "schedule": sched, "mode": args.mode, "op": args.op,
                  "parallelism": f"replicas x{ws}",
                  "l2": f"{2 * P * n * (2 if wl.dtype == 'bf16' else 4) / 2**30:.2f} GiB moved per step > 129 MB L2"}

        def step():
            gar.gar_allreduce(plan, ptrs, args.mode, stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        # untimed load window of the same step, so the clock samples (every 100 ms)
        # see the GPU under this load; the timed region follows without a pause
        t_end = time.time() + args.clock_window
        while time.time() < t_end:
            for _ in range(8):
                step()
            torch.cuda.synchronize()
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()
        start = torch.cuda.Event(enable_timing=True)
        end = torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for _ in range(args.steps):
            step()
        end.record(stream)
        torch.cuda.synchronize()
    if dist is not None:
        dist.barrier()
    ms = max_over_ranks(start.elapsed_time(end) / args.steps, dist, "cuda")
    if args.workload == "batched_425B" or args.mode == "fused":
        value = job_gbs(bytes_step, ws, ms)
    else:
        value = job_gbs(_alg_bytes(P, n, dtype), ws, ms)
    clocks = clk.summary()
    clocks["window"] = (f"{args.clock_window:.1f} s of untimed steps right before the timed "
                        f"{args.steps}, sampled every 100 ms through both")
    kernel_gbs = bytes_step / (ms * 1e-3) / 1e9

    out = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": dtype,
        "data": "synthetic (seeded, generated on the GPU; see gar_inputs.py)",
        "config": config,
        "gpu_launches": args.steps * launches_per_step,
        "roofline": {"bound": "hbm", "achieved": round(kernel_gbs, 1), "peak": hbm_peak,
                     "unit": "GB/s", "frac": round(kernel_gbs / hbm_peak, 4),
                     "traffic": _committed_traffic(gar) if headline else None,
                     "peak_kind": peak_kind, "kernel": kernel_desc,
                     "algorithmic_bytes_per_launch": bytes_step // launches_per_step
                     if launches_per_step == 1 else None,
                     "algorithmic_bytes_per_step": bytes_step},
        "clocks": clocks,
    }
    if args.workload != "batched_425B":
        es = 2 if dtype == "bf16" else 4
        out["algbw"] = {"value": round(n * es / (ms * 1e-3) / 1e9, 2), "unit": "GB/s",
                        "definition": "per-rank algorithm bandwidth, NCCL convention: "
                                      "bytes per rank (n * element size) / time"}
    if args.workload == "batched_425B":
        out["reductions_per_s"] = round(gar_inputs.BATCHED["count"] * ws / (ms * 1e-3), 1)

    # ---- end to end through the host-buffer entry point
    if not args.no_e2e and plan is not None:
        out["e2e"] = _e2e(gar, plan, inp, P, n, dtype, args, stream, dist)

    if rank == 0 and not args.no_rows:
        out["rows"] = measure_rows(gar, gar_inputs, stream, hbm_peak)
    if rank == 0 and not args.no_cpu:
        out["cpu_baseline"] = cpu_baseline_sample(target_s=args.cpu_seconds)
        out["cpu_baseline_mt"] = cpu_column_baseline()
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()
    if rank == 0:
        print(json.dumps(out), flush=True)


def headline_kernel_sha(gar) -> str:
    """sha1 (12 hex digits) of the generated source of the headline fused kernel."""
    import hashlib
    plan = gar.gar_plan_create(24, 16777216, "f32", "sum", 10)
    return hashlib.sha1(gar.gar_plan_fused_source(plan).encode()).hexdigest()[:12]


def _committed_traffic(gar):
    """DRAM bytes per launch of the headline fused kernel from the committed ncu summary
    (profiles/fused_p24_64mib_f32.txt), or None when absent or when the generated kernel
    differs from the one the counters were taken on."""
    path = os.path.join(ROOT, "profiles", "fused_p24_64mib_f32.txt")
    try:
        fields = {}
        with open(path) as f:
            for line in f:
                if ":" in line and not line.startswith(" "):
                    k, v = line.split(":", 1)
                    fields[k.strip()] = v.strip()
        if fields.get("kernel_source_sha1") != headline_kernel_sha(gar):
            return None
        return int(fields["dram_bytes_per_launch"].split()[0])
    except Exception:
        return None


def _link_ceiling(host_in, host_out, dev_dst, dev_src, reps=3):
    """GB/s of the host link with both directions busy: host_in -> dev_dst and dev_src ->
    host_out (pinned, one copy each) on two streams at once; best of `reps`."""
    import torch
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    nbytes = host_in.numel() * host_in.element_size() + dev_src.numel() * dev_src.element_size()
    best = None
    for _ in range(reps):
        torch.cuda.synchronize()
        start, mid, end = (torch.cuda.Event(enable_timing=True) for _ in range(3))
        start.record(s1)
        s2.wait_event(start)
        with torch.cuda.stream(s1):
            dev_dst.copy_(host_in, non_blocking=True)
        with torch.cuda.stream(s2):
            host_out.copy_(dev_src, non_blocking=True)
        mid.record(s2)
        s1.wait_event(mid)
        end.record(s1)
        torch.cuda.synchronize()
        ms = start.elapsed_time(end)
        best = ms if best is None else min(best, ms)
    return nbytes / (best * 1e-3) / 1e9


def _e2e(gar, plan, inp, P, n, dtype, args, stream, dist):
    import torch
    host_in = inp.cpu().pin_memory()
    host_out = torch.empty_like(host_in).pin_memory()
    dev = torch.empty_like(inp)
    hin = [host_in[x] for x in range(P)]
    hout = [host_out[x] for x in range(P)]
    hp_in = gar.rank_pointers(hin)
    hp_out = gar.rank_pointers(hout)
    dp = gar.rank_pointers(dev)

    def step():
        gar.gar_allreduce_host(plan, hp_in, hp_out, dp, args.mode, stream)

    steps = max(1, min(args.steps, 10))
    ms = max_over_ranks(_time_loop(step, steps, 3, stream), dist, "cuda")
    ws = dist.get_world_size() if dist is not None else 1
    bytes_step = _alg_bytes(P, n, dtype)
    value = job_gbs(bytes_step, ws, ms)
    link = _link_ceiling(host_in, host_out, dev, inp)
    return {"value": round(value, 2), "unit": "GB/s",
            "ms_per_step": round(ms, 4), "h2d_bytes_per_step": bytes_step // 2,
            "d2h_bytes_per_step": bytes_step // 2, "steps": steps,
            "link_ceiling_gbs": round(link, 1), "frac_of_link": round(value / ws / link, 4),
            "link_ceiling": ("the same bytes moved by one cudaMemcpyAsync host-to-device and one "
                             "device-to-host, pinned memory, on two streams at once (best of 3, same run)"),
            "path": ("gar_allreduce_host on pinned host buffers: the fused kernel reads the P inputs "
                     "from and writes the P results to host memory over NVLink-C2C (no staging copies)")
            if args.mode == "fused" else
            ("gar_allreduce_host: P cudaMemcpyAsync to device buffers, the step-faithful "
             "launches, P cudaMemcpyAsync back, on one stream")}


def measure_rows(gar, gar_inputs, stream, hbm_peak):
    import torch
    rows = {}
    flusher = L2Flusher()

    # step-faithful mode on the headline workload
    wl = gar_inputs.WORKLOADS[HEADLINE]
    P, n = wl.P, wl.n
    inp = gar_inputs.rank_inputs(P, n, wl.dtype, wl.dist, wl.seed, device="cuda")
    plan = gar.gar_plan_create(P, n, "f32", "sum", 10)
    gar.ensure_workspace(plan)
    gar.gar_plan_prepare(plan, "step")
    ms = _time_loop(lambda: gar.gar_allreduce(plan, inp, "step", stream), 5, 3, stream)
    dram = _step_dram_bytes(gar, plan, P, n, "f32")
    rec = gar.gar_last_step_bytes(plan)
    _ws, pred, _S = gar.gar_plan_bytes(plan)
    rows["step_faithful_p24_64mib_f32_S10"] = {
        "ms": round(ms, 4), "GB/s_algorithmic": round(_alg_bytes(P, n, "f32") / ms / 1e6, 1),
        "dram_model_bytes": dram, "GB/s_dram_model": round(dram / ms / 1e6, 1),
        "frac_dram_model": round(dram / ms / 1e6 / hbm_peak, 4),
        "launches": plan.info()["n_launches"],
        "recorded_step_bytes_equal_predicted": rec == pred,
        "msg_bytes_total": sum(rec)}
    del inp

    # P=127 bf16, every step count, both modes (fused kernel timed alone per call)
    wl = gar_inputs.WORKLOADS["p127_8mib_bf16"]
    P, n = wl.P, wl.n
    inp = gar_inputs.rank_inputs(P, n, wl.dtype, wl.dist, wl.seed, device="cuda")
    sweep = {}
    for S in wl.steps:
        plan = gar.gar_plan_create(P, n, "bf16", "sum", S)
        gar.gar_plan_prepare(plan, "fused")
        # median of 5 loops of 10 launches (single short loops varied by up to 5 %)
        ms_f = statistics.median(
            _time_loop(lambda: gar.gar_allreduce(plan, inp, "fused", stream), 10, 3 if k == 0 else 1,
                       stream) for k in range(5))
        ent = {"fused_ms": round(ms_f, 4),
               "fused_GB/s": round(_alg_bytes(P, n, "bf16") / ms_f / 1e6, 1),
               "fused_frac": round(_alg_bytes(P, n, "bf16") / ms_f / 1e6 / hbm_peak, 4),
               "fused_combines_per_position": plan.info()["fused_combines"],
               "fused_width": plan.info()["fused_width"],
               "fused_regs": plan.info()["fused_regs"],
               "fused_form": {0: "single", 1: "breadth_first", 2: "two_lane"}[plan.info()["fused_form"]]}
        if S in (7, 10, 14):
            gar.ensure_workspace(plan)
            ms_s = _time_loop(lambda: gar.gar_allreduce(plan, inp, "step", stream), 2, 1, stream)
            ent["step_ms"] = round(ms_s, 3)
            ent["step_launches"] = plan.info()["n_launches"]
            dram = _step_dram_bytes(gar, plan, P, n, "bf16")
            ent["step_dram_model_bytes"] = dram
            ent["step_frac_dram_model"] = round(dram / ms_s / 1e6 / hbm_peak, 4)
            plan.workspace = None
            gar.gar_plan_set_workspace(plan, 0, 0)
        sweep[f"S{S}"] = ent
        torch.cuda.empty_cache()
    rows["p127_8mib_bf16"] = sweep
    del inp

    # P=8, 1 MiB per rank: L2-resident, so flush L2 (read-only sweep) before each eagerly
    # timed call; the graph replays time back-to-back calls with the data in L2
    wl = gar_inputs.WORKLOADS["p8_1mib_f32"]
    P, n = wl.P, wl.n
    inp = gar_inputs.rank_inputs(P, n, wl.dtype, wl.dist, wl.seed, device="cuda")
    sweep = {}
    for S in wl.steps:
        plan = gar.gar_plan_create(P, n, "f32", "sum", S)
        gar.ensure_workspace(plan)
        gar.gar_plan_prepare(plan, "fused")
        gar.gar_plan_prepare(plan, "step")
        ms_f = _time_loop(lambda: gar.gar_allreduce(plan, inp, "fused", stream), 20, 3, stream, flusher)
        ms_s = _time_loop(lambda: gar.gar_allreduce(plan, inp, "step", stream), 20, 3, stream, flusher)
        ptrs = gar.rank_pointer_array(inp)
        sweep[f"S{S}"] = {"fused_us": round(ms_f * 1e3, 2), "step_us": round(ms_s * 1e3, 2),
                          "fused_graph_us": round(_graph_us(gar, plan, ptrs, "fused"), 2),
                          "step_graph_us": round(_graph_us(gar, plan, ptrs, "step"), 2),
                          "fused_GB/s": round(_alg_bytes(P, n, "f32") / ms_f / 1e6, 1),
                          "msg_bytes_per_rank": sum(gar.gar_plan_bytes(plan)[1]) // P}
    rows["p8_1mib_f32_l2flushed"] = sweep

    # P=5, 1024 fp32: latency
    P, n = 5, 1024
    inp = gar_inputs.rank_inputs(P, n, "f32", ("uniform", -1.0, 1.0), 1234, device="cuda")
    lat = {}
    for S in (3, 4, 5, 6):
        plan = gar.gar_plan_create(P, n, "f32", "sum", S)
        gar.ensure_workspace(plan)
        gar.gar_plan_prepare(plan, "fused")
        gar.gar_plan_prepare(plan, "step")
        ms_f = _time_loop(lambda: gar.gar_allreduce(plan, inp, "fused", stream), 50, 5, stream)
        ms_s = _time_loop(lambda: gar.gar_allreduce(plan, inp, "step", stream), 50, 5, stream)
        ptrs = gar.rank_pointer_array(inp)
        lat[f"S{S}"] = {"fused_us": round(ms_f * 1e3, 2), "step_us": round(ms_s * 1e3, 2),
                        "fused_graph_us": round(_graph_us(gar, plan, ptrs, "fused"), 2),
                        "step_graph_us": round(_graph_us(gar, plan, ptrs, "step"), 2)}
    rows["p5_1k_f32_latency"] = lat

    # batched 425-byte Allreduces
    cfg = gar_inputs.BATCHED
    flat, layout = gar_inputs.batched_inputs(cfg["count"], cfg["Ps"], cfg["n"], "f32", cfg["dist"],
                                             cfg["seed"], device="cuda")
    out = torch.empty_like(flat)
    es = 4
    for op in cfg["ops"]:
        plans = [gar.gar_plan_create(P, cfg["n"], "f32", op, gar.GAR_STEPS_LO) for P in cfg["Ps"]]
        idx = {P: k for k, P in enumerate(cfg["Ps"])}
        desc = gar.make_batch_desc([idx[P] for (P, _o) in layout],
                                   [flat.data_ptr() + o * es for (_P, o) in layout],
                                   [out.data_ptr() + o * es for (_P, o) in layout])
        # 361 MB per call > 129 MB L2: back-to-back calls need no flush
        ms = _time_loop(lambda: gar.gar_allreduce_batched(plans, desc, cfg["count"], stream), 50, 5,
                        stream)
        nbytes = 2 * flat.numel() * es
        rows[f"batched_65536x425B_{op}"] = {
            "us": round(ms * 1e3, 2), "reductions_per_s": round(cfg["count"] / (ms * 1e-3), 1),
            "GB/s": round(nbytes / ms / 1e6, 1), "frac": round(nbytes / ms / 1e6 / hbm_peak, 4)}
    del flat, out
    torch.cuda.empty_cache()
    rows["groups_p64_4mib_f32"] = groups_row(gar, gar_inputs, stream, hbm_peak)
    rows["step_range_p24_64mib_f32"] = step_range_row(gar, gar_inputs, stream, hbm_peak)
    rows["cost_model_p127_bf16_step"] = cost_model_row(gar, gar_inputs, stream, hbm_peak)
    return rows


def step_range_row(gar, gar_inputs, stream, hbm_peak):
    """The whole step range on the headline workload, both modes: bandwidth-optimal
    (2L steps), fold schedules from 2L + 2 to 2(P-1) steps (the fold of 2(P-1) steps
    moves one vector per step), and the Ring (2(P-1) steps, every step by t)."""
    import torch
    wl = gar_inputs.WORKLOADS[HEADLINE]
    P, n = wl.P, wl.n
    inp = gar_inputs.rank_inputs(P, n, "f32", wl.dist, wl.seed, device="cuda")
    L = _l(P)
    scheds = [("bandwidth_optimal", gar.GAR_STEPS_BO)]
    scheds += [(f"fold_S{S}", S) for S in (2 * L + 2, 16, 22, 30, 2 * (P - 1))]
    scheds += [("ring", gar.GAR_STEPS_RING)]
    out = {}
    for name, steps in scheds:
        plan = gar.gar_plan_create(P, n, "f32", "sum", steps)
        gar.gar_plan_prepare(plan, "step")
        gar.gar_plan_prepare(plan, "fused")
        ms_s = _time_loop(lambda: gar.gar_allreduce(plan, inp, "step", stream), 5, 2, stream)
        ms_f = _time_loop(lambda: gar.gar_allreduce(plan, inp, "fused", stream), 10, 2, stream)
        dram = _step_dram_bytes(gar, plan, P, n, "f32")
        out[name] = {"S": plan.info()["S"], "step_ms": round(ms_s, 4),
                     "step_frac_dram_model": round(dram / ms_s / 1e6 / hbm_peak, 4),
                     "fused_ms": round(ms_f, 4),
                     "msg_bytes_per_rank": sum(gar.gar_plan_bytes(plan)[1]) // P}
    del inp
    torch.cuda.empty_cache()
    return out


def groups_row(gar, gar_inputs, stream, hbm_peak, P=64, n=1 << 20):
    """Cyclic group (Table 1a) against the XOR group (Table 1b: Recursive Halving at
    S = 2L, Recursive Doubling at S = L, their hybrid in between) for P = 64 x 4 MiB
    fp32: per-rank message volume and step-faithful / fused times."""
    import torch
    inp = gar_inputs.rank_inputs(P, n, "f32", ("normal", 0.0, 1.0), 11, device="cuda")
    L = _l(P)
    out = {}
    for group in ("cyclic", "xor"):
        for S in (L, L + 2, 2 * L - 1, 2 * L):
            plan = gar.gar_plan_create_group(P, n, "f32", "sum", S, group)
            gar.ensure_workspace(plan)
            gar.gar_plan_prepare(plan, "step")
            gar.gar_plan_prepare(plan, "fused")
            ms_s = _time_loop(lambda: gar.gar_allreduce(plan, inp, "step", stream), 5, 2, stream)
            ms_f = _time_loop(lambda: gar.gar_allreduce(plan, inp, "fused", stream), 10, 2, stream)
            out[f"{group}_S{S}"] = {"msg_bytes_per_rank": sum(gar.gar_plan_bytes(plan)[1]) // P,
                                    "step_ms": round(ms_s, 4), "fused_ms": round(ms_f, 4)}
            plan.workspace = None
            del plan
            torch.cuda.empty_cache()
    return out


def _paper_blocks(P, S):
    """Per-rank traffic and combine counts in blocks of the paper's cost model (eqs.
    bo_cost, intemediate_cost, lo_cost)."""
    L = _l(P)
    r = 2 * L - S
    if r == L:
        return P * L, P * (2 * L - 2)
    extra = 2 ** r - 1
    return 2 * (P - 1) + extra * (L - 1), (P - 1) + extra * (2 * L - 2)


def cost_model_row(gar, gar_inputs, stream, hbm_peak, P=127, dtype="bf16",
                   sizes=(425, 9 * 1024, 64 * 1024, 512 * 1024, 4 << 20, 8 << 20)):
    """Step-faithful mode as the paper's machine: measure every step count at several
    message sizes, fit the cost model's alpha (per step), beta (per byte moved) and gamma
    (per byte combined) by non-negative least squares on relative errors, and check
    whether eq. opt_number_of_steps (integer argmin, gar_optimal_steps) picks the
    measured-best S."""
    import numpy as np
    import torch
    from scipy.optimize import nnls
    es = 2 if dtype == "bf16" else 4
    L = _l(P)
    times, dram = {}, {}
    for m in sizes:
        n = max(1, m // es)
        raw = gar_inputs.rank_inputs(P, n, dtype, ("normal", 0.0, 1.0), 77, device="cuda")
        per16 = 16 // es
        inp = torch.zeros((P, (n + per16 - 1) // per16 * per16), dtype=raw.dtype, device="cuda")
        inp[:, :n] = raw          # rank rows padded to 16-byte multiples
        del raw
        for S in range(L, 2 * L + 1):
            plan = gar.gar_plan_create(P, n, dtype, "sum", S)
            gar.ensure_workspace(plan)
            gar.gar_plan_prepare(plan, "step")
            reps = 20 if m <= (64 << 10) else 5
            times[(m, S)] = _time_loop(lambda: gar.gar_allreduce(plan, inp, "step", stream), reps, 3,
                                       stream) * 1e-3
            dram[(m, S)] = _step_dram_bytes(gar, plan, P, n, dtype)
            plan.workspace = None
            del plan
            torch.cuda.empty_cache()
        del inp
    # relative least squares (each measurement weighted by 1/t), so the microsecond
    # small-message points count as much as the millisecond large-message ones
    A, y = [], []
    for (m, S), t in times.items():
        tr, co = _paper_blocks(P, S)
        u = m / P
        A.append([S / t, tr * u / t, co * u / t])
        y.append(1.0)
    coef, _res = nnls(np.array(A), np.array(y))
    fitted = tuple(float(c) for c in coef)
    # Derived model: alpha = per-step time at the smallest size (slope of t over S);
    # beta, gamma from the step kernels' DRAM traffic at the measured copy bandwidth --
    # every byte of a block sent is one partner read, every byte combined one own read
    # and one write, and all P ranks share one HBM, so a per-rank byte costs P bytes of
    # DRAM time.
    Ss = np.arange(L, 2 * L + 1, dtype=float)
    ts = np.array([times[(sizes[0], int(S))] for S in Ss])
    alpha_d = float(np.polyfit(Ss, ts, 1)[0])
    bw = hbm_peak * 1e9
    derived = (alpha_d, P / bw, 2 * P / bw)

    def evaluate(a, b, g):
        per, agree, worst = {}, 0, 1.0
        for m in sizes:
            meas = {S: times[(m, S)] for S in range(L, 2 * L + 1)}
            best_meas = min(meas, key=meas.get)
            best_model = gar.gar_optimal_steps(P, m, a, b, g)
            agree += int(best_meas == best_model)
            worst = max(worst, meas[best_model] / meas[best_meas])
            per[str(m)] = {"model_us": {f"S{S}": round(gar.gar_cost_model(P, S, m, a, b, g) * 1e6, 2)
                                        for S in meas},
                           "measured_best_S": best_meas, "model_best_S": best_model,
                           "model_choice_vs_best": round(meas[best_model] / meas[best_meas], 3)}
        return {"alpha_s": a, "beta_s_per_B": b, "gamma_s_per_B": g,
                "argmin_agreement": f"{agree}/{len(sizes)}", "worst_choice_vs_best": round(worst, 3),
                "per_size_bytes": per}

    measured = {str(m): {f"S{S}": round(times[(m, S)] * 1e6, 2) for S in range(L, 2 * L + 1)}
                for m in sizes}
    per_step_us = {str(m): {f"S{S}": round(times[(m, S)] * 1e6 / S, 2) for S in range(L, 2 * L + 1)}
                   for m in sizes}
    # Where the paper's linear per-message model breaks on this machine: a step that moves
    # d DRAM bytes should take alpha + d / HBM; the effective DRAM rate of each schedule
    # shows how far below HBM the small-message steps run (per-item latency, not bytes).
    eff = {str(m): {f"S{S}": round(dram[(m, S)] / times[(m, S)] / 1e9, 1) for S in range(L, 2 * L + 1)}
           for m in sizes}
    m_lo, m_hi = sizes[1], sizes[-1]
    violation = (
        f"beta is not constant: the step-faithful Allreduce moves its DRAM-model bytes at "
        f"{eff[str(m_hi)][f'S{2 * L}']} GB/s (S={2 * L}) and {eff[str(m_hi)][f'S{L}']} GB/s (S={L}) "
        f"at {m_hi} B per rank, but at {eff[str(m_lo)][f'S{2 * L}']} and {eff[str(m_lo)][f'S{L}']} GB/s "
        f"at {m_lo} B: below a few MB per step a launch is too small to reach HBM bandwidth, so the "
        f"cost of a byte grows as the blocks shrink, most for the many-block steps of small S")
    return {"P": P, "dtype": dtype, "mode": "step", "measured_us": measured,
            "measured_us_per_step": per_step_us, "effective_dram_GBps": eff,
            "linear_model_violation": violation,
            "fit_free": evaluate(*fitted), "fit_derived": evaluate(*derived),
            "derived_from": f"alpha: slope of time over S at {sizes[0]} B; beta = P / HBM, "
                            f"gamma = 2P / HBM with HBM = {hbm_peak} GB/s (measured copy)"}


# ---------------------------------------------------------------------------
# CPU oracle legs
# ---------------------------------------------------------------------------

def _oracle_time(P, n, S, dtype="f32", seed=1237):
    import numpy as np
    import gar_inputs
    from oracle import gar_oracle
    t = gar_inputs.rank_inputs(P, n, dtype, ("normal", 0.0, 1e-3), seed)
    xs = [t[x].numpy().copy() for x in range(P)]
    t0 = time.perf_counter()
    gar_oracle.allreduce(xs, S, "sum", dtype)
    return time.perf_counter() - t0


def cpu_baseline_sample(target_s=10.0):
    """The oracle as it stands (single-threaded numpy) on the headline workload's shape
    (P = 24, S = 10, fp32 sum) with at most the headline's elements per rank, repeated
    until about target_s seconds of CPU work.  Reported in the headline's unit
    (algorithmic GB/s per Allreduce)."""
    P, S = 24, 10
    n_max = 16777216
    n = 24 * 4096
    dt = _oracle_time(P, n, S)
    while dt < target_s / 10 and n * 2 <= n_max:
        n *= 2
        dt = _oracle_time(P, n, S)
    reps, total = 1, dt
    while total < target_s:
        total += _oracle_time(P, n, S)
        reps += 1
    sec = total / reps
    cores, model = _cpu_info()
    gbs = _alg_bytes(P, n, "f32") / sec / 1e9
    return {"value": round(gbs, 4), "unit": "GB/s", "cores": 1, "host_cores": cores,
            "cpu_model": model, "kind": "oracle", "seconds": round(total, 2),
            "sample": f"P=24, S=10 (bandwidth-optimal), fp32 sum, n={n} elements per rank "
                      f"(headline has {n_max}), {reps} Allreduce(s), mean time"}


def cpu_column_baseline(target_s=3.0):
    """The plain multi-threaded CPU Allreduce (oracle/column_reduce.c: rank-order column
    reduction written to every rank, one thread per host core) on the full headline
    shape, P = 24 x 16,777,216 fp32, repeated for about target_s seconds.  A second,
    stronger CPU baseline beside the single-threaded oracle; same unit."""
    import numpy as np
    from oracle import column_reduce as CR
    P, n = 24, 16777216
    rng = np.random.default_rng(0)
    xs = [(rng.standard_normal(n) * 1e-3).astype(np.float32) for _ in range(P)]
    outs = [np.empty(n, np.float32) for _ in range(P)]
    ip, op_ = [v.ctypes.data for v in xs], [o.ctypes.data for o in outs]
    cores, model = _cpu_info()
    CR.column_allreduce_ptrs(ip, op_, n, "f32", "sum", cores)      # warm-up (first touch)
    reps, total = 0, 0.0
    while total < target_s or reps < 3:
        t0 = time.perf_counter()
        CR.column_allreduce_ptrs(ip, op_, n, "f32", "sum", cores)
        total += time.perf_counter() - t0
        reps += 1
    sec = total / reps
    return {"value": round(_alg_bytes(P, n, "f32") / sec / 1e9, 3), "unit": "GB/s",
            "cores": cores, "cpu_model": model, "kind": "plain column reduction (C, pthreads)",
            "sample": f"P=24 x n=16777216 fp32 sum (the headline shape), {reps} runs, mean time"}


def run_reference(args):
    ws, rank, _local = _dist_env()
    if rank != 0:
        return
    P, S = 24, 10
    # size one step to ~(budget / steps) seconds (default budget 150 s)
    budget = 15.0 * args.cpu_seconds
    per_step = max(0.05, min(20.0, budget / max(1, args.steps + args.warmup)))
    n = 24 * 4096
    dt = _oracle_time(P, n, S)
    while dt < per_step / 2 and n * 2 <= 16777216:
        n *= 2
        dt = _oracle_time(P, n, S)
    for _ in range(args.warmup):
        _oracle_time(P, n, S)
    times = [_oracle_time(P, n, S) for _ in range(args.steps)]
    sec = sum(times) / len(times)
    gbs = _alg_bytes(P, n, "f32") / sec / 1e9
    cores, model = _cpu_info()
    sample = (f"P=24, S=10 (bandwidth-optimal), fp32 sum, n={n} elements per rank per step "
              f"(headline has 16777216)")
    out = {"impl": "reference", "metric": METRIC, "value": round(gbs, 4), "unit": "GB/s",
           "n_gpus": ws, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": round(sec * 1e3, 2), "higher_is_better": True, "scaling": "weak",
           "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded N(0,1e-3) fp32)",
           "config": {"workload": HEADLINE, "P": P, "steps_S": S, "schedule": "bandwidth-optimal",
                      "n_per_rank_sampled": n},
           "cpu_baseline": {"value": round(gbs, 4), "unit": "GB/s", "cores": 1, "host_cores": cores,
                            "cpu_model": model, "kind": "oracle", "sample": sample},
           "e2e": {"value": round(gbs, 4), "unit": "GB/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0},
           "gpu_launches": 0}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-rows", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=10.0)
    ap.add_argument("--workload", default=HEADLINE,
                    help="gar_inputs.WORKLOADS key or batched_425B (default: the headline)")
    ap.add_argument("--S", type=int, default=None, help="step count (default: 2*ceil(log2 P))")
    ap.add_argument("--mode", default="fused", choices=["fused", "step", "persistent"])
    ap.add_argument("--op", default="sum", choices=["sum", "max", "min"])
    ap.add_argument("--clock-window", type=float, default=CLOCK_WINDOW_S,
                    help="seconds of untimed steps sampled for clocks before the timed region "
                         "(0 for profiling runs: fewer launches before the captured ones)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
