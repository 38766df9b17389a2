#!/usr/bin/env python
"""Benchmark of the lineage expand -> FIFO batch -> gather-commit -> assemble
pass on GB300 (one JSON line on stdout from rank 0).

Workload (default): the document->page configuration — 1,000,000 parents,
pages per parent lognormal(2.3, 1.0) in [1, 2000] (about 16.4M children),
payload lognormal(7.5, 0.8) bytes in [256 B, 64 KB], 5 % FAILED, results
arriving in 256 random waves, batch size 256.  Synthetic, seeded inputs
(workload/) stand in for the paper's corpora.

One step = ro_expand + ro_batch_ready (all children, flush) + 256 x
(ro_gather_commit + ro_assemble of the parents that wave completed), with the
inputs and the 39 GB result arena resident in HBM.  The wave loop is replayed
from a CUDA graph (it is launch-bound: 5 kernels per wave).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl reference]

Multi-GPU (torchrun): every rank runs its own source microbatch (weak
scaling, no collective on the data path); the step time is the max over
ranks.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "children/sec expand->gather->assemble at 1 GB300; payload GB/s as % of HBM peak"
K_ACOPY = 8
# DRAM bytes (read + write) per algorithmic byte of asm_copy, from the ncu
# capture of the largest wave of a 60,000-parent document->page pass.  The
# full-size bench is too large to capture with the full section set, so the
# per-launch traffic reported here scales that ratio by the bytes a launch
# assembles.
COPY_TRAFFIC_RATIO = 0.986


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--one-call-stream", action="store_true",
                    help="streaming: every Call admits on the context's stream (no Call streams)")
    ap.add_argument("--workload", default="docpage", choices=["docpage", "skew", "streaming"],
                    help="docpage: the 1M-document config (default); skew: 10M parents, "
                         "1,000 of them with 100k children, 32-byte results, one wave; "
                         "streaming: 4 Calls, 50M children, 1,000 readiness waves")
    ap.add_argument("--batch", type=int, default=256, help="streaming: batch size (32, 256, 2048)")
    ap.add_argument("--parents", type=int, default=1_000_000)
    ap.add_argument("--profile-all", action="store_true",
                    help="time every kernel (CUDA events) in the kernel-timing steps")
    ap.add_argument("--waves", type=int, default=256)
    ap.add_argument("--no-graph", action="store_true", help="launch the wave loop eagerly")
    ap.add_argument("--retry", action="store_true", help="ro_retry throughput (failed attempts)")
    ap.add_argument("--rq4", action="store_true",
                    help="failure-containment pass (GroupFailure at ordinal 0 of the largest parents)")
    ap.add_argument("--rq4-waves", type=int, default=64)
    ap.add_argument("--rq4-parents", type=int, default=99)
    ap.add_argument("--lists", action="store_true",
                    help="assemble with ro_assemble_list (per-member list entries, Section 4.2)")
    ap.add_argument("--filter-drop", type=float, default=0.0,
                    help="F.filter each wave's reports first; fraction the predicate rejects")
    ap.add_argument("--parent-bound", action="store_true",
                    help="reserve with ro_batch_ready_parent (Section 4.3), pages admitted in arrival order")
    ap.add_argument("--one-stream", action="store_true",
                    help="plan and copy on the context's stream (no overlap across waves)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--ref-parents", type=int, default=100_000,
                    help="parents in each --impl reference step (bounded CPU sample)")
    ap.add_argument("--cpu-parents", type=int, default=1_000_000,
                    help="parents in the oracle's bounded CPU sample")
    return ap.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ----------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples (200 ms) while the timed region runs."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []
        self.t = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.t:
            self.t.join(timeout=2)
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            parts = [p.strip() for p in ln.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for name, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------------------ ranks
def max_over_ranks(x: float) -> float:
    """Largest value of x over all ranks (gloo; host tensors only)."""
    import torch
    import torch.distributed as td
    t = torch.tensor([float(x)], dtype=torch.float64)
    td.all_reduce(t, op=td.ReduceOp.MAX)
    return float(t.item())


# ------------------------------------------------------------------ CPU oracle
def cpu_oracle_sample(parents: int, waves: int, salt: int = 0, min_seconds: float = 10.0, max_passes: int = 8):
    """Time the oracle (single-threaded C) on a bounded sample of the same
    workload: the first `parents` documents of the same distribution, one
    full pass (expand, batch_ready, every wave's commit and assembly with its
    payload bytes), repeated until `min_seconds` of CPU work have run.
    Returns (children/s, seconds, children per pass, bytes per pass, passes)."""
    from oracle import OracleCtx
    from workload import docpage, level_arena
    lv = docpage(parents=parents, waves=waves, salt=salt).top
    arena = level_arena(lv)
    reports = [lv.reports(lv.wave(w)) for w in range(lv.n_waves)]
    passes, total, dt = 0, 0, 0.0
    # one core, as a single-threaded baseline; the affinity is restored after
    prev = os.sched_getaffinity(0) if hasattr(os, "sched_getaffinity") else None
    core = min(prev) if prev else None
    if core is not None:
        os.sched_setaffinity(0, {core})
    try:
        while passes < max_passes and (passes == 0 or dt < min_seconds):
            o = OracleCtx()
            t0 = time.perf_counter()
            x = o.expand(lv.counts)["xid"]
            o.batch_ready(x, 0, None, lv.batch_size, flush=True)
            total = 0
            for ch, st, ln, of in reports:
                cm = o.gather_commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
                a = o.assemble(x, arena, parents=None, n_parents=max(cm["n_done"], 1))
                total += a["out_bytes"]
            dt += time.perf_counter() - t0
            o.close()
            passes += 1
    finally:
        if prev:
            os.sched_setaffinity(0, prev)
    return passes * lv.n_children / dt, dt, lv.n_children, total, passes, core


def host_cpu() -> dict:
    """The host the CPU baseline ran on: model name and logical CPUs."""
    model = None
    try:
        for line in open("/proc/cpuinfo"):
            if line.lower().startswith(("model name", "cpu model")):
                model = line.split(":", 1)[1].strip()
                break
        if model is None:   # Arm hosts name the part elsewhere
            out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
            for line in out.splitlines():
                if line.startswith("Model name:"):
                    model = line.split(":", 1)[1].strip()
                    break
    except Exception:
        pass
    return {"model": model, "nproc": os.cpu_count()}


def run_reference(args, rank):
    """The oracle as it stands, single-threaded on one host core: W untimed
    and K timed steps, each one full pass (expand, batch_ready, every wave's
    commit and assembly with its payload bytes) over a bounded sample of the
    document->page workload (its first --ref-parents parents)."""
    if rank != 0:
        return
    from oracle import OracleCtx
    from workload import docpage, level_arena
    lv = docpage(parents=args.ref_parents, waves=args.waves, salt=0).top
    arena = level_arena(lv)
    reports = [lv.reports(lv.wave(w)) for w in range(lv.n_waves)]

    def one_pass():
        o = OracleCtx()
        x = o.expand(lv.counts)["xid"]
        o.batch_ready(x, 0, None, lv.batch_size, flush=True)
        total = 0
        for ch, st, ln, of in reports:
            cm = o.gather_commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
            total += o.assemble(x, arena, parents=None, n_parents=max(cm["n_done"], 1))["out_bytes"]
        o.close()
        return total

    prev = os.sched_getaffinity(0) if hasattr(os, "sched_getaffinity") else None
    core = min(prev) if prev else None
    if core is not None:
        os.sched_setaffinity(0, {core})
    try:
        for _ in range(args.warmup):
            one_pass()
        times = []
        for _ in range(args.steps):
            t0 = time.perf_counter()
            S = one_pass()
            times.append(time.perf_counter() - t0)
    finally:
        if prev:
            os.sched_setaffinity(0, prev)
    dt = sum(times)
    v = args.steps * lv.n_children / dt
    line = {
        "impl": "reference", "metric": METRIC, "value": round(v, 1), "unit": "children/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(dt / args.steps * 1e3, 3),
        "ms_per_step_median": round(sorted(times)[len(times) // 2] * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8/u32/u64",
        "data": "synthetic",
        "config": {"workload": f"document->page, first {args.ref_parents} of 1,000,000 parents "
                               f"({lv.n_children} children, bounded CPU sample), {args.waves} waves, "
                               f"batch {lv.batch_size}",
                   "parents": args.ref_parents, "children": lv.n_children,
                   "assembled_bytes": S, "parallelism": "single-threaded oracle, one core"},
        "cpu_baseline": {"value": round(v, 1), "unit": "children/s", "cores": 1, "kind": "oracle",
                         "pinned_core": core, "host": host_cpu(),
                         "sample": f"{args.ref_parents} parents / {lv.n_children} children per step, "
                                   f"full pass with payload bytes, {args.steps} steps in {dt:.1f} s"},
        "e2e": {"value": round(v, 1), "unit": "children/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------------ GPU
class Pass:
    """Device-resident inputs and outputs of one document->page microbatch."""

    def __init__(self, lv, device, stream, lists=False, filter_drop=0.0, parent_bound=False):
        import torch
        from workload.device import fill_payload
        self.torch = torch
        self.lv = lv
        self.P, self.N, self.W, self.B = lv.n_parents, lv.n_children, lv.n_waves, lv.batch_size
        dev = torch.device("cuda", device)
        self.stream = stream
        i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to(dev)
        i64 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).to(dev)
        u8 = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        arr = lv.arrival
        self.counts = i32(lv.counts)
        # reports, in arrival order; wave w = [bounds[w], bounds[w+1])
        self.child = i32(arr)
        self.state = u8(lv.state[arr])
        self.length = i32(lv.length[arr])
        self.off = i64(lv.arena_off[arr])
        self.bounds = lv.wave_bounds.astype(np.int64)
        self.arena_bytes = int(lv.arena_bytes)
        self.arena = torch.empty(max(self.arena_bytes, 16), dtype=torch.uint8, device=dev)
        off_c, len_c = i64(lv.arena_off), i32(lv.length)
        fill_payload(self.arena, off_c, len_c, lv.payload_seed, stream)
        torch.cuda.synchronize(dev)
        del off_c, len_c
        self.out_cap = self.arena_bytes + 64
        self.out = torch.empty(self.out_cap, dtype=torch.uint8, device=dev)
        self.offsets = torch.empty(self.P + 1, dtype=torch.int64, device=dev)
        self.cp = torch.empty(self.N, dtype=torch.int32, device=dev)
        self.co = torch.empty(self.N, dtype=torch.int32, device=dev)
        self.batched = torch.empty(self.N + self.B, dtype=torch.int32, device=dev)
        self.n_batched = torch.zeros(1, dtype=torch.int64, device=dev)
        self.status = torch.empty(self.P, dtype=torch.uint8, device=dev)
        self.out_off = torch.empty(self.P + 1, dtype=torch.int64, device=dev)
        self.out_len = torch.empty(self.P, dtype=torch.int32, device=dev)
        self.cursor = torch.zeros(1, dtype=torch.int64, device=dev)
        self.out_bytes = torch.zeros(self.W, dtype=torch.int64, device=dev)
        self.lists = lists
        self.parent_bound = parent_bound
        if parent_bound:
            self.batch_off = torch.empty(self.N + 1, dtype=torch.int64, device=dev)
            self.n_batches = torch.zeros(1, dtype=torch.int64, device=dev)
        if lists:
            # wave w's list entries and entry ranges go to windows of their own,
            # sized by the parents whose last report arrives in that wave
            wave_of = np.empty(self.N, np.int64)
            for w in range(self.W):
                wave_of[arr[self.bounds[w]:self.bounds[w + 1]]] = w
            off = np.concatenate([[0], np.cumsum(lv.counts.astype(np.int64))])
            nz = np.flatnonzero(lv.counts > 0)
            last = np.maximum.reduceat(wave_of, off[nz]) if nz.size else np.zeros(0, np.int64)
            ent = np.bincount(last, weights=lv.counts[nz].astype(np.int64), minlength=self.W)
            par = np.bincount(last, minlength=self.W)
            self.ent_cap = ent.astype(np.int64)
            self.ent_at = np.concatenate([[0], np.cumsum(self.ent_cap)])
            self.base_at = np.concatenate([[0], np.cumsum(par + 1)])
            self.elem_base = torch.empty(int(self.base_at[-1]), dtype=torch.int64, device=dev)
            self.elem_state = torch.empty(max(self.N, 1), dtype=torch.uint8, device=dev)
            self.elem_off = torch.empty(max(self.N, 1), dtype=torch.int64, device=dev)
            self.elem_len = torch.empty(max(self.N, 1), dtype=torch.int32, device=dev)
            self.n_elems = torch.zeros(self.W, dtype=torch.int64, device=dev)
        self.keep = None
        if filter_drop > 0:
            rng = np.random.default_rng([0x46494C54, int(lv.payload_seed) & 0xFFFFFFFF])
            self.keep = u8((rng.random(self.N) >= filter_drop).astype(np.uint8))

    def expand(self, ro, ctx):
        st, n, ne, xid = ro.ro_expand(ctx, -1, self.counts, self.P, None, self.offsets, self.cp,
                                      self.co, self.N, None)
        if st != 0:
            raise RuntimeError(f"ro_expand: {st} {ro.ro_last_error(ctx)}")
        assert n == self.N
        return xid

    def waves(self, ro, ctx, xid):
        """batch_ready + every wave's commit and assemble; asynchronous."""
        L = ro.load()
        if self.parent_bound:   # batches of siblings, pages admitted in arrival order
            st = L.ro_batch_ready_parent(ctx, xid, 0, self.child.data_ptr(), self.N, self.B, 1,
                                         self.batched.data_ptr(), self.N + self.B,
                                         self.batch_off.data_ptr(), self.N + 1,
                                         self.n_batched.data_ptr(), self.n_batches.data_ptr(),
                                         None, None)
        else:
            st = L.ro_batch_ready(ctx, xid, 0, None, 0, self.B, 1, self.batched.data_ptr(),
                                  self.N + self.B, self.n_batched.data_ptr(), None, None)
        bad = st
        self.cursor.zero_()
        cb, sb, lb, ob = (self.child.data_ptr(), self.state.data_ptr(), self.length.data_ptr(),
                          self.off.data_ptr())
        ar, st_p, oo, ol, out = (self.arena.data_ptr(), self.status.data_ptr(),
                                 self.out_off.data_ptr(), self.out_len.data_ptr(),
                                 self.out.data_ptr())
        cur, obw = self.cursor.data_ptr(), self.out_bytes.data_ptr()
        for w in range(self.W):
            s, e = int(self.bounds[w]), int(self.bounds[w + 1])
            if self.keep is not None:
                bad |= L.ro_filter_reports(ctx, sb + s, self.keep.data_ptr() + s, e - s)
            bad |= L.ro_gather_commit(ctx, xid, e - s, None, cb + 4 * s, sb + s, lb + 4 * s,
                                      ob + 8 * s, None, self.arena_bytes, None, None, 0, None, None)
            if self.lists:
                a0, b0 = int(self.ent_at[w]), int(self.base_at[w])
                bad |= L.ro_assemble_list(
                    ctx, xid, ar, self.arena_bytes, None, self.P, None, st_p, oo, ol, out,
                    self.out_cap, cur, obw + 8 * w, None, self.elem_base.data_ptr() + 8 * b0,
                    self.elem_state.data_ptr() + a0, self.elem_off.data_ptr() + 8 * a0,
                    self.elem_len.data_ptr() + 4 * a0, int(self.ent_cap[w]),
                    self.n_elems.data_ptr() + 8 * w, None)
                continue
            bad |= L.ro_assemble(ctx, xid, ar, self.arena_bytes, None, self.P, None, st_p, oo, ol,
                                 out, self.out_cap, cur, obw + 8 * w, None)
        bad |= L.ro_ctx_join(ctx)   # the copies of the last waves, back into the context's stream
        if bad:
            raise RuntimeError(f"wave loop: status {bad}: {ro.ro_last_error(ctx)}")


def run_ours(args, rank, world, local_rank):
    import torch
    import __graft_entry__
    import paper_2609_18703_gb300 as ro
    from workload import docpage

    torch.cuda.set_device(local_rank)
    __graft_entry__.build()
    hbm_peak, peak_kind = peaks()
    if args.workload == "skew":
        from workload import skew
        # --parents scales the config (same 1-in-10,000 share of 100k-child parents)
        P = args.parents if args.parents != 1_000_000 else 10_000_000
        lv = skew(parents=P, heavy=max(1, P // 10_000), salt=rank).top
    else:
        lv = docpage(parents=args.parents, waves=args.waves, salt=rank).top
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    ps = Pass(lv, local_rank, stream, lists=args.lists, filter_drop=args.filter_drop,
              parent_bound=args.parent_bound)
    ctx = ro.ro_ctx_create(local_rank, stream, 1)
    if not args.one_stream:   # assembly planning and copies overlap later waves' commits
        plan_stream, copy_stream = torch.cuda.Stream(), torch.cuda.Stream()
        ro.ro_ctx_set_streams(ctx, plan_stream, copy_stream)

    def step_eager():
        ro.ro_ctx_reset(ctx)
        xid = ps.expand(ro, ctx)
        ps.waves(ro, ctx, xid)

    graph = None
    per_replay = 0

    def step_graph():
        ro.ro_ctx_reset(ctx)
        ps.expand(ro, ctx)
        graph.replay()

    # warm-up (sizes every buffer), then capture the wave loop once
    for _ in range(max(1, args.warmup)):
        step_eager()
    stream.synchronize()
    if ro.ro_ctx_sync(ctx) != 0:
        raise RuntimeError(ro.ro_last_error(ctx))
    if not args.no_graph:
        ro.ro_ctx_reset(ctx)
        xid = ps.expand(ro, ctx)
        ro.ro_ctx_profile_read(ctx)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=stream):
            ps.waves(ro, ctx, xid)
        per_replay = sum(v[0] for v in ro.ro_ctx_profile_read(ctx).values())   # captured launches
        for _ in range(args.warmup):
            step_graph()
    step = step_eager if graph is None else step_graph
    stream.synchronize()
    ro.ro_ctx_profile_read(ctx)   # reset launch counters

    # ---- timed region
    dist = world > 1
    if dist:
        import torch.distributed as td
        td.barrier()
    torch.cuda.synchronize()
    clocks = ClockSampler(local_rank)
    clocks.start()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    marks = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    t_start.record(stream)
    marks[0].record(stream)
    for k in range(args.steps):
        step()
        marks[k + 1].record(stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    step_ms = sorted(marks[k].elapsed_time(marks[k + 1]) for k in range(args.steps))
    if dist:
        td.barrier()
    clk = clocks.stop()
    ms_total = t_start.elapsed_time(t_end)
    prof = ro.ro_ctx_profile_read(ctx)
    launches_timed = sum(v[0] for v in prof.values())
    if graph is not None:   # replays launch the kernels captured once
        launches_timed += args.steps * per_replay
    st = ro.ro_ctx_sync(ctx)
    if st != 0:
        raise RuntimeError(f"device reported {st}: {ro.ro_last_error(ctx)}")
    S = int(ps.out_bytes.sum().item())
    if dist:
        ms_total = max_over_ranks(ms_total)
    ms_step = ms_total / args.steps
    value = world * ps.N / (ms_step * 1e-3)

    # ---- per-kernel timing of the copy kernel (events on its launch stream)
    # and, with --parent-bound, of the reservation's kernels
    res_kernels = ("ready_count", "ready_scatter") + tuple(k for k in ro.KERNELS if k.startswith("pb_"))
    mask = 1 << K_ACOPY
    if ps.parent_bound:
        for k in res_kernels:
            mask |= 1 << ro.KERNELS.index(k)
    if args.profile_all:
        mask = (1 << len(ro.KERNELS)) - 1
    ro.ro_ctx_profile(ctx, mask)
    kt_steps = max(2, min(args.steps, 5))
    for _ in range(kt_steps):
        step_eager()
    stream.synchronize()
    prof = ro.ro_ctx_profile_read(ctx)
    ro.ro_ctx_profile(ctx, 0)
    n_copy, _, copy_ms = prof["asm_copy"][0], prof["asm_copy"][1], prof["asm_copy"][2]
    copy_bytes = 2.0 * S * kt_steps   # payload read + write, algorithmic
    achieved = copy_bytes / (copy_ms * 1e-3) / 1e9 if copy_ms > 0 else 0.0
    pass_alg = 33.0 * ps.N + 25.0 * ps.P + 2.0 * S
    n_entries = int(ps.n_elems.sum().item()) if ps.lists else 0
    if ps.lists:   # per entry: state, offset, length; per listed parent: its range start
        pass_alg += 13.0 * n_entries + 8.0 * (ps.P + ps.W)
    if ps.keep is not None:   # F.filter reads state and predicate, writes state
        pass_alg += 3.0 * ps.N
    kernel_ms = {k: round(v[2] / kt_steps, 4) for k, v in prof.items() if v[1]}
    reservation = None
    if ps.parent_bound:
        nbt = int(ps.n_batches.item())
        res_ms = sum(prof[k][2] for k in res_kernels) / kt_steps
        # admission: candidate, phase read + write, queue entry; reservation:
        # queue entry, parent, phase read + write, batched entry; boundaries
        res_bytes = 40.0 * ps.N + 8.0 * (nbt + 1)
        pass_alg += 4.0 * ps.N + 8.0 * (nbt + 1)   # candidates in arrival order, boundaries
        res_gbs = res_bytes / (res_ms * 1e-3) / 1e9 if res_ms > 0 else 0.0
        reservation = {"policy": "parent-bound", "batch": ps.B, "entries": ps.N, "batches": nbt,
                       "ms": round(res_ms, 4), "entries_per_s": round(ps.N / (res_ms * 1e-3), 1),
                       "algorithmic_bytes": res_bytes, "achieved_gbs": round(res_gbs, 1),
                       "frac_of_hbm": round(res_gbs / hbm_peak, 4),
                       "kernel_ms": {k: round(prof[k][2] / kt_steps, 4) for k in res_kernels}}

    # ---- end to end through the C ABI with host buffers
    e2e = e2e_staged = None
    if not args.no_e2e:
        e2e, e2e_staged = run_e2e(args, ps, ro, ctx, stream, world)

    cpu = None
    if rank == 0 and not args.no_cpu:
        v_cpu, dt_cpu, n_cpu, _, p_cpu, core = cpu_oracle_sample(args.cpu_parents, args.waves, salt=rank)
        cpu = {"value": round(v_cpu, 1), "unit": "children/s", "cores": 1, "kind": "oracle",
               "pinned_core": core, "host": host_cpu(),
               "sample": f"document->page, first {args.cpu_parents} parents ({n_cpu} children) "
                         f"of the same distributions, {args.waves} waves, full pass with payload "
                         f"bytes, {p_cpu} passes in {dt_cpu:.1f} s"}

    if rank == 0:
        payload_gbs = 2.0 * S / (ms_step * 1e-3) / 1e9
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": "children/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
            "ms_per_step_median": round(step_ms[len(step_ms) // 2], 4),
            "ms_per_step_best": round(step_ms[0], 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "u8/u32/u64", "data": "synthetic",
            "config": {"workload": (f"document->page: {ps.P} parents, {ps.N} children, "
                                    f"{args.waves} arrival waves, batch {ps.B}"
                                    if args.workload == "docpage" else
                                    f"extreme skew: {ps.P} parents ({int((ps.lv.counts > 1).sum())} "
                                    f"with {int(ps.lv.counts.max())} children), {ps.N} children, "
                                    f"32-byte results, one arrival wave, batch {ps.B}"),
                       "parents": ps.P, "children": ps.N, "waves": ps.W,
                       "arena_bytes": ps.arena_bytes, "assembled_bytes": S,
                       "reservation": "parent-bound" if ps.parent_bound else "elastic",
                       "output": "list entries per member" if ps.lists else "bytes",
                       "list_entries": n_entries if ps.lists else None,
                       "filter_drop": args.filter_drop,
                       "cuda_graph": graph is not None,
                       "streams": 1 if args.one_stream else 3,
                       "l2": "inputs larger than L2 (39 GB arena)",
                       "parallelism": f"replicas x{world} (one microbatch per GPU)"},
            "payload_gbs": round(payload_gbs, 1),
            "payload_frac_of_hbm": round(payload_gbs / hbm_peak, 4),
            "algorithmic_gbs": round(pass_alg / (ms_step * 1e-3) / 1e9, 1),
            "algorithmic_frac_of_hbm": round(pass_alg / (ms_step * 1e-3) / 1e9 / hbm_peak, 4),
            "algorithmic_frac_of_nominal_8tbs": round(pass_alg / (ms_step * 1e-3) / 1e9 / 8000.0, 4),
            "roofline": {"kernel": "asm_copy", "bound": "hbm", "achieved": round(achieved, 1),
                         "peak": hbm_peak, "peak_kind": peak_kind, "unit": "GB/s",
                         "frac": round(achieved / hbm_peak, 4),
                         "traffic": round(COPY_TRAFFIC_RATIO * copy_bytes / max(n_copy, 1)),
                         "traffic_source": "ncu dram__bytes_read+write of the 60k-parent capture, "
                                           "scaled by bytes assembled per launch",
                         "launches": n_copy, "avg_launch_ms": round(copy_ms / max(n_copy, 1), 5)},
            "kernel_ms_per_step": kernel_ms,
            "parent_bound_reservation": reservation,
            "gpu_launches": int(launches_timed),
            "clocks": clk,
            "e2e": e2e,
            "e2e_staged": e2e_staged,
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    ro.ro_ctx_destroy(ctx)


def run_e2e(args, ps, ro, ctx, stream, world):
    """The same pass through the C ABI with the inputs and outputs in pinned
    host memory, every transfer inside the timed region.  Two forms:

    in place  each step copies the counts and each wave's reports to the
              device; ro_assemble reads the payloads it needs from the pinned
              host arena and writes the assembled bytes into a pinned host
              buffer (no staging copies of the arena or the output).
    staged    each step also copies each wave's payload range of the arena
              to the device and the assembled bytes back at the end.
    """
    import torch
    P, N, W = ps.P, ps.N, ps.W
    pin = lambda t: t.cpu().pin_memory()
    h_counts, h_child, h_state, h_len, h_off = (pin(ps.counts), pin(ps.child), pin(ps.state),
                                               pin(ps.length), pin(ps.off))
    # the arena is laid out in arrival order: wave w's payloads are one contiguous range
    off_np = ps.lv.arena_off[ps.lv.arrival]
    len_np = ps.lv.length[ps.lv.arrival]
    wave_lo, wave_hi = [], []
    for w in range(W):
        s, e = int(ps.bounds[w]), int(ps.bounds[w + 1])
        m = len_np[s:e] > 0
        lo = int(off_np[s:e][m].min()) if m.any() else 0
        hi = int((off_np[s:e][m] + len_np[s:e][m]).max()) if m.any() else 0
        wave_lo.append(lo)
        wave_hi.append(hi)
    try:
        h_arena = torch.empty(max(ps.arena_bytes, 16), dtype=torch.uint8).pin_memory()
        h_out = torch.empty(ps.out_cap, dtype=torch.uint8).pin_memory()
    except Exception as exc:   # host memory
        return {"value": None, "unit": "children/s", "note": f"pinned host buffers unavailable: {exc}"}, None
    _d2h_chunks(ps.arena, h_arena)
    L = ro.load()
    reports_h2d = 4 * P + N * (4 + 1 + 4 + 8)

    def begin():
        ps.counts.copy_(h_counts, non_blocking=True)
        ro.ro_ctx_reset(ctx)
        xid = ps.expand(ro, ctx)
        L.ro_batch_ready(ctx, xid, 0, None, 0, ps.B, 1, ps.batched.data_ptr(), N + ps.B,
                         ps.n_batched.data_ptr(), None, None)
        ps.cursor.zero_()
        return xid

    def wave_reports(w):
        s, e = int(ps.bounds[w]), int(ps.bounds[w + 1])
        for d, h in ((ps.child, h_child), (ps.state, h_state), (ps.length, h_len), (ps.off, h_off)):
            d[s:e].copy_(h[s:e], non_blocking=True)
        return s, e

    def commit(xid, s, e):
        L.ro_gather_commit(ctx, xid, e - s, None, ps.child.data_ptr() + 4 * s,
                           ps.state.data_ptr() + s, ps.length.data_ptr() + 4 * s,
                           ps.off.data_ptr() + 8 * s, None, ps.arena_bytes, None, None, 0, None,
                           None)

    def step_in_place():
        xid = begin()
        for w in range(W):
            s, e = wave_reports(w)
            commit(xid, s, e)
            L.ro_assemble(ctx, xid, h_arena.data_ptr(), ps.arena_bytes, None, P, None,
                          ps.status.data_ptr(), ps.out_off.data_ptr(), ps.out_len.data_ptr(),
                          h_out.data_ptr(), ps.out_cap, ps.cursor.data_ptr(),
                          ps.out_bytes.data_ptr() + 8 * w, None)
        L.ro_ctx_join(ctx)
        return int(ps.cursor.item())   # synchronises

    def step_staged():
        xid = begin()
        for w in range(W):
            s, e = wave_reports(w)
            lo, hi = wave_lo[w], wave_hi[w]
            if hi > lo:
                ps.arena[lo:hi].copy_(h_arena[lo:hi], non_blocking=True)
            commit(xid, s, e)
            L.ro_assemble(ctx, xid, ps.arena.data_ptr(), ps.arena_bytes, None, P, None,
                          ps.status.data_ptr(), ps.out_off.data_ptr(), ps.out_len.data_ptr(),
                          ps.out.data_ptr(), ps.out_cap, ps.cursor.data_ptr(),
                          ps.out_bytes.data_ptr() + 8 * w, None)
        L.ro_ctx_join(ctx)
        torch.cuda.current_stream().synchronize()
        S = int(ps.cursor.item())
        h_out[:S].copy_(ps.out[:S])
        return S

    def timed(step):
        step()
        torch.cuda.synchronize()
        steps = max(1, min(args.steps, 3))
        t0 = time.perf_counter()
        S = 0
        for _ in range(steps):
            S = step()
        torch.cuda.synchronize()
        return (time.perf_counter() - t0) / steps, S

    dt_s, S = timed(step_staged)
    staged = {"value": round(world * N / dt_s, 1), "unit": "children/s",
              "h2d_bytes_per_step": int(reports_h2d + sum(h - l for l, h in zip(wave_lo, wave_hi))),
              "d2h_bytes_per_step": int(S), "ms_per_step": round(dt_s * 1e3, 3)}
    ref = h_out[:S].clone()   # the staged pass's assembled bytes
    dt, S2 = timed(step_in_place)
    same = S2 == S and torch.equal(h_out[:S2], ref)
    e2e = {"value": round(world * N / dt, 1), "unit": "children/s",
           "h2d_bytes_per_step": int(reports_h2d + S2), "d2h_bytes_per_step": int(S2 + 8),
           "ms_per_step": round(dt * 1e3, 3),
           "how": "counts and reports copied to the device per wave; the copy kernel reads the "
                  "needed payload bytes from the pinned host arena and writes the assembled bytes "
                  "into pinned host memory in place",
           "matches_staged_output": bool(same)}
    return e2e, staged


def _d2h_chunks(src, dst):
    chunk = 1 << 30
    for s in range(0, src.numel(), chunk):
        dst[s:s + chunk].copy_(src[s:s + chunk])
    return dst


def run_rq4(args, local_rank):
    """Failure containment on the GPU path (Section 4.4; the paper's RQ4 set-up,
    Section 6): the document->page level is dispatched over `--rq4-waves`
    readiness waves (each wave: admit its children, reserve batches of 256,
    commit the dispatched children's reports in FIFO order, assemble the
    parents they complete).  A poisoned pass reports GroupFailure at ordinal 0
    of the `--rq4-parents` largest parents; a clean pass does not.  Prints one
    JSON line with both pass times and the suppressed-sibling counts."""
    import torch
    import __graft_entry__
    import paper_2609_18703_gb300 as ro
    from workload import docpage
    from workload.device import fill_payload
    torch.cuda.set_device(local_rank)
    __graft_entry__.build()
    lv = docpage(parents=args.parents, waves=1).top
    dev = torch.device("cuda", local_rank)
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    P, N, W, B = lv.n_parents, lv.n_children, args.rq4_waves, 256
    rng = np.random.default_rng(0x52415934)
    ready = rng.permutation(N).astype(np.int64)                 # readiness order
    bounds = np.linspace(0, N, W + 1).astype(np.int64)
    off_p = np.concatenate([[0], np.cumsum(lv.counts.astype(np.int64))])
    big = np.argsort(-lv.counts.astype(np.int64), kind="stable")[:args.rq4_parents]
    triggers = off_p[big]
    t = lambda a, dt: torch.from_numpy(np.ascontiguousarray(a).view(dt)).to(dev)
    counts = t(lv.counts, np.int32)
    cand = t(ready.astype(np.uint32), np.int32)
    st_clean = t(lv.state, np.uint8)
    st_pois_np = lv.state.copy()
    st_pois_np[triggers] = ro.RO_GROUP_FAILURE
    st_pois = t(st_pois_np, np.uint8)
    length = t(lv.length, np.int32)
    aoff = t(lv.arena_off, np.int64)
    arena = torch.empty(max(int(lv.arena_bytes), 16), dtype=torch.uint8, device=dev)
    fill_payload(arena, aoff, length, lv.payload_seed, stream)
    offsets = torch.empty(P + 1, dtype=torch.int64, device=dev)
    cp = torch.empty(N, dtype=torch.int32, device=dev)
    co = torch.empty(N, dtype=torch.int32, device=dev)
    cap = int(np.max(np.diff(bounds))) + B
    batched = torch.zeros(cap, dtype=torch.int32, device=dev)
    nb = torch.zeros(1, dtype=torch.int64, device=dev)
    status = torch.empty(P, dtype=torch.uint8, device=dev)
    out_off = torch.empty(P + 1, dtype=torch.int64, device=dev)
    out = torch.empty(int(lv.arena_bytes) + 64, dtype=torch.uint8, device=dev)
    cursor = torch.zeros(1, dtype=torch.int64, device=dev)
    ctx = ro.ro_ctx_create(local_rank, stream, 1)
    L = ro.load()

    def one_pass(states):
        ro.ro_ctx_reset(ctx)
        st, n, _, x = ro.ro_expand(ctx, -1, counts, P, None, offsets, cp, co, N, None)
        assert st == 0 and n == N
        cursor.zero_()
        for w in range(W):
            s0, s1 = int(bounds[w]), int(bounds[w + 1])
            L.ro_batch_ready(ctx, x, 0, cand.data_ptr() + 4 * s0, s1 - s0, B, 1,
                             batched.data_ptr(), cap, nb.data_ptr(), None, None)
            idx = batched.long()
            # the dispatched children's reports (the executor's side of the protocol)
            r_st, r_len, r_off = states[idx], length[idx], aoff[idx]
            L.ro_gather_commit(ctx, x, cap, nb.data_ptr(), batched.data_ptr(), r_st.data_ptr(),
                               r_len.data_ptr(), r_off.data_ptr(), None, int(lv.arena_bytes),
                               None, None, 0, None, None)
            L.ro_assemble(ctx, x, arena.data_ptr(), int(lv.arena_bytes), None, P, None,
                          status.data_ptr(), out_off.data_ptr(), None, out.data_ptr(), out.numel(),
                          cursor.data_ptr(), None, None)
        L.ro_ctx_join(ctx)

    res = {}
    for name, states in (("clean", st_clean), ("poisoned", st_pois)):
        one_pass(states)                       # warm-up
        ro.ro_ctx_stats(ctx)                   # clears nothing; read below as deltas
        before = ro.ro_ctx_stats(ctx)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        e0.record(stream)
        one_pass(states)
        e1.record(stream)
        torch.cuda.synchronize()
        after = ro.ro_ctx_stats(ctx)
        assert after.pop("status") == 0, ro.ro_last_error(ctx)
        before.pop("status")
        d = {k: after[k] - before[k] for k in after}
        res[name] = {"ms_per_pass": round(e0.elapsed_time(e1), 3),
                     "children_per_s": round(N / (e0.elapsed_time(e1) * 1e-3), 1),
                     "accepted": d["accepted"], "rej_barrier": d["rej_barrier"],
                     "siblings_not_dispatched": d["barrier_not_dispatched"],
                     "siblings_suppressed_in_flight": d["barrier_in_flight"],
                     "queue_dropped": d["queue_dropped"], "bytes_assembled": int(cursor.item())}
    siblings = int(lv.counts[big].astype(np.int64).sum()) - len(big)
    print(json.dumps({"rq4": {
        "workload": f"document->page: {P} parents, {N} children, dispatched over {W} readiness "
                    f"waves, batches of {B}; GroupFailure at ordinal 0 of the {len(big)} largest parents",
        "poisoned_parents": int(len(big)), "poisoned_parent_siblings": siblings,
        "share_of_children_in_poisoned_parents": round(int(lv.counts[big].sum()) / N, 4),
        **res}}), flush=True)
    ro.ro_ctx_destroy(ctx)


def streaming_plan(lv, B):
    """Host-side schedule of the streaming pass: per readiness wave, the
    candidates, and the children each Call's FIFO queue reserves in that wave
    (whole batches of B, everything on the last wave), ordered by the
    per-child key.  Only the workload's own draws are used: each Call's queue
    is its children in readiness order, and wave w reserves the whole batches
    its queue holds after admitting wave w's children."""
    W = lv.ready_bounds.size - 1
    call_of = lv.parent_call[np.repeat(np.arange(lv.n_parents), lv.counts.astype(np.int64))]
    per_call = [lv.readiness[call_of[lv.readiness] == c] for c in range(lv.n_calls)]
    wave_of = np.empty(lv.n_children, np.int64)
    for w in range(W):
        wave_of[lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]]] = w
    # children of Call c admitted by the end of wave w (its queue is in readiness order)
    ends = [np.searchsorted(wave_of[q], np.arange(W), side="right") for q in per_call]
    reports = []
    taken = [0] * lv.n_calls
    for w in range(W):
        got = []
        for c in range(lv.n_calls):
            q, admitted = per_call[c], int(ends[c][w])
            upto = admitted if w == W - 1 else (admitted // B) * B
            got.append(q[taken[c]:upto])
            taken[c] = upto
        g = np.concatenate(got)
        reports.append(g[np.argsort(lv.key[g], kind="stable")].astype(np.uint32))
    return reports


def run_streaming(args, local_rank):
    """The streaming multi-Call configuration (4 Calls, 50M children of 1 KB,
    2 % FAILED, 1,000 readiness waves): per wave, each Call admits the wave's
    ready children into its FIFO queue and reserves whole batches of B; the
    reserved children's results arrive in that wave (ordered by a per-child
    key) and are committed; the parents they complete are assembled.  The
    wave loop is captured once in a CUDA graph and replayed; every input is
    resident.  One JSON line: children/s over the whole pass."""
    import torch
    import __graft_entry__
    import paper_2609_18703_gb300 as ro
    from workload import streaming
    from workload.device import fill_payload

    torch.cuda.set_device(local_rank)
    __graft_entry__.build()
    hbm_peak, peak_kind = peaks()
    B = args.batch
    lv = streaming(batch_size=B).top
    N, P, W = lv.n_children, lv.n_parents, lv.ready_bounds.size - 1
    reports = streaming_plan(lv, B)
    assert sum(r.size for r in reports) == N
    dev = torch.device("cuda", local_rank)
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to(dev)
    i64 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).to(dev)
    u8 = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
    counts = i32(lv.counts)
    calls = u8(lv.parent_call)
    cand = i32(lv.readiness)
    rep_all = np.concatenate(reports)
    rb = np.concatenate([[0], np.cumsum([r.size for r in reports])]).astype(np.int64)
    r_child, r_state = i32(rep_all), u8(lv.state[rep_all])
    r_len, r_off = i32(lv.length[rep_all]), i64(lv.arena_off[rep_all])
    arena = torch.empty(max(int(lv.arena_bytes), 16), dtype=torch.uint8, device=dev)
    fill_payload(arena, i64(lv.arena_off), i32(lv.length), lv.payload_seed, stream)
    out_cap = int(lv.arena_bytes) + 64
    out = torch.empty(out_cap, dtype=torch.uint8, device=dev)
    offsets = torch.empty(P + 1, dtype=torch.int64, device=dev)
    cp = torch.empty(N, dtype=torch.int32, device=dev)
    co = torch.empty(N, dtype=torch.int32, device=dev)
    # each Call admits on a stream of its own, into a batch list of its own
    batched = [torch.empty(N + B, dtype=torch.int32, device=dev) for _ in range(lv.n_calls)]
    status = torch.empty(P, dtype=torch.uint8, device=dev)
    out_off = torch.empty(P + 1, dtype=torch.int64, device=dev)
    out_len = torch.empty(P, dtype=torch.int32, device=dev)
    cursor = torch.zeros(1, dtype=torch.int64, device=dev)
    torch.cuda.synchronize()
    ctx = ro.ro_ctx_create(local_rank, stream, lv.n_calls)
    ro.ro_ctx_set_streams(ctx, torch.cuda.Stream(), torch.cuda.Stream())
    call_streams = [torch.cuda.Stream() for _ in range(lv.n_calls)] if not args.one_call_stream else []
    ro.ro_ctx_set_call_streams(ctx, call_streams)
    L = ro.load()

    def expand():
        ro.ro_ctx_reset(ctx)
        st, n, _, xid = ro.ro_expand(ctx, -1, counts, P, calls, offsets, cp, co, N, None)
        if st != 0 or n != N:
            raise RuntimeError(f"ro_expand: {st} {ro.ro_last_error(ctx)}")
        return xid

    def waves(xid):
        bad = 0
        cursor.zero_()
        for w in range(W):
            c0, c1 = int(lv.ready_bounds[w]), int(lv.ready_bounds[w + 1])
            for c in range(lv.n_calls):
                bad |= L.ro_batch_ready(ctx, xid, c, cand.data_ptr() + 4 * c0, c1 - c0, B,
                                        int(w == W - 1), batched[c].data_ptr(), N + B, None, None,
                                        None)
            s, e = int(rb[w]), int(rb[w + 1])
            bad |= L.ro_gather_commit(ctx, xid, e - s, None, r_child.data_ptr() + 4 * s,
                                      r_state.data_ptr() + s, r_len.data_ptr() + 4 * s,
                                      r_off.data_ptr() + 8 * s, None, int(lv.arena_bytes), None,
                                      None, 0, None, None)
            bad |= L.ro_assemble(ctx, xid, arena.data_ptr(), int(lv.arena_bytes), None, P, None,
                                 status.data_ptr(), out_off.data_ptr(), out_len.data_ptr(),
                                 out.data_ptr(), out_cap, cursor.data_ptr(), None, None)
        bad |= L.ro_ctx_join(ctx)
        if bad:
            raise RuntimeError(f"wave loop: {bad}: {ro.ro_last_error(ctx)}")

    for _ in range(max(1, args.warmup)):
        waves(expand())
    stream.synchronize()
    if ro.ro_ctx_sync(ctx) != 0:
        raise RuntimeError(ro.ro_last_error(ctx))
    stats = ro.ro_ctx_stats(ctx)
    xid = expand()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        waves(xid)
    for _ in range(args.warmup):
        expand()
        g.replay()
    torch.cuda.synchronize()
    steps = max(1, args.steps)
    clocks = ClockSampler(local_rank)
    clocks.start()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(steps + 1)]
    ms = []
    for k in range(steps):
        expand()   # synchronises (host counts); timed per pass below, expansion included
        ev[k].record(stream)
        g.replay()
        ev[k + 1].record(stream)
        torch.cuda.synchronize()
        ms.append(ev[k].elapsed_time(ev[k + 1]))
    clk = clocks.stop()
    if ro.ro_ctx_sync(ctx) != 0:
        raise RuntimeError(ro.ro_last_error(ctx))
    S = int(cursor.item())
    ms.sort()
    med = ms[len(ms) // 2]
    line = {
        "metric": "children/s, streaming multi-Call pass (admission, batching, commit, assembly)",
        "value": round(N / (med * 1e-3), 1), "unit": "children/s", "n_gpus": 1, "steps": steps,
        "warmup": args.warmup, "ms_per_step_median": round(med, 3), "ms_per_step_best": round(ms[0], 3),
        "higher_is_better": True, "dtype": "u8/u32/u64", "data": "synthetic",
        "config": {"workload": f"streaming: {lv.n_calls} Calls, {P} parents, {N} children of 1 KB, "
                               f"2 % FAILED, {W} readiness waves, batch {B}",
                   "assembled_bytes": S, "kernels_per_wave": 4 * 2 + 3 + 2,
                   "admissions": "on the context's stream" if args.one_call_stream
                                 else "one stream per Call",
                   "timed": "the captured wave loop (expansion outside)"},
        "payload_gbs": round(2.0 * S / (med * 1e-3) / 1e9, 1),
        "payload_frac_of_hbm": round(2.0 * S / (med * 1e-3) / 1e9 / hbm_peak, 4),
        "accepted_per_pass": stats["accepted"] // max(1, args.warmup),
        "clocks": clk,
    }
    print(json.dumps(line), flush=True)
    ro.ro_ctx_destroy(ctx)


def run_retry_bench(args, local_rank):
    """Throughput of ro_retry (Section 4.4, Eq. 2's retry edge): every child of
    the document->page level is dispatched, then a seeded random 1/16 of them
    (one failed attempt of ~1M Grains, in random order) is retried; between
    repetitions the recovery group is reserved again (READY -> IN-FLIGHT).
    Only the ro_retry calls are timed (CUDA events on the context's stream)."""
    import torch
    import __graft_entry__
    import paper_2609_18703_gb300 as ro
    from workload import docpage
    torch.cuda.set_device(local_rank)
    __graft_entry__.build()
    hbm_peak, peak_kind = peaks()
    lv = docpage(parents=args.parents, waves=1).top
    dev = torch.device("cuda", local_rank)
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    P, N = lv.n_parents, lv.n_children
    rng = np.random.default_rng(0x52415935)
    pick = rng.permutation(N)[: N // 16].astype(np.uint32)
    counts = torch.from_numpy(lv.counts.view(np.int32)).to(dev)
    lst = torch.from_numpy(pick.view(np.int32)).to(dev)
    offsets = torch.empty(P + 1, dtype=torch.int64, device=dev)
    cp = torch.empty(N, dtype=torch.int32, device=dev)
    co = torch.empty(N, dtype=torch.int32, device=dev)
    batched = torch.empty(N + 256, dtype=torch.int32, device=dev)
    ctx = ro.ro_ctx_create(local_rank, stream, 1)
    st, n, _, x = ro.ro_expand(ctx, -1, counts, P, None, offsets, cp, co, N, None)
    assert st == 0
    st, nb, _ = ro.ro_batch_ready(ctx, x, 0, None, 0, 256, 1, batched, N + 256)
    assert st == 0 and nb == N
    L = ro.load()
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    for i in range(args.warmup + args.steps):
        if i >= args.warmup:
            ev[i - args.warmup][0].record(stream)
        L.ro_retry(ctx, x, 0, lst.data_ptr(), lst.numel(), None)
        if i >= args.warmup:
            ev[i - args.warmup][1].record(stream)
        L.ro_batch_ready(ctx, x, 0, None, 0, 256, 1, batched.data_ptr(), N + 256, None, None, None)
    torch.cuda.synchronize()
    stats = ro.ro_ctx_stats(ctx)
    assert stats.pop("status") == 0, ro.ro_last_error(ctx)
    assert stats["retried"] == (args.warmup + args.steps) * lst.numel()
    ms = sum(a.elapsed_time(b) for a, b in ev) / args.steps
    k = lst.numel()
    # algorithmic bytes per retried Grain: list entry 4 read, phase word read
    # and rewritten (8), record word read for the Call (8) and len claimed and
    # cleared (12), recovery-queue entry 4 written
    alg = 36.0 * k
    print(json.dumps({"retry": {
        "workload": f"document->page: {N} children in flight; one failed attempt of {k} Grains "
                    f"(random order) retried per call",
        "ms_per_call": round(ms, 4), "grains_per_s": round(k / (ms * 1e-3), 1),
        "algorithmic_gbs": round(alg / (ms * 1e-3) / 1e9, 1), "peak_gbs": hbm_peak,
        "peak_kind": peak_kind, "frac": round(alg / (ms * 1e-3) / 1e9 / hbm_peak, 4),
        "steps": args.steps, "warmup": args.warmup}}), flush=True)
    ro.ro_ctx_destroy(ctx)


def main():
    args = parse()
    if args.retry:
        run_retry_bench(args, int(os.environ.get("LOCAL_RANK", "0")))
        return
    if args.rq4:
        run_rq4(args, int(os.environ.get("LOCAL_RANK", "0")))
        return
    if args.workload == "streaming" and args.impl != "reference":
        run_streaming(args, int(os.environ.get("LOCAL_RANK", "0")))
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as td
        td.init_process_group("gloo")
    if args.impl == "reference":
        run_reference(args, rank)
    else:
        run_ours(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as td
        td.barrier()
        td.destroy_process_group()


if __name__ == "__main__":
    main()
