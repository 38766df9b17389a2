#!/usr/bin/env python
"""Benchmark of the lineage expand -> FIFO batch -> gather-commit -> assemble
pass on GB300 (one JSON line on stdout from rank 0).

Workloads (``--workload``; synthetic, seeded inputs from workload/ stand in
for the paper's corpora):

  docpage    (default) document->page: 1,000,000 parents, pages per parent
             lognormal(2.3, 1.0) in [1, 2000] (about 16.4M children), payload
             lognormal(7.5, 0.8) bytes in [256 B, 64 KB], 5 % FAILED, results
             arriving in 256 random waves, batch size 256
  tiny       1,000 parents, lognormal(2.0, 1.0) in [1, 500], 64 B records,
             3 % FAILED, one arrival wave, batch 64
  video      video->clip->frame: 100,000 videos, Pareto(1.5) clips (at most
             1,000), 8-64 frames per clip of 512 B; frames gathered into
             clips, then the clips' results gathered into videos
  skew       10,000,000 parents, 1,000 of them with 100,000 children, 32 B
             records, one arrival wave
  streaming  4 Calls, 50,000,050 children of 1 KB, 1,000 readiness waves,
             batch --batch (32, 256 or 2048)

One step = the whole pass: ro_expand + ro_batch_ready (all children, flush)
+ every arrival wave's ro_gather_commit and ro_assemble of the parents that
wave completed (both levels for video), with the inputs and the result
arena resident in HBM.  The wave loop is replayed from a CUDA graph.

    python bench.py [--workload W] [--gpus N] [--steps K] [--warmup W] [--impl reference]

Multi-GPU (torchrun): every rank runs its own source microbatch (weak
scaling, no collective on the data path); the step time is the max over
ranks.  ``--impl reference`` times the oracle (plain single-threaded C) on
one host core, on bounded samples of the same draw.
"""
from __future__ import annotations

import argparse
import hashlib
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
WORKLOADS = ("docpage", "tiny", "video", "skew", "streaming")
L2_BYTES = 129 * 1024 * 1024


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=100)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="docpage", choices=WORKLOADS)
    ap.add_argument("--admissions", default="calls", choices=["calls", "call-streams", "one-stream"],
                    help="streaming: one ro_batch_ready_calls per wave (default), or one "
                         "ro_batch_ready per Call on streams of their own, or on the context's stream")
    ap.add_argument("--batch", type=int, default=256, help="streaming: batch size (32, 256, 2048)")
    ap.add_argument("--children", type=int, default=50_000_000, help="streaming: children in total")
    ap.add_argument("--parents", type=int, default=1_000_000,
                    help="docpage: documents; skew: parents when not 1,000,000 (else 10M)")
    ap.add_argument("--videos", type=int, default=100_000)
    ap.add_argument("--profile-all", action="store_true",
                    help="time every kernel (CUDA events) in the kernel-timing steps (default)")
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
    ap.add_argument("--ref-parents", type=int, default=None,
                    help="top-level parents in each --impl reference step (bounded CPU sample of "
                         "the same draw; default per workload)")
    ap.add_argument("--cpu-parents", type=int, default=None,
                    help="top-level parents of the cpu_baseline sample (default per workload)")
    return ap.parse_args(argv)


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


# ----------------------------------------------------------------------- clocks
class ClockSampler:
    """nvidia-smi samples (every 50 ms) while the timed region runs."""
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
                 "-lms", "50"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
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



# ------------------------------------------------------------------ workloads
# Top-level parents of the oracle's bounded samples of the drawn workload:
# cpu_baseline times whole passes over CPU_SAMPLE parents (about 10-30 s of
# one core); each --impl reference step is one pass over REF_SAMPLE parents
# (about a second).  None = the whole workload.
CPU_SAMPLE = {"tiny": None, "docpage": None, "video": None, "skew": 1_000_000, "streaming": 200_000}
REF_SAMPLE = {"tiny": None, "docpage": 100_000, "video": 10_000, "skew": 250_000, "streaming": 50_000}


def draw(args, salt: int = 0):
    """The workload this run measures (seeded; rank r draws with salt r)."""
    from workload import docpage, skew, streaming, tiny, video
    if args.workload == "tiny":
        return tiny(salt=salt)
    if args.workload == "video":
        return video(videos=args.videos, salt=salt)
    if args.workload == "skew":
        # --parents scales the config (same 1-in-10,000 share of 100k-child parents)
        P = args.parents if args.parents != 1_000_000 else 10_000_000
        return skew(parents=P, heavy=max(1, P // 10_000), salt=salt)
    if args.workload == "streaming":
        return streaming(total_children=args.children, batch_size=args.batch, salt=salt)
    return docpage(parents=args.parents, waves=args.waves, salt=salt)


def arena_total(wl) -> int:
    return int(sum(lv.arena_bytes for lv in wl.levels))


def workload_config(args, wl) -> dict:
    """The workload part of both arms' lines (the same for the same flags)."""
    lv = wl.top
    big = arena_total(wl) > L2_BYTES
    l2 = (f"inputs larger than L2 ({arena_total(wl) / 1e9:.1f} GB arena)" if big else
          "L2 flushed between timed steps (a 256 MB write outside each step's events)")
    if args.workload == "video":
        top, leaf = wl.levels
        return {"workload": f"video->clip->frame: {top.n_parents} videos, {top.n_children} clips, "
                            f"{leaf.n_children} frames of 512 B; frames gathered into clips, clips "
                            f"into videos; one arrival wave per level, batch {leaf.batch_size}",
                "parents": top.n_parents, "children": top.n_children + leaf.n_children,
                "levels": 2, "waves": 2, "batch": leaf.batch_size,
                "arena_bytes": leaf.arena_bytes, "l2": l2}
    if args.workload == "streaming":
        W = lv.ready_bounds.size - 1
        return {"workload": f"streaming: {lv.n_calls} Calls, {lv.n_parents} parents, {lv.n_children} "
                            f"children of 1 KB, 2 % FAILED, {W} readiness waves, batch {lv.batch_size}",
                "parents": lv.n_parents, "children": lv.n_children, "waves": W,
                "batch": lv.batch_size, "calls": lv.n_calls, "arena_bytes": lv.arena_bytes, "l2": l2}
    if args.workload == "skew":
        desc = (f"extreme skew: {lv.n_parents} parents ({int((lv.counts > 1).sum())} with "
                f"{int(lv.counts.max())} children), {lv.n_children} children, 32-byte results, "
                f"one arrival wave, batch {lv.batch_size}")
    elif args.workload == "tiny":
        desc = (f"tiny: {lv.n_parents} parents, {lv.n_children} children, 64-byte results, "
                f"3 % FAILED, one arrival wave, batch {lv.batch_size}")
    else:
        desc = (f"document->page: {lv.n_parents} parents, {lv.n_children} children, "
                f"{lv.n_waves} arrival waves, batch {lv.batch_size}")
    return {"workload": desc, "parents": lv.n_parents, "children": lv.n_children,
            "waves": lv.n_waves, "batch": lv.batch_size, "arena_bytes": lv.arena_bytes, "l2": l2}


def oracle_pass_fn(kind: str, wl):
    """One full pass of the oracle over workload `wl` (host arrays, its own
    host arena, built here and not timed): a callable returning (children
    processed, bytes assembled)."""
    from oracle import OracleCtx
    from workload import level_arena
    if kind == "video":
        top, leaf = wl.levels
        arena = level_arena(leaf)
        reports = leaf.reports(leaf.wave(0))

        def one():
            o = OracleCtx()
            try:
                x0 = o.expand(top.counts)["xid"]
                o.batch_ready(x0, 0, None, top.batch_size, flush=True)
                x1 = o.expand(leaf.counts, parent_xid=x0)["xid"]
                o.batch_ready(x1, 0, None, leaf.batch_size, flush=True)
                cm1 = o.gather_commit(x1, *reports, arena_bytes=leaf.arena_bytes)
                a1 = o.assemble(x1, arena, parents=None, n_parents=max(cm1["n_done"], 1))
                lvl1 = a1["out"][:a1["out_bytes"]]
                cm0 = o.gather_commit(x0, cm1["done"], a1["parent_status"], a1["out_len"],
                                      a1["out_off"][:-1], arena_bytes=a1["out_bytes"])
                a0 = o.assemble(x0, lvl1, parents=None, n_parents=max(cm0["n_done"], 1))
                return top.n_children + leaf.n_children, a1["out_bytes"] + a0["out_bytes"]
            finally:
                o.close()
        return one
    lv = wl.top
    arena = level_arena(lv)
    if kind == "streaming":
        B, n_ready = lv.batch_size, lv.ready_bounds.size - 1

        def one():
            o = OracleCtx(lv.n_calls)
            try:
                x = o.expand(lv.counts, parent_call=lv.parent_call)["xid"]
                total = 0
                for w in range(n_ready):
                    cand = lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]]
                    got = np.concatenate([
                        o.batch_ready(x, c, cand, B, flush=(w == n_ready - 1), cap=cand.size + B)["batched"]
                        for c in range(lv.n_calls)])
                    got = got[np.argsort(lv.key[got], kind="stable")]
                    cm = o.gather_commit(x, *lv.reports(got), arena_bytes=lv.arena_bytes)
                    total += o.assemble(x, arena, parents=None, n_parents=max(cm["n_done"], 1))["out_bytes"]
                return lv.n_children, total
            finally:
                o.close()
        return one
    reports = [lv.reports(lv.wave(w)) for w in range(lv.n_waves)]

    def one():
        o = OracleCtx()
        try:
            x = o.expand(lv.counts)["xid"]
            o.batch_ready(x, 0, None, lv.batch_size, flush=True)
            total = 0
            for ch, st, ln, of in reports:
                cm = o.gather_commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
                total += o.assemble(x, arena, parents=None, n_parents=max(cm["n_done"], 1))["out_bytes"]
            return lv.n_children, total
        finally:
            o.close()
    return one


def _sample(wl, parents):
    from workload import subset
    if parents is None or parents >= wl.top.n_parents:
        return wl, wl.top.n_parents
    return subset(wl, parents), parents


class _OneCore:
    """Pin this process to one host core (the oracle is single-threaded)."""

    def __enter__(self):
        self.prev = os.sched_getaffinity(0) if hasattr(os, "sched_getaffinity") else None
        self.core = min(self.prev) if self.prev else None
        if self.core is not None:
            os.sched_setaffinity(0, {self.core})
        return self

    def __exit__(self, *exc):
        if self.prev:
            os.sched_setaffinity(0, self.prev)


def cpu_baseline(args, wl, min_seconds: float = 10.0) -> dict:
    """The oracle as it stands, single-threaded on one host core, timed on a
    bounded sample of the GPU arm's own draw: whole passes (with payload
    bytes) repeated until `min_seconds` of CPU work have run."""
    k = args.cpu_parents if args.cpu_parents is not None else CPU_SAMPLE[args.workload]
    sample, kp = _sample(wl, k)
    one = oracle_pass_fn(args.workload, sample)
    passes, dt, n = 0, 0.0, 0
    with _OneCore() as pin:
        while passes == 0 or dt < min_seconds:
            t0 = time.perf_counter()
            n, _ = one()
            dt += time.perf_counter() - t0
            passes += 1
    whole = kp >= wl.top.n_parents
    what = "the whole workload" if whole else f"its first {kp} of {wl.top.n_parents} parents"
    return {"value": round(passes * n / dt, 1), "unit": "children/s", "cores": 1, "kind": "oracle",
            "pinned_core": pin.core, "host": host_cpu(),
            "sample": f"the GPU arm's draw, {what} ({n} children), full pass with payload bytes, "
                      f"{passes} passes in {dt:.1f} s"}


def run_reference(args, rank):
    """The oracle as it stands, single-threaded on one host core: W untimed
    and K timed steps, each one full pass (with payload bytes) over a bounded
    sample (the first --ref-parents top-level parents) of the same draw the
    GPU arm's rank 0 measures.  The line carries the GPU arm's config."""
    if rank != 0:
        return
    wl = draw(args, salt=0)
    cfg = workload_config(args, wl)
    k = args.ref_parents if args.ref_parents is not None else REF_SAMPLE[args.workload]
    sample, kp = _sample(wl, k)
    one = oracle_pass_fn(args.workload, sample)
    times = []
    n = S = 0
    with _OneCore() as pin:
        for _ in range(args.warmup):
            one()
        for _ in range(args.steps):
            t0 = time.perf_counter()
            n, S = one()
            times.append(time.perf_counter() - t0)
    dt = sum(times)
    v = args.steps * n / dt
    whole = kp >= wl.top.n_parents
    what = "the whole workload" if whole else f"the first {kp} of {wl.top.n_parents} parents"
    line = {
        "impl": "reference", "metric": METRIC, "value": round(v, 1), "unit": "children/s",
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(dt / args.steps * 1e3, 3),
        "ms_per_step_median": round(sorted(times)[len(times) // 2] * 1e3, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8/u32/u64",
        "data": "synthetic", "config": cfg,
        "parallelism": "single-threaded oracle, one host core (rank 0 only)",
        "cpu_baseline": {"value": round(v, 1), "unit": "children/s", "cores": 1, "kind": "oracle",
                         "pinned_core": pin.core, "host": host_cpu(),
                         "sample": f"each step one full pass with payload bytes over {what} of the "
                                   f"same draw ({n} children, {S} bytes assembled); {args.steps} "
                                   f"steps in {dt:.1f} s"},
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



class VideoPass:
    """Device-resident inputs and outputs of the video->clip->frame pass: the
    frames' reports are gathered into clips (one arrival wave), then the
    clips' assembled results (list, outcome, length, offset: the layout of a
    report array) are committed as the reports of the videos' expansion and
    gathered again from the clips' output."""

    def __init__(self, wl, device, stream):
        import torch
        from workload.device import fill_payload
        self.torch = torch
        top, leaf = wl.levels
        self.top, self.leaf, self.lv = top, leaf, leaf
        self.levels = [leaf, top]
        self.V, self.C, self.F = top.n_parents, top.n_children, leaf.n_children
        self.P, self.N = self.V + self.C, self.C + self.F   # over both levels
        self.W, self.B = 2, leaf.batch_size
        self.lists, self.parent_bound, self.keep = False, False, None
        dev = torch.device("cuda", device)
        self.stream = stream
        i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).to(dev)
        i64 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).to(dev)
        u8 = lambda a: torch.from_numpy(np.ascontiguousarray(a)).to(dev)
        z = lambda n, dt: torch.empty(max(n, 1), dtype=dt, device=dev)
        self.counts0, self.counts1 = i32(top.counts), i32(leaf.counts)
        arr = leaf.arrival
        self.child, self.state = i32(arr), u8(leaf.state[arr])
        self.length, self.off = i32(leaf.length[arr]), i64(leaf.arena_off[arr])
        self.arena_bytes = int(leaf.arena_bytes)
        self.arena = torch.empty(max(self.arena_bytes, 16), dtype=torch.uint8, device=dev)
        off_c, len_c = i64(leaf.arena_off), i32(leaf.length)
        fill_payload(self.arena, off_c, len_c, leaf.payload_seed, stream)
        torch.cuda.synchronize(dev)
        del off_c, len_c
        self.out1_cap = self.arena_bytes + 64
        self.out0_cap = self.out1_cap + 64
        self.out1 = torch.empty(self.out1_cap, dtype=torch.uint8, device=dev)
        self.out0 = torch.empty(self.out0_cap, dtype=torch.uint8, device=dev)
        self.off0, self.cp0, self.co0 = z(self.V + 1, torch.int64), z(self.C, torch.int32), z(self.C, torch.int32)
        self.off1, self.cp1, self.co1 = z(self.C + 1, torch.int64), z(self.F, torch.int32), z(self.F, torch.int32)
        self.batched0, self.batched1 = z(self.C + self.B, torch.int32), z(self.F + self.B, torch.int32)
        self.n_batched = torch.zeros(2, dtype=torch.int64, device=dev)
        self.done1 = z(self.C, torch.int32)
        self.n_done1 = torch.zeros(1, dtype=torch.int64, device=dev)
        self.status1, self.out_off1, self.out_len1 = (z(self.C, torch.uint8), z(self.C + 1, torch.int64),
                                                      z(self.C, torch.int32))
        self.status0, self.out_off0, self.out_len0 = (z(self.V, torch.uint8), z(self.V + 1, torch.int64),
                                                      z(self.V, torch.int32))
        self.cursor = torch.zeros(2, dtype=torch.int64, device=dev)
        self.out_bytes = torch.zeros(2, dtype=torch.int64, device=dev)

    def expand(self, ro, ctx):
        st, n, _, x0 = ro.ro_expand(ctx, -1, self.counts0, self.V, None, self.off0, self.cp0,
                                    self.co0, self.C, None)
        if st != 0 or n != self.C:
            raise RuntimeError(f"ro_expand (videos): {st} {ro.ro_last_error(ctx)}")
        st, n, _, x1 = ro.ro_expand(ctx, x0, self.counts1, self.C, None, self.off1, self.cp1,
                                    self.co1, self.F, None)
        if st != 0 or n != self.F:
            raise RuntimeError(f"ro_expand (clips): {st} {ro.ro_last_error(ctx)}")
        return (x0, x1)

    def waves(self, ro, ctx, xids, arena=None, out1=None, out0=None):
        """Both levels' batch_ready, commit and assemble; asynchronous.  The
        arena and the two outputs may be given as pinned host tensors."""
        L = ro.load()
        x0, x1 = xids
        arena = self.arena if arena is None else arena
        out1 = self.out1 if out1 is None else out1
        out0 = self.out0 if out0 is None else out0
        nb = self.n_batched.data_ptr()
        bad = L.ro_batch_ready(ctx, x0, 0, None, 0, self.B, 1, self.batched0.data_ptr(),
                               self.C + self.B, nb, None, None)
        bad |= L.ro_batch_ready(ctx, x1, 0, None, 0, self.B, 1, self.batched1.data_ptr(),
                                self.F + self.B, nb + 8, None, None)
        self.cursor.zero_()
        cur, obw = self.cursor.data_ptr(), self.out_bytes.data_ptr()
        # frames -> clips
        bad |= L.ro_gather_commit(ctx, x1, self.F, None, self.child.data_ptr(), self.state.data_ptr(),
                                  self.length.data_ptr(), self.off.data_ptr(), None, self.arena_bytes,
                                  None, self.done1.data_ptr(), self.C, self.n_done1.data_ptr(), None)
        bad |= L.ro_assemble(ctx, x1, arena.data_ptr(), self.arena_bytes, None, self.C, None,
                             self.status1.data_ptr(), self.out_off1.data_ptr(),
                             self.out_len1.data_ptr(), out1.data_ptr(), self.out1_cap, cur, obw, None)
        # the clips' results (written by the copy) become the videos' reports
        bad |= L.ro_ctx_join(ctx)
        bad |= L.ro_gather_commit(ctx, x0, self.C, self.n_done1.data_ptr(), self.done1.data_ptr(),
                                  self.status1.data_ptr(), self.out_len1.data_ptr(),
                                  self.out_off1.data_ptr(), None, self.out1_cap, None, None, 0, None, None)
        bad |= L.ro_assemble(ctx, x0, out1.data_ptr(), self.out1_cap, None, self.V, None,
                             self.status0.data_ptr(), self.out_off0.data_ptr(),
                             self.out_len0.data_ptr(), out0.data_ptr(), self.out0_cap, cur + 8,
                             obw + 8, None)
        bad |= L.ro_ctx_join(ctx)
        if bad:
            raise RuntimeError(f"video pass: status {bad}: {ro.ro_last_error(ctx)}")


# -------------------------------------------------------------------- roofline
# Algorithmic bytes of each kernel per pass (the boundary I/O its step must
# move; internal lineage state is not counted), from the pass's totals:
# P parents and N children summed over levels, R reports, S bytes
# assembled, M members of the assembled Present parents and Z of them that
# contribute bytes.
def kernel_alg_bytes(info: dict) -> dict:
    P, N, R, S, M, Z = (info[k] for k in ("P", "N", "R", "S", "M", "Z"))
    return {
        "expand_scan": 4 * P + 8 * (P + info["levels"]),     # counts in, offsets out
        "expand_fill": 8 * N,                                  # parent and ordinal per child
        "ready_scatter": 4 * N,                                # the batch list
        "ready_fused": 4 * N,                                  # the same, one-pass admission
        "commit_scatter": 21 * R,                              # report (17) + lineage (4)
        "commit_plan": 13 * P + 16 * M + 16 * Z,               # list + records in + plan out
        "asm_members": 16 * M + 16 * Z,                        # records in, plan out (lists)
        "asm_copy": 2 * S,                                     # payload read + write
    }


# ncu DRAM traffic (dram__bytes_read.sum + dram__bytes_write.sum) per launch
# of a kernel, from one capture of the workload named by its description (the
# line's config.workload) run with the default options, with the sha256
# (first 16 hex digits) of the kernel's source file at capture time; another
# workload or size, a non-default run option, or a source that has changed
# since makes the bench report traffic as null.
KERNEL_SOURCE = {"expand_scan": "k_expand.cu", "expand_fill": "k_expand.cu",
                 "ready_count": "k_ready.cu", "ready_scatter": "k_ready.cu", "ready_fused": "k_ready.cu",
                 "commit_scatter": "k_commit.cu", "commit_fix": "k_commit.cu",
                 "commit_plan": "k_complete.cu", "asm_members": "k_assemble.cu",
                 "asm_copy": "k_assemble.cu"}
# (workload description, kernel) -> (bytes per launch, source sha16, how it was captured)
TRAFFIC = {
    ("document->page: 1000000 parents, 16399843 children, 256 arrival waves, batch 256", "asm_copy"): (
        82359700, "17d3df01e8ba8a81",
        "ncu dram__bytes_read.sum + dram__bytes_write.sum (one pass) of all 256 asm_copy launches "
        "of one full-size 1M-document step, averaged per launch: 12.99 GB read, 8.09 GB written "
        "(the last writes of each launch leave L2 after it ends)"),
}


def source_sha16(kernel: str):
    f = KERNEL_SOURCE.get(kernel)
    if not f:
        return None
    with open(os.path.join(ROOT, "paper_2609_18703_gb300", "csrc", f), "rb") as fh:
        return hashlib.sha256(fh.read()).hexdigest()[:16]


def measured_traffic(workload_desc: str, kernel: str, default_run: bool = True):
    t = TRAFFIC.get((workload_desc, kernel))
    if not default_run or not t or t[1] != source_sha16(kernel):
        return None, None
    return t[0], t[2]


def level_totals(levels) -> dict:
    """Members of the Present parents and those contributing bytes, from the
    workload's draws (a parent is Suppressed when a member FAILED)."""
    from workload import FAILED, PRESENT
    M = Z = 0
    for lv in levels:
        if lv.state is None:
            continue
        off = np.concatenate([[0], np.cumsum(lv.counts.astype(np.int64))])
        bad = np.zeros(lv.n_parents, bool)
        nz = np.flatnonzero(lv.counts > 0)
        if nz.size:
            f = (lv.state == FAILED).astype(np.int64)
            bad[nz] = np.add.reduceat(f, off[nz]) > 0
        ok_child = np.repeat(~bad, lv.counts.astype(np.int64))
        M += int(ok_child.sum())
        Z += int((ok_child & (lv.state == PRESENT) & (lv.length > 0)).sum())
    return {"M": M, "Z": Z}


def run_ours(args, rank, world, local_rank):
    import torch
    import __graft_entry__
    import paper_2609_18703_gb300 as ro

    torch.cuda.set_device(local_rank)
    __graft_entry__.build()
    hbm_peak, peak_kind = peaks()
    wl = draw(args, salt=rank)
    cfg = workload_config(args, wl)
    stream = torch.cuda.Stream()
    torch.cuda.set_stream(stream)
    if args.workload == "video":
        ps = VideoPass(wl, local_rank, stream)
    else:
        ps = Pass(wl.top, local_rank, stream, lists=args.lists, filter_drop=args.filter_drop,
                  parent_bound=args.parent_bound)
    ctx = ro.ro_ctx_create(local_rank, stream, 1)
    if not args.one_stream:   # completion lists, plans and copies overlap later waves' commits
        plan_stream, copy_stream = torch.cuda.Stream(), torch.cuda.Stream()
        ro.ro_ctx_set_streams(ctx, plan_stream, copy_stream)
    # inputs smaller than L2: flush it between timed steps (outside their events)
    flush = None
    if arena_total(wl) <= L2_BYTES:
        flush = torch.empty(256 << 20, dtype=torch.uint8, device=torch.device("cuda", local_rank))

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
    ev0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for k in range(args.steps):
        if flush is not None:
            flush.fill_(k & 0xFF)
        ev0[k].record(stream)
        step()
        ev1[k].record(stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    step_ms = sorted(ev0[k].elapsed_time(ev1[k]) for k in range(args.steps))
    if dist:
        td.barrier()
    clk = clocks.stop()
    ms_total = t_start.elapsed_time(t_end) if flush is None else sum(step_ms)
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

    # ---- per-kernel timing (CUDA events on each kernel's launch stream) in
    # eager steps; the roofline is the dominant kernel's
    ro.ro_ctx_profile(ctx, (1 << len(ro.KERNELS)) - 1)
    kt_steps = max(2, min(args.steps, 5))
    for _ in range(kt_steps):
        step_eager()
    stream.synchronize()
    prof = ro.ro_ctx_profile_read(ctx)
    ro.ro_ctx_profile(ctx, 0)
    levels = [wl.leaf] if args.workload == "video" else [wl.top]
    tot = level_totals(levels)
    if args.workload == "video":   # the clips' reports: every clip Present, with bytes
        tot["M"] += ps.C
        tot["Z"] += ps.C
    info = {"P": ps.P, "N": ps.N, "R": ps.N, "S": S, "levels": len(wl.levels), **tot}
    alg = kernel_alg_bytes(info)
    kernel_ms = {k: round(v[2] / kt_steps, 4) for k, v in prof.items() if v[1]}
    # the roofline's kernel: the one that moves the most algorithmic bytes
    dom = max((k for k in alg if k in kernel_ms), key=lambda k: alg[k])
    n_launch = prof[dom][0] // kt_steps
    dom_ms = kernel_ms[dom]
    achieved = alg[dom] / (dom_ms * 1e-3) / 1e9 if dom_ms > 0 else 0.0
    default_run = not (ps.parent_bound or ps.lists or ps.keep is not None or args.one_stream
                       or graph is None)
    traffic, traffic_src = measured_traffic(cfg["workload"], dom, default_run)
    pass_alg = 33.0 * ps.N + 25.0 * ps.P + 2.0 * S
    n_entries = int(ps.n_elems.sum().item()) if ps.lists else 0
    if ps.lists:   # per entry: state, offset, length; per listed parent: its range start
        pass_alg += 13.0 * n_entries + 8.0 * (ps.P + ps.W)
    if ps.keep is not None:   # F.filter reads state and predicate, writes state
        pass_alg += 3.0 * ps.N
    reservation = None
    if ps.parent_bound:
        res_kernels = ("ready_count", "ready_scatter") + tuple(k for k in ro.KERNELS if k.startswith("pb_"))
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
        if args.workload == "video":
            e2e = run_e2e_video(args, ps, ro, ctx, world)
        else:
            e2e, e2e_staged = run_e2e(args, ps, ro, ctx, stream, world)

    cpu = None
    if rank == 0 and not args.no_cpu:
        cpu = cpu_baseline(args, wl)

    if rank == 0:
        payload_gbs = 2.0 * S / (ms_step * 1e-3) / 1e9
        line = {
            "metric": METRIC, "value": round(value, 1), "unit": "children/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
            "ms_per_step_median": round(step_ms[len(step_ms) // 2], 4),
            "ms_per_step_best": round(step_ms[0], 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "u8/u32/u64", "data": "synthetic", "config": cfg,
            "parallelism": f"replicas x{world} (one microbatch per GPU)",
            "run": {"reservation": "parent-bound" if ps.parent_bound else "elastic",
                    "output": "list entries per member" if ps.lists else "bytes",
                    "list_entries": n_entries if ps.lists else None,
                    "filter_drop": args.filter_drop, "cuda_graph": graph is not None,
                    "streams": 1 if args.one_stream else 3},
            "assembled_bytes": S,
            "payload_gbs": round(payload_gbs, 1),
            "payload_frac_of_hbm": round(payload_gbs / hbm_peak, 4),
            "algorithmic_gbs": round(pass_alg / (ms_step * 1e-3) / 1e9, 1),
            "algorithmic_frac_of_hbm": round(pass_alg / (ms_step * 1e-3) / 1e9 / hbm_peak, 4),
            "algorithmic_frac_of_nominal_8tbs": round(pass_alg / (ms_step * 1e-3) / 1e9 / 8000.0, 4),
            "roofline": {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1),
                         "peak": hbm_peak, "peak_kind": peak_kind, "unit": "GB/s",
                         "frac": round(achieved / hbm_peak, 4),
                         "traffic": None if traffic is None else round(traffic),
                         "traffic_source": traffic_src,
                         "algorithmic_bytes_per_launch": round(alg[dom] / max(n_launch, 1)),
                         "launches_per_step": n_launch,
                         "avg_launch_ms": round(dom_ms / max(n_launch, 1), 5)},
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


def run_e2e_video(args, ps, ro, ctx, world):
    """The video pass through the C ABI with host buffers, in place: each
    step copies both levels' counts and the frames' reports to the device;
    the frames' copy reads their payloads from the pinned host arena and
    writes the clips' results into pinned host memory, which the videos'
    copy reads in turn, writing its result into pinned host memory too."""
    import torch
    pin = lambda t: t.cpu().pin_memory()
    h = [(d, pin(d)) for d in (ps.counts0, ps.counts1, ps.child, ps.state, ps.length, ps.off)]
    try:
        h_arena = torch.empty(max(ps.arena_bytes, 16), dtype=torch.uint8).pin_memory()
        h_out1 = torch.empty(ps.out1_cap, dtype=torch.uint8).pin_memory()
        h_out0 = torch.empty(ps.out0_cap, dtype=torch.uint8).pin_memory()
    except Exception as exc:   # host memory
        return {"value": None, "unit": "children/s", "note": f"pinned host buffers unavailable: {exc}"}
    _d2h_chunks(ps.arena, h_arena)
    h2d_inputs = sum(t.numel() * t.element_size() for _, t in h)

    def step():
        for d, t in h:
            d.copy_(t, non_blocking=True)
        ro.ro_ctx_reset(ctx)
        xids = ps.expand(ro, ctx)
        ps.waves(ro, ctx, xids, arena=h_arena, out1=h_out1, out0=h_out0)
        return [int(x) for x in ps.cursor.tolist()]   # synchronises

    step()
    torch.cuda.synchronize()
    steps = max(1, min(args.steps, 3))
    t0 = time.perf_counter()
    S1 = S0 = 0
    for _ in range(steps):
        S1, S0 = step()
    torch.cuda.synchronize()
    dt = (time.perf_counter() - t0) / steps
    same = torch.equal(h_out0[:S0], ps.out0[:S0].cpu()) if S0 else True
    return {"value": round(world * ps.N / dt, 1), "unit": "children/s",
            "h2d_bytes_per_step": int(h2d_inputs + 2 * S1), "d2h_bytes_per_step": int(S1 + S0 + 16),
            "ms_per_step": round(dt * 1e3, 3),
            "how": "counts and frame reports copied to the device each step; both levels' copies "
                   "read their payloads from and write their results into pinned host memory in place",
            "matches_device_output": bool(same)}


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


def run_streaming(args, rank, world, local_rank):
    """The streaming multi-Call configuration (4 Calls, 50M children of 1 KB,
    2 % FAILED, 1,000 readiness waves): per wave, each Call admits the wave's
    ready children into its FIFO queue and reserves whole batches of B; the
    reserved children's results arrive in that wave (ordered by a per-child
    key) and are committed; the parents they complete are assembled.  The
    wave loop is captured once in a CUDA graph and replayed; every input is
    resident.  One step = the expansion plus the wave loop."""
    import torch
    import __graft_entry__
    import paper_2609_18703_gb300 as ro
    from workload.device import fill_payload

    torch.cuda.set_device(local_rank)
    __graft_entry__.build()
    hbm_peak, peak_kind = peaks()
    wl = draw(args, salt=rank)
    cfg = workload_config(args, wl)
    lv = wl.top
    B = lv.batch_size
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
    arena_bytes = int(lv.arena_bytes)
    arena = torch.empty(max(arena_bytes, 16), dtype=torch.uint8, device=dev)
    fill_payload(arena, i64(lv.arena_off), i32(lv.length), lv.payload_seed, stream)
    out_cap = arena_bytes + 64
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
    call_streams = [torch.cuda.Stream() for _ in range(lv.n_calls)] if args.admissions == "call-streams" else []
    ro.ro_ctx_set_call_streams(ctx, call_streams)
    L = ro.load()
    import ctypes
    n_calls = lv.n_calls
    c_calls = (ctypes.c_uint32 * n_calls)(*range(n_calls))
    c_batched = (ctypes.c_void_p * n_calls)(*[b.data_ptr() for b in batched])
    c_caps = (ctypes.c_uint64 * n_calls)(*([N + B] * n_calls))

    def expand():
        ro.ro_ctx_reset(ctx)
        st, n, _, xid = ro.ro_expand(ctx, -1, counts, P, calls, offsets, cp, co, N, None)
        if st != 0 or n != N:
            raise RuntimeError(f"ro_expand: {st} {ro.ro_last_error(ctx)}")
        return xid

    def waves(xid, arena_t=None, out_t=None):
        arena_p = (arena if arena_t is None else arena_t).data_ptr()
        out_p = (out if out_t is None else out_t).data_ptr()
        bad = 0
        cursor.zero_()
        for w in range(W):
            c0, c1 = int(lv.ready_bounds[w]), int(lv.ready_bounds[w + 1])
            if args.admissions == "calls":   # every Call's admission in one launch
                bad |= L.ro_batch_ready_calls(ctx, xid, n_calls, c_calls, cand.data_ptr() + 4 * c0, c1 - c0,
                                              B, int(w == W - 1), c_batched, c_caps, None)
            else:
                for c in range(n_calls):
                    bad |= L.ro_batch_ready(ctx, xid, c, cand.data_ptr() + 4 * c0, c1 - c0, B,
                                            int(w == W - 1), batched[c].data_ptr(), N + B, None, None,
                                            None)
            s, e = int(rb[w]), int(rb[w + 1])
            bad |= L.ro_gather_commit(ctx, xid, e - s, None, r_child.data_ptr() + 4 * s,
                                      r_state.data_ptr() + s, r_len.data_ptr() + 4 * s,
                                      r_off.data_ptr() + 8 * s, None, arena_bytes, None,
                                      None, 0, None, None)
            bad |= L.ro_assemble(ctx, xid, arena_p, arena_bytes, None, P, None,
                                 status.data_ptr(), out_off.data_ptr(), out_len.data_ptr(),
                                 out_p, out_cap, cursor.data_ptr(), None, None)
        bad |= L.ro_ctx_join(ctx)
        if bad:
            raise RuntimeError(f"wave loop: {bad}: {ro.ro_last_error(ctx)}")

    for _ in range(max(1, args.warmup)):
        waves(expand())
    stream.synchronize()
    if ro.ro_ctx_sync(ctx) != 0:
        raise RuntimeError(ro.ro_last_error(ctx))
    xid = expand()
    ro.ro_ctx_profile_read(ctx)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        waves(xid)
    per_replay = sum(v[0] for v in ro.ro_ctx_profile_read(ctx).values())
    for _ in range(args.warmup):
        expand()
        g.replay()
    torch.cuda.synchronize()
    ro.ro_ctx_profile_read(ctx)
    steps = max(1, args.steps)
    clocks = ClockSampler(local_rank)
    clocks.start()
    ev0 = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    ev1 = [torch.cuda.Event(enable_timing=True) for _ in range(steps)]
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for k in range(steps):
        ev0[k].record(stream)
        expand()   # synchronises (host counts)
        g.replay()
        ev1[k].record(stream)
    t_end.record(stream)
    torch.cuda.synchronize()
    clk = clocks.stop()
    launches = sum(v[0] for v in ro.ro_ctx_profile_read(ctx).values()) + steps * per_replay
    if ro.ro_ctx_sync(ctx) != 0:
        raise RuntimeError(ro.ro_last_error(ctx))
    S = int(cursor.item())
    ms = sorted(ev0[k].elapsed_time(ev1[k]) for k in range(steps))
    ms_step = t_start.elapsed_time(t_end) / steps

    # per-kernel timing in one eager pass; the dominant kernel's roofline
    ro.ro_ctx_profile(ctx, (1 << len(ro.KERNELS)) - 1)
    waves(expand())
    stream.synchronize()
    prof = ro.ro_ctx_profile_read(ctx)
    ro.ro_ctx_profile(ctx, 0)
    tot = level_totals([lv])
    alg = kernel_alg_bytes({"P": P, "N": N, "R": N, "S": S, "levels": 1, **tot})
    for k in ("ready_scatter", "ready_fused"):   # every Call reads every candidate list
        alg[k] += 4 * N * lv.n_calls
    kernel_ms = {k: round(v[2], 4) for k, v in prof.items() if v[1]}
    dom = max((k for k in alg if k in kernel_ms), key=lambda k: alg[k])
    n_launch = prof[dom][0]
    achieved = alg[dom] / (kernel_ms[dom] * 1e-3) / 1e9 if kernel_ms[dom] > 0 else 0.0
    traffic, traffic_src = measured_traffic(cfg["workload"], dom)
    pass_alg = 33.0 * N + 25.0 * P + 2.0 * S + 4.0 * N * lv.n_calls

    # end to end in place: candidates and reports copied per wave from pinned
    # host memory; the copy reads the host arena and writes host output
    e2e = None
    if not args.no_e2e:
        e2e = _streaming_e2e(args, lv, [counts, calls, cand, r_child, r_state, r_len, r_off],
                             arena, out, out_cap, cursor, expand, waves, S)
    cpu = None
    if rank == 0 and not args.no_cpu:
        cpu = cpu_baseline(args, wl)
    if rank == 0:
        payload_gbs = 2.0 * S / (ms_step * 1e-3) / 1e9
        line = {
            "metric": METRIC, "value": round(world * N / (ms_step * 1e-3), 1), "unit": "children/s",
            "n_gpus": world, "steps": steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 4),
            "ms_per_step_median": round(ms[len(ms) // 2], 4), "ms_per_step_best": round(ms[0], 4),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "u8/u32/u64",
            "data": "synthetic", "config": cfg,
            "parallelism": f"replicas x{world} (one microbatch per GPU)",
            "run": {"cuda_graph": True,
                    "admissions": {"calls": "all Calls in one launch (ro_batch_ready_calls)",
                                   "call-streams": "one ro_batch_ready per Call, each on a stream of its own",
                                   "one-stream": "one ro_batch_ready per Call, on the context's stream"}[args.admissions],
                    "kernels_per_wave": round(per_replay / W, 2)},
            "assembled_bytes": S,
            "payload_gbs": round(payload_gbs, 1),
            "payload_frac_of_hbm": round(payload_gbs / hbm_peak, 4),
            "algorithmic_gbs": round(pass_alg / (ms_step * 1e-3) / 1e9, 1),
            "algorithmic_frac_of_hbm": round(pass_alg / (ms_step * 1e-3) / 1e9 / hbm_peak, 4),
            "roofline": {"kernel": dom, "bound": "hbm", "achieved": round(achieved, 1),
                         "peak": hbm_peak, "peak_kind": peak_kind, "unit": "GB/s",
                         "frac": round(achieved / hbm_peak, 4),
                         "traffic": None if traffic is None else round(traffic),
                         "traffic_source": traffic_src,
                         "algorithmic_bytes_per_launch": round(alg[dom] / max(n_launch, 1)),
                         "launches_per_step": n_launch,
                         "avg_launch_ms": round(kernel_ms[dom] / max(n_launch, 1), 5)},
            "kernel_ms_per_step": kernel_ms,
            "gpu_launches": int(launches),
            "clocks": clk, "e2e": e2e, "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    ro.ro_ctx_destroy(ctx)


def _streaming_e2e(args, lv, inputs, arena, out, out_cap, cursor, expand, waves, S_dev):
    """The streaming pass through the C ABI with host buffers, in place: each
    step copies the counts, Calls, readiness candidates and reports to the
    device from pinned host memory; the copy kernel reads the payloads it
    needs from the pinned host arena and writes the assembled bytes into
    pinned host memory."""
    import torch
    h_inputs = [(d, d.cpu().pin_memory()) for d in inputs]
    try:
        h_arena = torch.empty(arena.numel(), dtype=torch.uint8).pin_memory()
        h_out = torch.empty(out_cap, dtype=torch.uint8).pin_memory()
    except Exception as exc:
        return {"value": None, "unit": "children/s", "note": f"pinned host buffers unavailable: {exc}"}
    _d2h_chunks(arena, h_arena)
    h2d_inputs = sum(d.numel() * d.element_size() for d in inputs)

    def step():
        for d, h in h_inputs:
            d.copy_(h, non_blocking=True)
        xid = expand()   # synchronises
        waves(xid, arena_t=h_arena, out_t=h_out)
        return int(cursor.item())

    step()
    torch.cuda.synchronize()
    steps = max(1, min(args.steps, 2))
    t0 = time.perf_counter()
    S = 0
    for _ in range(steps):
        S = step()
    torch.cuda.synchronize()
    dt = (time.perf_counter() - t0) / steps
    same = S == S_dev and torch.equal(h_out[:S], out[:S].cpu())
    return {"value": round(lv.n_children / dt, 1), "unit": "children/s",
            "h2d_bytes_per_step": int(h2d_inputs + S), "d2h_bytes_per_step": int(S + 8),
            "ms_per_step": round(dt * 1e3, 3),
            "how": "counts, Calls, candidates and reports copied to the device each step; the copy "
                   "kernel reads the needed payload bytes from the pinned host arena and writes the "
                   "assembled bytes into pinned host memory in place",
            "matches_device_output": bool(same)}


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
    # algorithmic bytes per retried Grain: list entry 4 read, its 16-byte slot
    # read (phase word, claim in len, Call), phase word and len rewritten (8),
    # recovery-queue entry 4 written
    alg = 32.0 * k
    print(json.dumps({"retry": {
        "workload": f"document->page: {N} children in flight; one failed attempt of {k} Grains "
                    f"(random order) retried per call",
        "ms_per_call": round(ms, 4), "grains_per_s": round(k / (ms * 1e-3), 1),
        "algorithmic_gbs": round(alg / (ms * 1e-3) / 1e9, 1), "peak_gbs": hbm_peak,
        "peak_kind": peak_kind, "frac": round(alg / (ms * 1e-3) / 1e9 / hbm_peak, 4),
        "steps": args.steps, "warmup": args.warmup}}), flush=True)
    ro.ro_ctx_destroy(ctx)


def main(argv=None):
    args = parse(argv)
    if args.retry:
        run_retry_bench(args, int(os.environ.get("LOCAL_RANK", "0")))
        return
    if args.rq4:
        run_rq4(args, int(os.environ.get("LOCAL_RANK", "0")))
        return
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as td
        td.init_process_group("gloo")
    if args.impl == "reference":
        run_reference(args, rank)
    elif args.workload == "streaming":
        run_streaming(args, rank, world, local_rank)
    else:
        run_ours(args, rank, world, local_rank)
    if world > 1:
        import torch.distributed as td
        td.barrier()
        td.destroy_process_group()


if __name__ == "__main__":
    main()
