#!/usr/bin/env python
"""Benchmark of the Similarity Chunk Rolling sparse-prefill path on GB300.

One step = steps (a)-(d) of the path over one layer of the workload, in the
order of chunked prefill (Algorithm 2): for every outer chunk, the block
representatives, fingerprints and anchor clusters of the chunk, then one
selection and one block-sparse causal attention call per unit (cluster, or
sub-chunk in the per-sub-chunk mode). The same layer with all units in one
launch per step is reported as "batched". Inputs are resident in HBM before
timing; they are larger than L2 (Q, K, V of the 128K workload are 1.6 GB).

Prints one JSON line (rank 0). ``--impl reference`` times the CPU fp64 oracle
instead, on the same bounded sample of the same workload as the CPU leg.
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
sys.path.insert(0, ROOT)

from synth import generate_layer, workload  # noqa: E402

METRIC = "sparse-prefill tokens/sec and TTFT at 128K ctx on 1 GB300; % of roofline"
DEFAULT_WORKLOAD = "llama8b-128k"
KERNEL_SRC = os.path.join(ROOT, "paper_2609_31568_gb300", "csrc", "attn.cu")
PROFILE_DIR = os.path.join(ROOT, "profiles")


def parse_args():
    ap = argparse.ArgumentParser(description=__doc__)
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["scale", "reference"], default="scale")
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--mode", choices=["cluster", "subchunk"], default="cluster")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--selection-check", action="store_true",
                    help="without the CPU baseline: still compare the GPU selection with the oracle's steps (a)-(c)")
    ap.add_argument("--no-other-configs", action="store_true",
                    help="skip the side runs of the other workload configs after the headline")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-full", action="store_true",
                    help="skip timing the oracle over every row of the 4K and 32K layers")
    ap.add_argument("--no-baseline-mode", action="store_true",
                    help="skip timing the per-sub-chunk selection mode alongside")
    ap.add_argument("--paged", type=int, default=0, metavar="P",
                    help="keep K and V in a paged cache of P-token pages (shuffled page order)")
    ap.add_argument("--decode", action="store_true",
                    help="decode steps with the selection cache at the end of the context (one JSON line)")
    ap.add_argument("--stage", choices=["select"], default=None,
                    help="time one stage alone over the whole layer (one JSON line): 'select' = scale_select "
                         "(steps (b)-(c)) after one step (a)")
    ap.add_argument("--sweep", action="store_true",
                    help="clustering-threshold sweep (theta x L_max) on planted-topic data: cluster sizes, "
                         "overlap ratio rho, boundary recall and step time (one JSON line)")
    return ap.parse_args()


# --------------------------------------------------------------------------- helpers


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            pk = json.load(f)
        return dict(hbm=pk.get("hbm_gbs", 6800.0), bf16=pk.get("bf16_tflops", 1900.0),
                    bf16_sustained=pk.get("bf16_tflops_sustained", 1700.0), source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sustained=1700.0, source="fallback")


def launches(w, selects: int = 1, builds: int = 1) -> dict:
    """Kernels the path launches for workload w with `builds` step-(a) calls and
    `selects` select + attend calls (block size 1 skips the representatives,
    scores in four kernels and gathers the distant keys through a per-unit
    list)."""
    tok = w.block_size == 1
    build = (2 if tok else 3) + (1 if w.max_cluster_subchunks > 1 else 0)
    # the top-k is one kernel, or 8 (init, 4 histogram passes, count, scan,
    # emit) for units of more than 64K candidates
    topk = 8 if tok and w.n_blocks > 65536 else 1
    if tok:
        select = 4 + topk
    else:
        # logits, then statistics + vote + top-k in one kernel up to 4096 blocks
        select = 2 if w.n_blocks <= 4096 and w.num_q_heads <= 256 else 3 + topk
    attend = 3 if tok else 1
    return {"build_reps": build * builds, "select": select * selects, "attend": attend * selects,
            "total": build * builds + (select + attend) * selects}


def host_link_gbs(host, dev_bytes, stream) -> dict:
    """H2D and D2H bandwidth of one pinned copy each way (up to 512 MB), timed
    with CUDA events: what the host link gave the end-to-end call on this machine."""
    import torch

    n = min(host.numel() * host.element_size(), dev_bytes.numel(), 512 << 20)
    src = host.view(torch.uint8).reshape(-1)[:n]
    dst = dev_bytes[:n]
    out = {}
    for name, (a, b) in (("h2d", (dst, src)), ("d2h", (src, dst))):
        a.copy_(b, non_blocking=True)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        a.copy_(b, non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize()
        out[name] = n / (e0.elapsed_time(e1) / 1e3) / 1e9
    return out


def key_counts(w, unit_start, n_units, sel, cnt, per_subchunk):
    """Sum over query rows of |K(p)|, the distinct keys each row attends to (Eq. 10)."""
    total = 0
    for u in range(n_units):
        a = u if per_subchunk else int(unit_start[u])
        b = u + 1 if per_subchunk else int(unit_start[u + 1])
        s, e = a * w.sub_chunk, min(w.n_tokens, b * w.sub_chunk)
        W = max(0, s - w.n_local)
        D = min(w.n_sink, W)
        for blk in sel[u, : int(cnt[u])]:
            lo = max(int(blk) * w.block_size, w.n_sink)
            hi = min((int(blk) + 1) * w.block_size, W)
            D += max(0, hi - lo)
        n = e - s
        total += n * D + n * (s - W + 1) + n * (n - 1) // 2
    return total


def kernel_source_hash(path: str) -> str:
    """sha256[:16] of a CUDA source with its comments and blank lines removed:
    a change to the code changes it, a change to a comment does not."""
    with open(path) as f:
        txt = f.read()
    txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
    txt = re.sub(r"//[^\n]*", "", txt)
    code = "\n".join(ln.rstrip() for ln in txt.splitlines() if ln.strip())
    return hashlib.sha256(code.encode()).hexdigest()[:16]


def profile_counters(workload_name: str) -> dict:
    """ncu counters of the attention kernel on this workload, from the
    machine-readable sidecar committed beside its summary
    (profiles/attn_<workload>_ncu.json). Empty when there is none or when the
    kernel's code changed since the capture (the hash of its source without
    comments is stored with it)."""
    path = os.path.join(PROFILE_DIR, f"attn_{workload_name}_ncu.json")
    if not os.path.exists(path):
        return {}
    with open(path) as f:
        rec = json.load(f)
    return rec if rec.get("kernel_code_sha16") == kernel_source_hash(KERNEL_SRC) else {}


class ClockSampler:
    """nvidia-smi samples every 200 ms while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int = 0):
        self.dev = device_index
        self.proc = None
        self.path = None

    def start(self):
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        try:
            import torch

            uuid = str(torch.cuda.get_device_properties(self.dev).uuid)
            sel = ["-i", uuid if uuid.startswith("GPU-") else "GPU-" + uuid]
        except Exception:
            sel = ["-i", str(self.dev)]
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", *sel, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
            time.sleep(0.4)
        except FileNotFoundError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    mx.append(float(parts[2]))
                except ValueError:
                    continue
                for n, val in zip(names, parts[5:9]):
                    if val.lower() == "active":
                        reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "samples": len(sm)}


# --------------------------------------------------------------------------- oracle timing

# The oracle's row sample: the same seeded rows in the main arm's CPU leg and
# in the reference arm, so that the two report the same quantity.
ORACLE_ROWS = 512
ORACLE_ROW_SEED = 7
# Workloads the CPU leg also times in full (every row of Eq. 10).
FULL_ORACLE_WORKLOADS = ("gqa4-4k", "llama8b-32k")


def _cores() -> int:
    omp = os.environ.get("OMP_NUM_THREADS")
    if omp:
        return int(omp)
    return len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()


def oracle_sample(w, q, k, v, per_subchunk, rows=ORACLE_ROWS, seed=ORACLE_ROW_SEED):
    """One timed run of the oracle on a bounded sample: steps (a)-(c) over the
    whole layer, Eq. 10 on `rows` seeded rows (all rows when rows >= N). The
    throughput extrapolates the per-row time of Eq. 10 to every row."""
    import oracle

    t0 = time.perf_counter()
    ref = oracle.run_path(w, q, k, v, per_subchunk=per_subchunk)
    t_abc = time.perf_counter() - t0
    if rows >= w.n_tokens:
        sample = np.arange(w.n_tokens, dtype=np.int64)
    else:
        sample = np.sort(np.random.default_rng(seed).choice(w.n_tokens, size=rows, replace=False))
    t1 = time.perf_counter()
    oracle.attention_rows(q=q, k=k, v=v, sub_chunk=w.sub_chunk, block_size=w.block_size,
                          top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                          attn_scale=1.0 / np.sqrt(w.head_dim), per_subchunk=per_subchunk,
                          unit_start=ref["unit_start"], sel=ref["sel"],
                          sel_count=ref["sel_count"], rows=sample)
    t_d = time.perf_counter() - t1
    n = len(sample)
    t_full = t_abc + t_d / n * w.n_tokens
    return dict(tokens_per_s=w.n_tokens / t_full, t_full=t_full, t_abc=t_abc, t_d=t_d, t_run=t_abc + t_d,
                rows=n, extrapolated=n < w.n_tokens, cores=_cores(), ref=ref)


def sample_label(w, r) -> str:
    if not r["extrapolated"]:
        return (f"the whole layer: steps (a)-(c) and Eq. 10 on all {w.n_tokens} rows "
                f"({r['t_abc']:.2f} s + {r['t_d']:.2f} s)")
    return (f"steps (a)-(c) over all {w.n_tokens} tokens ({r['t_abc']:.2f} s) + Eq. 10 on {r['rows']} "
            f"seeded rows ({r['t_d']:.2f} s); Eq. 10's time per row extrapolated to all {w.n_tokens} rows")


def selection_agreement(w, ref, sel, cnt) -> dict:
    """GPU selection against the oracle's, unit by unit: identical, different
    at a near-tie (oracle k-th vs (k+1)-th relative gap < 1e-3: both are
    correct), and different otherwise (a parity failure)."""
    n = len(ref["sel_count"])
    match = near = bad = 0
    for u in range(n):
        c = int(ref["sel_count"][u])
        if int(cnt[u]) == c and np.array_equal(sel[u, :c], ref["sel"][u, :c]):
            match += 1
        elif ref["gap"][u] < 1e-3:
            near += 1
        else:
            bad += 1
    return {"selection_match_units": match, "near_tie_units": near, "selection_mismatch_units": bad,
            "units": n, "near_tie_gap": 1e-3}


# --------------------------------------------------------------------------- arms


def workload_config(w, mode_name: str) -> dict:
    """The workload keys of the JSON line's config, shared by both arms."""
    return {"workload": w.name, "n_tokens": w.n_tokens, "q_heads": w.num_q_heads, "kv_heads": w.num_kv_heads,
            "head_dim": w.head_dim, "sub_chunk": w.sub_chunk, "outer_chunk": w.outer_chunk,
            "max_cluster_subchunks": w.max_cluster_subchunks, "block_size": w.block_size, "top_k": w.top_k,
            "n_sink": w.n_sink, "n_local": w.n_local, "theta": w.theta, "mode": mode_name}


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_reference(args):
    """The oracle as the reference arm: every step is the same bounded sample
    as the main arm's CPU leg (steps (a)-(c) over the layer + Eq. 10 on
    ORACLE_ROWS seeded rows). ms_per_step is the time of what ran; value is
    the extrapolated whole-layer throughput, labelled as such."""
    world, rank, local = dist_setup(args)
    if rank != 0:
        return 0
    w = workload(args.workload)
    per_sub = args.mode == "subchunk"
    q, k, v = generate_layer(w)
    runs = []
    for i in range(args.warmup + args.steps):
        r = oracle_sample(w, q, k, v, per_sub)
        r.pop("ref")
        if i >= args.warmup:
            runs.append(r)
    t_full = statistics.mean(r["t_full"] for r in runs)
    t_run = statistics.mean(r["t_run"] for r in runs)
    value = w.n_tokens / t_full
    last = runs[-1]
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": t_run * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": dict(workload_config(w, args.mode), parallelism="host cores (oracle)"),
        "extrapolated": last["extrapolated"], "rows_timed": last["rows"], "rows_total": w.n_tokens,
        "ms_per_step_extrapolated": t_full * 1e3,
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": last["cores"], "kind": "oracle",
                         "sample": "per step: " + sample_label(w, last), "extrapolated": last["extrapolated"],
                         "rows_timed": last["rows"], "rows_total": w.n_tokens},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


def loop_calls(w, mode_sub: bool):
    """One step of chunked prefill as Algorithm 2 orders it: for every outer
    chunk, step (a) over the chunk, then one selection and one attention call
    per unit. A per-sub-chunk unit is one sub-chunk; in SCR mode the calls
    cover the chunk's clusters (one per chunk when theta admits every
    sub-chunk and the outer chunk is one cluster long, as in the timed
    workloads). Returns [(chunk range, [unit ranges])]."""
    out = []
    for t0 in range(0, w.n_tokens, w.outer_chunk):
        t1 = min(w.n_tokens, t0 + w.outer_chunk)
        units = ([(a, min(t1, a + w.sub_chunk)) for a in range(t0, t1, w.sub_chunk)] if mode_sub else [(t0, t1)])
        out.append(((t0, t1), units))
    return out


# The other workload configs, each run after the headline as its own process
# (Algorithm 2 loop in both modes, plus the whole-sequence launches), with the
# GPU selection compared with the oracle's where steps (a)-(c) fit in seconds.
OTHER_CONFIGS = (("gqa4-4k", True), ("llama8b-32k", True), ("llama8b-64k-32l", False), ("llama8b-1m", True),
                 ("llama8b-128k-tok", True), ("llama8b-1m-tok", False))
OTHER_STEPS, OTHER_WARMUP = 3, 3


def other_configs() -> dict:
    """Side runs of the other configs: per workload the SCR and per-sub-chunk
    loops (TTFT of one layer, or of the stack), attention throughput, selection
    time and retrieval calls, and the selection agreement with the oracle."""
    import subprocess

    out = {}
    for name, check in OTHER_CONFIGS:
        cmd = [sys.executable, os.path.abspath(__file__), "--workload", name, "--steps", str(OTHER_STEPS),
               "--warmup", str(OTHER_WARMUP), "--no-e2e", "--no-cpu-baseline", "--no-other-configs"]
        if check:
            cmd.append("--selection-check")
        t0 = time.perf_counter()
        r = subprocess.run(cmd, capture_output=True, text=True, cwd=ROOT)
        wall = time.perf_counter() - t0
        lines = [ln for ln in r.stdout.splitlines() if ln.startswith("{")]
        if r.returncode != 0 or not lines:
            out[name] = {"error": (r.stderr.strip().splitlines() or ["no output"])[-1][:300], "rc": r.returncode}
            continue
        d = json.loads(lines[-1])
        o = d.get("other_mode", {})
        rec = {
            "n_tokens": d["config"]["n_tokens"], "layers": d["config"].get("layers", 1),
            "steps": d["steps"], "warmup": d["warmup"], "wall_s": round(wall, 1),
            "cluster": {"ttft_ms": d["ms_per_step"], "tokens_per_s": d["value"],
                        "attention_tflops": d["roofline"]["achieved"], "attention_frac": d["roofline"]["frac"],
                        "select_ms": d.get("stages_ms", {}).get("select"),
                        "retrieval_calls": d["retrieval_calls"], "units": d["units"],
                        "batched_ms": d.get("batched", {}).get("ms_per_step")},
            "subchunk": {"ttft_ms": o.get("ms_per_step"), "tokens_per_s": o.get("tokens_per_s"),
                         "attention_tflops": o.get("attn_tflops"),
                         "select_ms": o.get("stages_ms", {}).get("select"),
                         "retrieval_calls": o.get("retrieval_calls"), "units": o.get("units"),
                         "batched_ms": o.get("batched", {}).get("ms_per_step")},
            "scr_over_subchunk": d.get("scr_over_subchunk"), "attn_flops_ratio": d.get("attn_flops_ratio"),
            "clocks": d.get("clocks"),
        }
        if "selection_match_units" in d:
            rec["selection"] = {k: d[k] for k in ("selection_match_units", "near_tie_units",
                                                  "selection_mismatch_units")}
        out[name] = rec
    return out


def run_scale(args):
    import torch

    world, rank, local = dist_setup(args)
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    import paper_2609_31568_gb300 as pkg
    from paper_2609_31568_gb300 import scale as S

    pkg.build()
    S.load()
    w = workload(args.workload)
    mode = S.SCALE_MODE_PER_SUBCHUNK if args.mode == "subchunk" else S.SCALE_MODE_PER_CLUSTER
    per_sub = mode == S.SCALE_MODE_PER_SUBCHUNK
    # weak scaling: every rank prefills its own independent layer (seed + rank)
    q, k, v = generate_layer(w, seed=w.seed + rank)
    dev = [torch.from_numpy(x).view(torch.bfloat16).cuda() for x in (q, k, v)]
    p = S.params_for(w)
    stream = torch.cuda.current_stream()
    kv = None
    if args.paged:
        # K and V moved into a pool of pages in shuffled order (plus spare pages)
        P = args.paged
        n_pages = -(-w.n_tokens // P)
        order = torch.from_numpy(np.random.default_rng(1).permutation(n_pages + 4)[:n_pages].astype(np.int32)).cuda()
        pools = []
        for x in dev[1:]:
            pool = torch.zeros((n_pages + 4, P, w.num_kv_heads, w.head_dim), dtype=x.dtype, device="cuda")
            full = torch.zeros((n_pages * P, w.num_kv_heads, w.head_dim), dtype=x.dtype, device="cuda")
            full[: w.n_tokens] = x
            pool[order.long()] = full.view(n_pages, P, w.num_kv_heads, w.head_dim)
            pools.append(pool)
            del full
        kv = S.kv_pages(pools[0], pools[1], order, P)

    def barrier():
        if world > 1:
            torch.distributed.barrier()

    def build(buf_, t0, t1, whole):
        if kv is not None:
            if whole:
                S.scale_build_reps_paged(p, dev[0], kv, buf_.reps, buf_.fingerprints, buf_.unit_start,
                                         buf_.n_units, buf_.ws, stream)
            else:
                S.scale_build_reps_range_paged(p, t0, t1, dev[0], kv, buf_.reps, buf_.fingerprints,
                                               buf_.unit_start, buf_.n_units, buf_.ws, stream)
        elif whole:
            S.scale_build_reps(p, dev[0], dev[1], buf_.reps, buf_.fingerprints, buf_.unit_start,
                               buf_.n_units, buf_.ws, stream)
        else:
            S.scale_build_reps_range(p, t0, t1, dev[0], dev[1], buf_.reps, buf_.fingerprints,
                                     buf_.unit_start, buf_.n_units, buf_.ws, stream)

    def select(mode_, buf_, t0, t1):
        if kv is not None and w.block_size == 1:
            S.scale_select_tokens_paged(p, mode_, t0, t1, kv, buf_.fingerprints, buf_.unit_start,
                                        buf_.n_units, buf_.sel_blocks, buf_.sel_count, None, buf_.ws, stream)
        else:
            S.select(p, mode_, t0, t1, dev[1], buf_, stream)

    def attend(mode_, buf_, t0, t1):
        if kv is not None:
            S.scale_sparse_prefill_paged(p, mode_, t0, t1, dev[0], kv, buf_.unit_start, buf_.n_units,
                                         buf_.sel_blocks, buf_.sel_count, buf_.out, buf_.ws, stream)
        else:
            S.scale_sparse_prefill(p, mode_, t0, t1, *dev, buf_.unit_start, buf_.n_units,
                                   buf_.sel_blocks, buf_.sel_count, buf_.out, buf_.ws, stream)

    def step_plan(mode_, batched):
        """[(build range, [(select/attend range)])] of one step."""
        if batched:
            return [((0, w.n_tokens), [(0, w.n_tokens)])]
        return loop_calls(w, mode_ == S.SCALE_MODE_PER_SUBCHUNK)

    def timed(mode_, batched, steps, warmup, buf_, sample_clocks=False):
        """Time `steps` steps (CUDA events on the launch stream): the whole step,
        and the three stages summed over their calls within it."""
        plan = step_plan(mode_, batched)
        n_calls = sum(len(u) for _, u in plan)

        def one(ev):
            def rec(stage, j):
                if ev is not None:
                    ev[stage][j].record(stream)

            j = 0
            for (c0, c1), units in plan:
                for i, (t0, t1) in enumerate(units):
                    rec(0, j)
                    if i == 0:
                        build(buf_, c0, c1, batched)
                    rec(1, j)
                    select(mode_, buf_, t0, t1)
                    rec(2, j)
                    attend(mode_, buf_, t0, t1)
                    rec(3, j)
                    j += 1

        for _ in range(warmup):
            one(None)
        torch.cuda.synchronize()
        barrier()
        torch.cuda.synchronize()
        evs = [[[torch.cuda.Event(enable_timing=True) for _ in range(n_calls)] for _ in range(4)]
               for _ in range(steps)]
        clocks = ClockSampler(torch.cuda.current_device()) if sample_clocks else None
        if clocks:
            clocks.start()
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for i in range(steps):
            one(evs[i])
        end.record(stream)
        torch.cuda.synchronize()
        clk = clocks.stop() if clocks else None
        barrier()
        total = start.elapsed_time(end) / steps
        # stage sums per step (a unit after its chunk's first has no build)
        stages = [statistics.mean(sum(e[jj][c].elapsed_time(e[jj + 1][c]) for c in range(n_calls)) for e in evs)
                  for jj in range(3)]
        st = S.scale_get_device_status(buf_.ws)
        if st != S.SCALE_OK:
            raise RuntimeError(f"device status {st}: {S.status_string(st)}")
        return {"ms_per_step": total, "tokens_per_s": w.n_tokens / (total / 1e3),
                "stages_ms": {"build_reps": stages[0], "select": stages[1], "sparse_attention": stages[2]},
                "build_calls": len(plan), "select_attend_calls": n_calls,
                "gpu_launches": launches(w, n_calls, len(plan))["total"]}, clk

    def unit_stats(mode_, buf_):
        sub = mode_ == S.SCALE_MODE_PER_SUBCHUNK
        n = w.n_subchunks if sub else int(buf_.n_units.item())
        us = buf_.unit_start.cpu().numpy()
        sel = buf_.sel_blocks.cpu().numpy()
        cnt = buf_.sel_count.cpu().numpy()
        keys = key_counts(w, us, n, sel, cnt, sub)
        _, calls = S.scale_retrieval_calls(p, mode_, None if sub else us[: n + 1], n)
        return n, calls, 4.0 * w.head_dim * w.num_q_heads * keys, sel[:n], cnt[:n]

    buf = pkg.allocate(p, mode)
    # headline: the chunked-prefill loop of Algorithm 2
    head, clk = timed(mode, False, args.steps, args.warmup, buf, sample_clocks=True)
    ms = head["ms_per_step"]
    if world > 1:
        t = torch.tensor([ms], device="cuda")
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        ms = float(t.item())
    n_units, calls, flops, sel_gpu, cnt_gpu = unit_stats(mode, buf)
    peaks = load_peaks()
    attn_ms = head["stages_ms"]["sparse_attention"]
    n_attn = head["select_attend_calls"]
    achieved = flops / (attn_ms / 1e3) / 1e12
    prof = profile_counters(w.name) if kv is None else {}
    mode_name = "subchunk" if per_sub else "cluster"
    line = {
        "metric": METRIC,
        "value": world * w.n_tokens / (ms / 1e3),
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": ms,
        "ttft_ms": ms,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "bf16",
        "data": "synthetic",
        "config": {**workload_config(w, mode_name), "parallelism": f"independent layers x{world}",
                   "loop": ("Algorithm 2: per outer chunk scale_build_reps_range, then one scale_select and "
                            "one scale_sparse_prefill per unit (" +
                            ("sub-chunk" if per_sub else "cluster; one per outer chunk at theta = -1") + ")"),
                   "kv_layout": f"paged, {args.paged}-token pages" if args.paged else "contiguous",
                   "l2": "inputs larger than L2 (Q+K+V %.2f GB)" % ((q.nbytes + k.nbytes + v.nbytes) / 1e9)},
        "stages_ms": head["stages_ms"],
        "calls_per_step": {"build_reps_range": head["build_calls"], "select": n_attn, "sparse_prefill": n_attn},
        "retrieval_calls": calls,
        "units": n_units,
        "roofline": {"bound": "tensor", "kernel": "k_sparse_attn", "achieved": achieved,
                     "peak": peaks["bf16"], "unit": "TFLOP/s", "frac": achieved / peaks["bf16"],
                     "peak_source": f"bf16 burst, of {peaks['source']}",
                     "frac_of_sustained": achieved / peaks["bf16_sustained"],
                     "launches_per_step": n_attn,
                     "algorithmic_flops_per_launch": flops / n_attn,
                     "ms_per_launch": attn_ms / n_attn,
                     "traffic": prof.get("traffic_bytes_per_launch"),
                     "tensor_pipe_active_pct": prof.get("tensor_pipe_active_pct"),
                     "counters_from": prof.get("summary")},
        "gpu_launches": args.steps * head["gpu_launches"],
        "clocks": clk,
    }

    if rank == 0:
        bat, _ = timed(mode, True, max(3, args.steps // 2), 2, buf)
        line["batched"] = dict(bat, loop="whole sequence: scale_build_reps, scale_select, scale_sparse_prefill "
                                         "(all units of the layer in one launch each)")

    if not args.no_baseline_mode and rank == 0:
        other = S.SCALE_MODE_PER_SUBCHUNK if not per_sub else S.SCALE_MODE_PER_CLUSTER
        buf2 = pkg.allocate(p, other)
        o_loop, _ = timed(other, False, max(3, args.steps // 2), 2, buf2)
        o_bat, _ = timed(other, True, max(3, args.steps // 2), 2, buf2)
        n2, calls2, flops2, _, _ = unit_stats(other, buf2)
        other_name = "subchunk" if other == S.SCALE_MODE_PER_SUBCHUNK else "cluster"
        line["other_mode"] = dict(o_loop, mode=other_name, retrieval_calls=calls2, units=n2,
                                  attn_tflops=flops2 / (o_loop["stages_ms"]["sparse_attention"] / 1e3) / 1e12,
                                  batched=o_bat)
        scr, sub = (head, o_loop) if not per_sub else (o_loop, head)
        scr_b, sub_b = (line["batched"], o_bat) if not per_sub else (o_bat, line["batched"])
        f_scr, f_sub = (flops, flops2) if not per_sub else (flops2, flops)
        line["scr_over_subchunk"] = scr["ms_per_step"] / sub["ms_per_step"]
        line["scr_over_subchunk_batched"] = scr_b["ms_per_step"] / sub_b["ms_per_step"]
        line["attn_flops_ratio"] = f_scr / f_sub
        line["retrieval"] = {
            "cluster": {"calls": calls if not per_sub else calls2,
                        "select_ms": scr["stages_ms"]["select"]},
            "subchunk": {"calls": calls2 if not per_sub else calls,
                         "select_ms": sub["stages_ms"]["select"]}}
        del buf2

    if not args.no_e2e:
        qh, kh, vh = (torch.from_numpy(x).pin_memory() for x in (q, k, v))
        oh = torch.empty(qh.shape, dtype=torch.int16).pin_memory()
        arena = torch.empty(S.scale_prefill_host_arena_size(p, mode), dtype=torch.uint8, device="cuda")
        S.scale_prefill_host(p, mode, qh, kh, vh, oh, arena, stream)
        reps = max(5, args.steps // 2)
        link = host_link_gbs(qh, arena, stream)
        torch.cuda.synchronize()
        barrier()
        per_call = []
        for _ in range(reps):
            t0 = time.perf_counter()
            S.scale_prefill_host(p, mode, qh, kh, vh, oh, arena, stream)
            per_call.append(time.perf_counter() - t0)
        # The median call: host-device copies share the host's memory system
        # with other jobs on the machine, and a call now and then stalls on
        # it (the mean and the extremes are reported beside).
        t_e2e = statistics.median(per_call)
        if world > 1:
            t = torch.tensor([t_e2e], device="cuda")
            torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
            t_e2e = float(t.item())
        line["e2e"] = {"value": world * w.n_tokens / t_e2e, "unit": "tokens/s",
                       "h2d_bytes_per_step": int(q.nbytes + k.nbytes + v.nbytes),
                       "d2h_bytes_per_step": int(q.nbytes), "ms_per_step": t_e2e * 1e3,
                       "stat": f"median of {reps} calls", "ms_mean": sum(per_call) / reps * 1e3,
                       "ms_min": min(per_call) * 1e3, "ms_max": max(per_call) * 1e3,
                       "host_link_gbs": link,
                       "api": "scale_prefill_host (pinned host buffers; pieces of outer chunks, copies "
                              "overlapped with the compute)"}
        del arena

    if rank == 0 and world == 1 and args.no_cpu_baseline and args.selection_check:
        import oracle

        line.update(selection_agreement(w, oracle.run_path(w, q, k, v, per_subchunk=per_sub), sel_gpu, cnt_gpu))

    if rank == 0 and world == 1 and not args.no_other_configs and w.name == DEFAULT_WORKLOAD and not args.paged:
        line["other_configs"] = other_configs()

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        r = oracle_sample(w, q, k, v, per_sub)
        line.update(selection_agreement(w, r["ref"], sel_gpu, cnt_gpu))
        line["cpu_baseline"] = {
            "value": r["tokens_per_s"], "unit": "tokens/s", "cores": r["cores"], "kind": "oracle",
            "sample": sample_label(w, r), "extrapolated": r["extrapolated"], "rows_timed": r["rows"],
            "rows_total": w.n_tokens, "ms_run": r["t_run"] * 1e3}
        if not args.no_cpu_full and w.name == DEFAULT_WORKLOAD:
            full = {}
            for name in FULL_ORACLE_WORKLOADS:
                wf = workload(name)
                qf, kf, vf = generate_layer(wf)
                rf = oracle_sample(wf, qf, kf, vf, per_sub, rows=wf.n_tokens)
                full[name] = {"tokens_per_s": rf["tokens_per_s"], "s": rf["t_full"], "extrapolated": False,
                              "sample": sample_label(wf, rf)}
            line["cpu_baseline"]["full_layers"] = full

    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


SWEEP_WORKLOAD = "llama8b-128k-topics"
SWEEP_THETAS = (0.95, 0.97, 0.99)
SWEEP_SMAX = (2, 4, 8)


def cosine_stats(fp: np.ndarray) -> dict:
    """Distribution of cos(v_i, v_{i+1}) over consecutive sub-chunks (the paper's Table 2 format)."""
    vt = fp / np.linalg.norm(fp, axis=1, keepdims=True)
    c = np.sum(vt[1:] * vt[:-1], axis=1)
    return {"mean": float(c.mean()), "min": float(c.min()), "max": float(c.max()),
            "p10": float(np.percentile(c, 10)), "median": float(np.median(c)),
            "p90": float(np.percentile(c, 90))}


def boundary_recall(w, unit_start: np.ndarray) -> dict:
    """Share of planted topic boundaries at which a cluster opens: at the
    sub-chunk that contains the boundary or at the first one after it."""
    from synth import topic_segments

    starts, _ = topic_segments(w, 0, w.seed)
    opened = set(int(x) for x in unit_start[:-1])
    hits = 0
    for b in starts[1:]:
        i = int(b) // w.sub_chunk
        hits += (i in opened) or (i + 1 in opened)
    return {"boundaries": int(len(starts) - 1), "recalled": int(hits)}


def run_sweep(args):
    """Alg. 1's threshold branch on planted-topic data: for every (L_max, theta),
    the step time, the clusters formed, their retrieval calls, and the overlap
    ratio of Sec. IV-C against the per-sub-chunk union (both with member
    queries scored on the cluster's candidates and with the members' own
    per-sub-chunk selections)."""
    import torch

    import paper_2609_31568_gb300 as pkg
    from paper_2609_31568_gb300 import fidelity as F
    from paper_2609_31568_gb300 import scale as S

    pkg.build()
    S.load()
    w0 = workload(args.workload if args.workload != DEFAULT_WORKLOAD else SWEEP_WORKLOAD)
    q, k, v = generate_layer(w0)
    dev = [torch.from_numpy(x).view(torch.bfloat16).cuda() for x in (q, k, v)]
    stream = torch.cuda.current_stream()
    CL, SUB = S.SCALE_MODE_PER_CLUSTER, S.SCALE_MODE_PER_SUBCHUNK
    peaks = load_peaks()

    def step(p, mode, buf, steps, warmup):
        for _ in range(warmup):
            pkg.run_path(p, mode, *dev, buf)
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
        torch.cuda.synchronize()
        for e in ev:
            e[0].record(stream)
            S.scale_build_reps(p, dev[0], dev[1], buf.reps, buf.fingerprints, buf.unit_start,
                               buf.n_units, buf.ws, stream)
            e[1].record(stream)
            S.select(p, mode, 0, w0.n_tokens, dev[1], buf, stream)
            e[2].record(stream)
            S.scale_sparse_prefill(p, mode, 0, w0.n_tokens, *dev, buf.unit_start, buf.n_units,
                                   buf.sel_blocks, buf.sel_count, buf.out, buf.ws, stream)
            e[3].record(stream)
        torch.cuda.synchronize()
        st = S.scale_get_device_status(buf.ws)
        if st != S.SCALE_OK:
            raise RuntimeError(f"device status {st}: {S.status_string(st)}")
        stages = [statistics.mean(x[j].elapsed_time(x[j + 1]) for x in ev) for j in range(3)]
        return sum(stages), stages

    steps, warmup = max(3, args.steps // 4), max(2, args.warmup)
    pb = S.params_for(w0)
    bufb = pkg.allocate(pb, SUB)
    ms_b, st_b = step(pb, SUB, bufb, steps, warmup)
    M = w0.n_subchunks
    sel_sub = bufb.sel_blocks.cpu().numpy()
    cnt_sub = bufb.sel_count.cpu().numpy()
    _, calls_b = S.scale_retrieval_calls(pb, SUB, None, M)
    keys_b = key_counts(w0, None, M, sel_sub, cnt_sub, True)
    cos = cosine_stats(bufb.fingerprints.double().cpu().numpy())
    del bufb

    rows = []
    for s_max in SWEEP_SMAX:
        for theta in SWEEP_THETAS:
            w = w0.replace(max_cluster_subchunks=s_max, theta=theta)
            p = S.params_for(w)
            buf = pkg.allocate(p, CL)
            ms, st = step(p, CL, buf, steps, warmup)
            n = int(buf.n_units.item())
            us = buf.unit_start[: n + 1].cpu().numpy()
            sizes = np.diff(us)
            sel = buf.sel_blocks.cpu().numpy()
            cnt = buf.sel_count.cpu().numpy()
            same = {}
            for j in range(1, s_max):
                fpj = F.member_query_fingerprints(buf.fingerprints, buf.unit_start, n, j)
                sj, cj = torch.empty_like(buf.sel_blocks), torch.empty_like(buf.sel_count)
                S.scale_select(p, CL, 0, w.n_tokens, buf.reps, fpj, buf.unit_start, buf.n_units,
                               sj, cj, None, buf.ws, stream)
                same[j] = (sj.cpu().numpy(), cj.cpu().numpy())
            if S.scale_get_device_status(buf.ws) != S.SCALE_OK:
                raise RuntimeError("device status after member selections")
            rho_same, _ = F.overlap_ratios(us, sel, cnt, lambda u, j: same[j][0][u, : same[j][1][u]])
            rho_own, _ = F.overlap_ratios(
                us, sel, cnt, lambda u, j: sel_sub[us[u] + j, : cnt_sub[us[u] + j]])
            _, calls = S.scale_retrieval_calls(p, CL, us, n)
            keys = key_counts(w, us, n, sel, cnt, False)
            flops = 4.0 * w.head_dim * w.num_q_heads * keys
            hist = {str(c): int(np.count_nonzero(sizes == c)) for c in range(1, s_max + 1)}
            rows.append({
                "l_max_subchunks": s_max, "theta": theta, "ms_per_step": ms,
                "stages_ms": {"build_reps": st[0], "select": st[1], "sparse_attention": st[2]},
                "units": n, "retrieval_calls": calls,
                "mean_cluster_tokens": float(w.n_tokens / n), "cluster_sizes": hist,
                "full_clusters": float(np.mean(sizes == s_max)),
                "rho_same_candidates": F.summary(rho_same), "rho_own_selection": F.summary(rho_own),
                "boundary_recall": boundary_recall(w, us),
                "attn_tflops": flops / (st[2] / 1e3) / 1e12,
                "attn_flops_vs_per_subchunk": keys / keys_b,
            })
            del buf
            torch.cuda.empty_cache()
    line = {
        "metric": "clustering-threshold sweep: cluster sizes, overlap ratio, retrieval calls, step time",
        "workload": w0.name, "n_tokens": w0.n_tokens, "sub_chunk": w0.sub_chunk,
        "outer_chunk": w0.outer_chunk, "block_size": w0.block_size, "top_k_blocks": w0.top_k,
        "top_k_tokens": w0.top_k * w0.block_size, "steps": steps, "warmup": warmup,
        "data": "synthetic, planted topics", "consecutive_cosine": cos,
        "per_subchunk": {"ms_per_step": ms_b, "retrieval_calls": calls_b, "units": M,
                         "stages_ms": {"build_reps": st_b[0], "select": st_b[1], "sparse_attention": st_b[2]},
                         "attn_tflops": 4.0 * w0.head_dim * w0.num_q_heads * keys_b / (st_b[2] / 1e3) / 1e12},
        "peak_bf16_sustained_tflops": peaks["bf16_sustained"],
        "sweep": rows,
    }
    print(json.dumps(line), flush=True)
    return 0


DECODE_WORKLOAD = "llama8b-1m-tok"


def run_decode(args):
    """Decode steps at the end of the context: every step retrieving (no
    cache) against the selection cache reusing a retrieval for up to 16 steps.
    Queries are a random walk from the last prompt query (consecutive decode
    queries are close); K and V are the workload's. Attention-only TPOT."""
    import torch

    import paper_2609_31568_gb300 as pkg
    from paper_2609_31568_gb300 import scale as S
    from synth import bf16_bits_to_f32, f64_to_bf16_bits

    pkg.build()
    S.load()
    w = workload(args.workload if args.workload != DEFAULT_WORKLOAD else DECODE_WORKLOAD)
    n_steps = 64
    q, k, v = generate_layer(w)
    rng = np.random.default_rng(3)
    x = bf16_bits_to_f32(q[w.n_tokens - n_steps]).astype(np.float64)
    walk = []
    for _ in range(n_steps):
        walk.append(f64_to_bf16_bits(x))
        x = x + 0.07 * np.linalg.norm(x) / np.sqrt(x.size) * rng.standard_normal(x.shape)
    qd = torch.from_numpy(np.stack(walk)).view(torch.bfloat16).cuda()
    kd, vd = (torch.from_numpy(t).view(torch.bfloat16).cuda() for t in (k, v))
    del q
    positions = list(range(w.n_tokens - n_steps, w.n_tokens))
    stream = torch.cuda.current_stream()
    res = {}
    for label, theta, s_max in (("retrieve_every_step", 2.0, 1), ("selection_cache", -1.0, 16)):
        p = S.params_for(w, theta=theta, max_cluster_subchunks=s_max)
        cache = torch.empty(S.scale_decode_cache_size(p), dtype=torch.uint8, device="cuda")
        ws = torch.empty(S.scale_decode_workspace_size(p), dtype=torch.uint8, device="cuda")
        S.scale_workspace_init(ws)
        out = torch.empty((w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
        for _ in range(max(1, args.warmup)):
            S.scale_decode_cache_init(cache)
            for i, t in enumerate(positions[:8]):
                S.scale_decode_step(p, t, qd[i], kd, vd, cache, out, ws, stream)
        torch.cuda.synchronize()
        S.scale_decode_cache_init(cache)
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(n_steps + 1)]
        ev[0].record(stream)
        for i, t in enumerate(positions):
            S.scale_decode_step(p, t, qd[i], kd, vd, cache, out, ws, stream)
            ev[i + 1].record(stream)
        torch.cuda.synchronize()
        ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(n_steps)]
        st = S.scale_get_device_status(ws)
        if st != S.SCALE_OK:
            raise RuntimeError(f"device status {st}: {S.status_string(st)}")
        res[label] = {"tpot_ms": statistics.mean(ms), "retrieving_step_ms": ms[0],
                      "reusing_step_ms": statistics.median(ms[1:]) if s_max > 1 else None,
                      "retrievals": -(-n_steps // s_max)}
    line = {"metric": "decode TPOT (attention only) with the selection cache", "workload": w.name,
            "context": w.n_tokens, "top_k_tokens": w.top_k, "steps": n_steps,
            "value": 1000.0 / res["selection_cache"]["tpot_ms"], "unit": "tokens/s",
            "speedup_from_cache": res["retrieve_every_step"]["tpot_ms"] / res["selection_cache"]["tpot_ms"],
            "data": "synthetic (random-walk decode queries)", **res}
    print(json.dumps(line), flush=True)
    return 0


def run_stack(args):
    """Multi-layer workload: attention-only TTFT of a chunked prefill over all layers.

    Per step, for each outer chunk (in order) and each layer: step (a) over the
    chunk (scale_build_reps_range), then scale_select and scale_sparse_prefill
    restricted to that chunk's tokens -- the dependency order of a real chunked
    prefill, where a layer's Q, K and V of later chunks do not exist yet."""
    import torch

    world, rank, local = dist_setup(args)
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl")
    import paper_2609_31568_gb300 as pkg
    from paper_2609_31568_gb300 import scale as S

    pkg.build()
    S.load()
    w = workload(args.workload)
    p = S.params_for(w)
    stream = torch.cuda.current_stream()
    layers = []
    for l in range(w.layers):
        q, k, v = generate_layer(w, layer=l, seed=w.seed + l + 1000 * rank)
        layers.append([torch.from_numpy(x).view(torch.bfloat16).cuda() for x in (q, k, v)])
        del q, k, v
    def measure(mode, steps, warmup):
        bufs = [pkg.allocate(p, mode) for _ in layers]
        plan = loop_calls(w, mode == S.SCALE_MODE_PER_SUBCHUNK)
        n_attn = sum(len(u) for _, u in plan) * len(layers)

        def step(ev=None):
            i = 0
            for (c0, c1), units in plan:
                for dev, b in zip(layers, bufs):
                    S.scale_build_reps_range(p, c0, c1, dev[0], dev[1], b.reps, b.fingerprints, b.unit_start,
                                             b.n_units, b.ws, stream)
                    for t0, t1 in units:
                        S.select(p, mode, t0, t1, dev[1], b, stream)
                        if ev is not None:
                            ev[i][0].record(stream)
                        S.scale_sparse_prefill(p, mode, t0, t1, *dev, b.unit_start, b.n_units, b.sel_blocks,
                                               b.sel_count, b.out, b.ws, stream)
                        if ev is not None:
                            ev[i][1].record(stream)
                        i += 1

        for _ in range(warmup):
            step()
        torch.cuda.synchronize()
        if world > 1:
            torch.distributed.barrier()
        clocks = ClockSampler(torch.cuda.current_device())
        clocks.start()
        evs = [[[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(n_attn)] for _ in range(steps)]
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for i in range(steps):
            step(evs[i])
        end.record(stream)
        torch.cuda.synchronize()
        clk = clocks.stop()
        if world > 1:
            torch.distributed.barrier()
        ms = start.elapsed_time(end) / steps
        attn_ms = sum(e[0].elapsed_time(e[1]) for ev in evs for e in ev) / steps
        for b in bufs:
            st = S.scale_get_device_status(b.ws)
            if st != S.SCALE_OK:
                raise RuntimeError(f"device status {st}: {S.status_string(st)}")
        per_sub = mode == S.SCALE_MODE_PER_SUBCHUNK
        keys, calls, units = 0, 0, 0
        for b in bufs:
            n = w.n_subchunks if per_sub else int(b.n_units.item())
            us = b.unit_start.cpu().numpy()
            keys += key_counts(w, us, n, b.sel_blocks.cpu().numpy(), b.sel_count.cpu().numpy(), per_sub)
            units += n
            calls += S.scale_retrieval_calls(p, mode, None if per_sub else us[: n + 1], n)[1]
        del bufs
        launch_count = w.layers * launches(w, n_attn // w.layers, len(plan))["total"]
        return ms, attn_ms, clk, 4.0 * w.head_dim * w.num_q_heads * keys, calls, units, launch_count, n_attn

    mode = S.SCALE_MODE_PER_SUBCHUNK if args.mode == "subchunk" else S.SCALE_MODE_PER_CLUSTER
    ms, attn_ms, clk, flops, calls, units, n_launch, n_attn = measure(mode, args.steps, args.warmup)
    if world > 1:
        t = torch.tensor([ms], device="cuda")
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        ms = float(t.item())
    peaks = load_peaks()
    achieved = flops / (attn_ms / 1e3) / 1e12
    line = {
        "metric": METRIC, "value": world * w.n_tokens / (ms / 1e3), "unit": "tokens/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "ttft_ms": ms,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic",
        "config": {"workload": w.name, "n_tokens": w.n_tokens, "layers": w.layers, "mode": args.mode,
                   "outer_chunk": w.outer_chunk,
                   "loop": ("Algorithm 2, chunk-major: per outer chunk and layer scale_build_reps_range, then one "
                            "scale_select and one scale_sparse_prefill per unit"),
                   "parallelism": f"independent stacks x{world}", "l2": "inputs larger than L2"},
        "stages_ms": {"sparse_attention_total": attn_ms, "other": ms - attn_ms},
        "retrieval_calls": calls, "units": units,
        "roofline": {"bound": "tensor", "kernel": "k_sparse_attn", "achieved": achieved,
                     "peak": peaks["bf16"], "unit": "TFLOP/s", "frac": achieved / peaks["bf16"],
                     "peak_source": f"bf16 burst, of {peaks['source']}",
                     "frac_of_sustained": achieved / peaks["bf16_sustained"],
                     "launches_per_step": n_attn, "algorithmic_flops_per_launch": flops / n_attn,
                     "traffic": None},
        "gpu_launches": args.steps * n_launch,
        "clocks": clk,
    }
    if not args.no_baseline_mode and rank == 0:
        other = S.SCALE_MODE_PER_SUBCHUNK if mode == S.SCALE_MODE_PER_CLUSTER else S.SCALE_MODE_PER_CLUSTER
        ms2, attn2, _, flops2, calls2, units2, _, _ = measure(other, max(2, args.steps // 2), 1)
        line["other_mode"] = {"mode": "subchunk" if other == S.SCALE_MODE_PER_SUBCHUNK else "cluster",
                              "ms_per_step": ms2, "tokens_per_s": w.n_tokens / (ms2 / 1e3),
                              "sparse_attention_ms": attn2, "retrieval_calls": calls2, "units": units2,
                              "attn_tflops": flops2 / (attn2 / 1e3) / 1e12}
        per_sub_first = mode == S.SCALE_MODE_PER_SUBCHUNK
        line["scr_over_subchunk"] = (ms2 / ms) if per_sub_first else (ms / ms2)
        line["attn_flops_ratio"] = (flops2 / flops) if per_sub_first else (flops / flops2)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # the oracle on layer 0 (steps (a)-(c) in full, Eq. 10 on the fixed row
        # sample), extrapolated to every row of every layer
        q0, k0, v0 = generate_layer(w, layer=0, seed=w.seed + 0)
        r = oracle_sample(w, q0, k0, v0, mode == S.SCALE_MODE_PER_SUBCHUNK)
        line["cpu_baseline"] = {
            "value": r["tokens_per_s"] / w.layers, "unit": "tokens/s", "cores": r["cores"], "kind": "oracle",
            "sample": f"layer 0 of {w.layers}: " + sample_label(w, r) + f"; times {w.layers} layers",
            "extrapolated": True, "rows_timed": r["rows"], "rows_total": w.n_tokens * w.layers,
            "ms_run": r["t_run"] * 1e3}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def run_stage(args):
    """One stage of the path timed alone over the whole layer: scale_select
    (steps (b) and (c): scoring of every unit's candidates, soft vote, top-k)
    on the representatives and fingerprints of one step (a), in the chosen
    mode; CUDA events around each call on the launch stream."""
    import torch

    import paper_2609_31568_gb300 as pkg
    from paper_2609_31568_gb300 import scale as S

    pkg.build()
    S.load()
    w = workload(args.workload)
    mode = S.SCALE_MODE_PER_SUBCHUNK if args.mode == "subchunk" else S.SCALE_MODE_PER_CLUSTER
    q, k, v = generate_layer(w)
    dev = [torch.from_numpy(x).view(torch.bfloat16).cuda() for x in (q, k)]
    del q, k, v
    p = S.params_for(w)
    buf = pkg.allocate(p, mode)
    stream = torch.cuda.current_stream()
    S.scale_build_reps(p, dev[0], dev[1], buf.reps, buf.fingerprints, buf.unit_start, buf.n_units, buf.ws, stream)
    for _ in range(args.warmup):
        S.select(p, mode, 0, w.n_tokens, dev[1], buf, stream)
    torch.cuda.synchronize()
    times = []
    for _ in range(args.steps):
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        S.select(p, mode, 0, w.n_tokens, dev[1], buf, stream)
        e1.record(stream)
        torch.cuda.synchronize()
        times.append(e0.elapsed_time(e1))
    st = S.scale_get_device_status(buf.ws)
    if st != S.SCALE_OK:
        raise RuntimeError(f"device status {st}: {S.status_string(st)}")
    n = w.n_subchunks if mode == S.SCALE_MODE_PER_SUBCHUNK else int(buf.n_units.item())
    line = {"metric": "selection (steps (b)-(c)) time per call", "stage": "select", "unit": "us",
            "value": statistics.median(times) * 1e3, "min": min(times) * 1e3, "steps": args.steps,
            "warmup": args.warmup, "units": n, "config": workload_config(w, args.mode), "data": "synthetic",
            "higher_is_better": False}
    print(json.dumps(line), flush=True)
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.stage:
        return run_stage(args)
    if args.sweep:
        return run_sweep(args)
    if args.decode:
        return run_decode(args)
    if workload(args.workload).layers > 1:
        return run_stack(args)
    return run_scale(args)


if __name__ == "__main__":
    sys.exit(main())
