#!/usr/bin/env python
"""Benchmark of the Similarity Chunk Rolling sparse-prefill path on GB300.

One step = steps (a)-(d) of the path over one layer of the workload: block
representatives + fingerprints + anchor clusters, cluster-level selection,
block-sparse causal attention. Inputs are resident in HBM before timing; they
are larger than L2 (Q, K, V of the 128K workload are 1.6 GB).

Prints one JSON line (rank 0). ``--impl reference`` times the CPU fp64 oracle
instead, on a bounded sample of the same workload.
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
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-chunk-loop", action="store_true",
                    help="skip timing the per-outer-chunk loop of range calls alongside")
    ap.add_argument("--no-baseline-mode", action="store_true",
                    help="skip timing the per-sub-chunk selection mode alongside")
    ap.add_argument("--cpu-seconds", type=float, default=12.0,
                    help="target CPU time of the oracle sample")
    ap.add_argument("--paged", type=int, default=0, metavar="P",
                    help="keep K and V in a paged cache of P-token pages (shuffled page order)")
    ap.add_argument("--decode", action="store_true",
                    help="decode steps with the selection cache at the end of the context (one JSON line)")
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
    # the top-k is one kernel, or 12 (init, 4 x (histogram, pick), count, scan,
    # emit) for units of more than 64K candidates
    topk = 12 if tok and w.n_blocks > 65536 else 1
    select = (4 if tok else 3) + topk
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


def profile_traffic(workload_name: str):
    """Per-launch DRAM bytes of the attention kernel on this workload from the
    committed ncu summary (profiles/attn_<workload>_ncu.md), or None when there
    is none or the kernel source changed since the capture."""
    summary = os.path.join(PROFILE_DIR, f"attn_{workload_name}_ncu.md")
    if not os.path.exists(summary):
        return None
    with open(KERNEL_SRC, "rb") as f:
        sha = hashlib.sha256(f.read()).hexdigest()[:16]
    vals = {}
    with open(summary) as f:
        for line in f:
            if ": " in line and line.strip().startswith("- "):
                k, v = line.strip()[2:].split(": ", 1)  # keys may hold a colon ("sha256[:16]")
                vals[k.strip()] = v.strip()
    if vals.get("attn.cu sha256[:16]") != sha:
        return None
    try:
        return float(vals["traffic bytes per full launch"])
    except (KeyError, ValueError):
        return None


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


def oracle_sample(w, q, k, v, per_subchunk, cpu_seconds, rows_first=32):
    """Time the oracle on a bounded sample: steps (a)-(c) over the whole layer,
    step (d) on a growing set of seeded rows until about cpu_seconds; the
    throughput is extrapolated from the per-row time to all rows."""
    import oracle

    t0 = time.perf_counter()
    ref = oracle.run_path(w, q, k, v, per_subchunk=per_subchunk)
    t_abc = time.perf_counter() - t0
    rng = np.random.default_rng(7)
    n_rows, t_d, done = rows_first, 0.0, 0
    while True:
        rows = np.sort(rng.integers(0, w.n_tokens, size=n_rows))
        t1 = time.perf_counter()
        oracle.attention_rows(q=q, k=k, v=v, sub_chunk=w.sub_chunk, block_size=w.block_size,
                              top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                              attn_scale=1.0 / np.sqrt(w.head_dim), per_subchunk=per_subchunk,
                              unit_start=ref["unit_start"], sel=ref["sel"],
                              sel_count=ref["sel_count"], rows=rows)
        t_d += time.perf_counter() - t1
        done += n_rows
        if t_abc + t_d >= cpu_seconds or done >= w.n_tokens:
            break
        n_rows = min(w.n_tokens, max(n_rows, int(n_rows * max(1.5, (cpu_seconds - t_abc) / max(t_d, 1e-3) * 0.6))))
    t_full = t_abc + t_d / done * w.n_tokens
    cores = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else os.cpu_count()
    omp = os.environ.get("OMP_NUM_THREADS")
    return dict(tokens_per_s=w.n_tokens / t_full, t_full=t_full, t_abc=t_abc, t_d=t_d, rows=done,
                cores=int(omp) if omp else cores)


# --------------------------------------------------------------------------- arms


def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def run_reference(args):
    world, rank, local = dist_setup(args)
    if rank != 0:
        return 0
    w = workload(args.workload)
    per_sub = args.mode == "subchunk"
    q, k, v = generate_layer(w)
    times, last = [], None
    for i in range(args.warmup + args.steps):
        r = oracle_sample(w, q, k, v, per_sub, cpu_seconds=max(1.0, args.cpu_seconds / 4), rows_first=16)
        if i >= args.warmup:
            times.append(r["t_full"])
            last = r
    t = statistics.mean(times)
    value = w.n_tokens / t
    sample = (f"per step: steps (a)-(c) over all {w.n_tokens} tokens ({last['t_abc']:.2f} s) + "
              f"Eq. 10 on {last['rows']} seeded rows ({last['t_d']:.2f} s), extrapolated per row")
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
        "n_gpus": 1, "steps": args.steps, "warmup": args.warmup, "ms_per_step": t * 1e3,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": w.name, "n_tokens": w.n_tokens, "mode": args.mode, "theta": w.theta},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": last["cores"], "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


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
    buf = pkg.allocate(p, mode)
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

    def timed(mode_, steps, warmup, buf_):
        ev = [[torch.cuda.Event(enable_timing=True) for _ in range(4)] for _ in range(steps)]
        for _ in range(warmup):
            pkg.run_path(p, mode_, *dev, buf_)
        torch.cuda.synchronize()
        barrier()
        torch.cuda.synchronize()
        clocks = ClockSampler(torch.cuda.current_device())
        clocks.start()
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for i in range(steps):
            e = ev[i]
            e[0].record(stream)
            if kv is not None:
                S.scale_build_reps_paged(p, dev[0], kv, buf_.reps, buf_.fingerprints, buf_.unit_start,
                                         buf_.n_units, buf_.ws, stream)
            else:
                S.scale_build_reps(p, dev[0], dev[1], buf_.reps, buf_.fingerprints, buf_.unit_start,
                                   buf_.n_units, buf_.ws, stream)
            e[1].record(stream)
            if kv is not None and w.block_size == 1:
                S.scale_select_tokens_paged(p, mode_, 0, w.n_tokens, kv, buf_.fingerprints, buf_.unit_start,
                                            buf_.n_units, buf_.sel_blocks, buf_.sel_count, None, buf_.ws,
                                            stream)
            else:
                S.select(p, mode_, 0, w.n_tokens, dev[1], buf_, stream)
            e[2].record(stream)
            if kv is not None:
                S.scale_sparse_prefill_paged(p, mode_, 0, w.n_tokens, dev[0], kv, buf_.unit_start,
                                             buf_.n_units, buf_.sel_blocks, buf_.sel_count, buf_.out,
                                             buf_.ws, stream)
            else:
                S.scale_sparse_prefill(p, mode_, 0, w.n_tokens, *dev, buf_.unit_start, buf_.n_units,
                                       buf_.sel_blocks, buf_.sel_count, buf_.out, buf_.ws, stream)
            e[3].record(stream)
        end.record(stream)
        torch.cuda.synchronize()
        clk = clocks.stop()
        barrier()
        total = start.elapsed_time(end) / steps
        stages = [statistics.mean(x[j].elapsed_time(x[j + 1]) for x in ev) for j in range(3)]
        st = S.scale_get_device_status(buf_.ws)
        if st != S.SCALE_OK:
            raise RuntimeError(f"device status {st}: {S.status_string(st)}")
        return total, stages, clk

    ms, stages, clk = timed(mode, args.steps, args.warmup, buf)
    if world > 1:
        t = torch.tensor([ms], device="cuda")
        torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
        ms = float(t.item())

    n_units = w.n_subchunks if per_sub else int(buf.n_units.item())
    us = buf.unit_start.cpu().numpy()
    sel = buf.sel_blocks.cpu().numpy()
    cnt = buf.sel_count.cpu().numpy()
    keys = key_counts(w, us, n_units, sel, cnt, per_sub)
    flops = 4.0 * w.head_dim * w.num_q_heads * keys
    peaks = load_peaks()
    attn_s = stages[2] / 1e3
    achieved = flops / attn_s / 1e12
    _, calls = S.scale_retrieval_calls(p, mode, us[: n_units + 1] if not per_sub else None, n_units)

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
        "config": {"workload": w.name, "n_tokens": w.n_tokens, "q_heads": w.num_q_heads,
                   "kv_heads": w.num_kv_heads, "head_dim": w.head_dim, "sub_chunk": w.sub_chunk,
                   "max_cluster_subchunks": w.max_cluster_subchunks, "block_size": w.block_size,
                   "top_k": w.top_k, "n_sink": w.n_sink, "n_local": w.n_local, "theta": w.theta,
                   "mode": args.mode, "parallelism": f"independent layers x{world}",
                   "kv_layout": f"paged, {args.paged}-token pages" if args.paged else "contiguous",
                   "l2": "inputs larger than L2 (Q+K+V %.2f GB)" % ((q.nbytes + k.nbytes + v.nbytes) / 1e9)},
        "stages_ms": {"build_reps": stages[0], "select": stages[1], "sparse_attention": stages[2]},
        "retrieval_calls": calls,
        "units": n_units,
        "roofline": {"bound": "tensor", "kernel": "k_sparse_attn", "achieved": achieved,
                     "peak": peaks["bf16_sustained"], "unit": "TFLOP/s",
                     "frac": achieved / peaks["bf16_sustained"],
                     "frac_of_burst": achieved / peaks["bf16"],
                     "peak_source": f"bf16 sustained, of {peaks['source']}",
                     "algorithmic_flops_per_launch": flops, "traffic": profile_traffic(w.name)},
        "gpu_launches": args.steps * launches(w)["total"],
        "clocks": clk,
    }

    if not args.no_baseline_mode and rank == 0:
        other = S.SCALE_MODE_PER_SUBCHUNK if not per_sub else S.SCALE_MODE_PER_CLUSTER
        buf2 = pkg.allocate(p, other)
        ms2, st2, _ = timed(other, max(3, args.steps // 2), 2, buf2)
        n2 = w.n_subchunks if other == S.SCALE_MODE_PER_SUBCHUNK else int(buf2.n_units.item())
        us2 = buf2.unit_start.cpu().numpy()
        _, calls2 = S.scale_retrieval_calls(
            p, other, us2[: n2 + 1] if other == S.SCALE_MODE_PER_CLUSTER else None, n2)
        line["other_mode"] = {"mode": "subchunk" if other == S.SCALE_MODE_PER_SUBCHUNK else "cluster",
                              "ms_per_step": ms2, "tokens_per_s": w.n_tokens / (ms2 / 1e3),
                              "stages_ms": {"build_reps": st2[0], "select": st2[1], "sparse_attention": st2[2]},
                              "retrieval_calls": calls2, "units": n2}
        del buf2

    if not args.no_chunk_loop and rank == 0:
        # Chunked prefill as Algorithm 2 orders it: per outer chunk, step (a)
        # over the chunk's range, then its selection and attention.
        chunks = [(t0, min(w.n_tokens, t0 + w.outer_chunk)) for t0 in range(0, w.n_tokens, w.outer_chunk)]

        def chunk_step():
            for t0, t1 in chunks:
                if kv is not None:
                    S.scale_build_reps_range_paged(p, t0, t1, dev[0], kv, buf.reps, buf.fingerprints,
                                                   buf.unit_start, buf.n_units, buf.ws, stream)
                    if w.block_size == 1:
                        S.scale_select_tokens_paged(p, mode, t0, t1, kv, buf.fingerprints, buf.unit_start,
                                                    buf.n_units, buf.sel_blocks, buf.sel_count, None, buf.ws,
                                                    stream)
                    else:
                        S.select(p, mode, t0, t1, None, buf, stream)
                    S.scale_sparse_prefill_paged(p, mode, t0, t1, dev[0], kv, buf.unit_start, buf.n_units,
                                                 buf.sel_blocks, buf.sel_count, buf.out, buf.ws, stream)
                else:
                    S.scale_build_reps_range(p, t0, t1, dev[0], dev[1], buf.reps, buf.fingerprints,
                                             buf.unit_start, buf.n_units, buf.ws, stream)
                    S.select(p, mode, t0, t1, dev[1], buf, stream)
                    S.scale_sparse_prefill(p, mode, t0, t1, *dev, buf.unit_start, buf.n_units,
                                           buf.sel_blocks, buf.sel_count, buf.out, buf.ws, stream)

        for _ in range(2):
            chunk_step()
        torch.cuda.synchronize()
        c_steps = max(3, args.steps // 2)
        start, end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        start.record(stream)
        for _ in range(c_steps):
            chunk_step()
        end.record(stream)
        torch.cuda.synchronize()
        st = S.scale_get_device_status(buf.ws)
        if st != S.SCALE_OK:
            raise RuntimeError(f"device status {st}: {S.status_string(st)}")
        ms_c = start.elapsed_time(end) / c_steps
        line["chunk_loop"] = {"ms_per_step": ms_c, "tokens_per_s": w.n_tokens / (ms_c / 1e3),
                              "outer_chunks": len(chunks),
                              "calls_per_step": 3 * len(chunks),
                              "kernel_launches_per_step": launches(w, len(chunks), len(chunks))["total"],
                              "loop": "per outer chunk: scale_build_reps_range, select, scale_sparse_prefill"}

    if not args.no_e2e:
        qh, kh, vh = (torch.from_numpy(x).pin_memory() for x in (q, k, v))
        oh = torch.empty(qh.shape, dtype=torch.int16).pin_memory()
        arena = torch.empty(S.scale_prefill_host_arena_size(p, mode), dtype=torch.uint8, device="cuda")
        S.scale_prefill_host(p, mode, qh, kh, vh, oh, arena, stream)
        reps = max(3, args.steps // 4)
        link = host_link_gbs(qh, arena, stream)
        torch.cuda.synchronize()
        barrier()
        per_call = []
        for _ in range(reps):
            t0 = time.perf_counter()
            S.scale_prefill_host(p, mode, qh, kh, vh, oh, arena, stream)
            per_call.append(time.perf_counter() - t0)
        t_e2e = sum(per_call) / reps
        if world > 1:
            t = torch.tensor([t_e2e], device="cuda")
            torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
            t_e2e = float(t.item())
        line["e2e"] = {"value": world * w.n_tokens / t_e2e, "unit": "tokens/s",
                       "h2d_bytes_per_step": int(q.nbytes + k.nbytes + v.nbytes),
                       "d2h_bytes_per_step": int(q.nbytes), "ms_per_step": t_e2e * 1e3,
                       "ms_min": min(per_call) * 1e3, "ms_median": statistics.median(per_call) * 1e3,
                       "host_link_gbs": link,
                       "api": "scale_prefill_host (pinned host buffers)"}
        del arena

    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        r = oracle_sample(w, q, k, v, per_sub, args.cpu_seconds)
        line["cpu_baseline"] = {
            "value": r["tokens_per_s"], "unit": "tokens/s", "cores": r["cores"], "kind": "oracle",
            "sample": (f"steps (a)-(c) over all {w.n_tokens} tokens ({r['t_abc']:.2f} s) + Eq. 10 on "
                       f"{r['rows']} seeded rows ({r['t_d']:.2f} s), time per row extrapolated to all rows")}

    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


SWEEP_WORKLOAD = "llama8b-128k-topics"
SWEEP_THETAS = (0.95, 0.97, 0.99)
SWEEP_SMAX = (2, 4, 8)


def cosine_stats(fp: np.ndarray) -> dict:
    """Distribution of cos(v_i, v_{i+1}) over consecutive sub-chunks (the paper's Table 1 format)."""
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
    chunks = [(t0, min(w.n_tokens, t0 + w.outer_chunk)) for t0 in range(0, w.n_tokens, w.outer_chunk)]

    def measure(mode, steps, warmup):
        bufs = [pkg.allocate(p, mode) for _ in layers]
        n_attn = len(chunks) * len(layers)

        def step(ev=None):
            i = 0
            for t0, t1 in chunks:
                for dev, b in zip(layers, bufs):
                    S.scale_build_reps_range(p, t0, t1, dev[0], dev[1], b.reps, b.fingerprints, b.unit_start,
                                             b.n_units, b.ws, stream)
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
        return ms, attn_ms, clk, 4.0 * w.head_dim * w.num_q_heads * keys, calls, units

    mode = S.SCALE_MODE_PER_SUBCHUNK if args.mode == "subchunk" else S.SCALE_MODE_PER_CLUSTER
    ms, attn_ms, clk, flops, calls, units = measure(mode, args.steps, args.warmup)
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
                   "outer_chunk": w.outer_chunk, "loop": "chunk-major: every layer per outer chunk",
                   "parallelism": f"independent stacks x{world}", "l2": "inputs larger than L2"},
        "stages_ms": {"sparse_attention_total": attn_ms, "other": ms - attn_ms},
        "retrieval_calls": calls, "units": units,
        "roofline": {"bound": "tensor", "kernel": "k_sparse_attn", "achieved": achieved,
                     "peak": peaks["bf16_sustained"], "unit": "TFLOP/s",
                     "frac": achieved / peaks["bf16_sustained"], "frac_of_burst": achieved / peaks["bf16"],
                     "peak_source": f"bf16 sustained, of {peaks['source']}",
                     "algorithmic_flops_per_step": flops, "traffic": None},
        "gpu_launches": args.steps * w.layers * launches(w, len(chunks), len(chunks))["total"],
        "clocks": clk,
    }
    if not args.no_baseline_mode and rank == 0:
        other = S.SCALE_MODE_PER_SUBCHUNK if mode == S.SCALE_MODE_PER_CLUSTER else S.SCALE_MODE_PER_CLUSTER
        ms2, attn2, _, flops2, calls2, units2 = measure(other, max(2, args.steps // 2), 1)
        line["other_mode"] = {"mode": "subchunk" if other == S.SCALE_MODE_PER_SUBCHUNK else "cluster",
                              "ms_per_step": ms2, "tokens_per_s": w.n_tokens / (ms2 / 1e3),
                              "sparse_attention_ms": attn2, "retrieval_calls": calls2, "units": units2,
                              "attn_tflops": flops2 / (attn2 / 1e3) / 1e12}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.destroy_process_group()
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    if args.decode:
        return run_decode(args)
    if workload(args.workload).layers > 1:
        return run_stack(args)
    return run_scale(args)


if __name__ == "__main__":
    sys.exit(main())
