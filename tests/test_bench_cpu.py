"""CPU checks of bench.py's bookkeeping: the attention kernel's ncu counters
are read from the committed sidecar of the same workload only while the
kernel source is unchanged, the launch counts follow the path's kernels, the
Algorithm 2 loop issues one selection and attention call per unit, and the
selection agreement counts near-ties apart from mismatches."""

import json
import os
import sys

import numpy as np

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from synth import workload  # noqa: E402


def test_profile_counters_follow_the_kernel_code(tmp_path, monkeypatch):
    src = tmp_path / "attn.cu"
    src.write_text("// kernel\nint v = 1;  // one\n")
    (tmp_path / "attn_wl-a_ncu.json").write_text(json.dumps(
        {"kernel_code_sha16": bench.kernel_source_hash(str(src)), "traffic_bytes_per_launch": 12345,
         "tensor_pipe_active_pct": 70.0}))
    monkeypatch.setattr(bench, "KERNEL_SRC", str(src))
    monkeypatch.setattr(bench, "PROFILE_DIR", str(tmp_path))
    assert bench.profile_counters("wl-a")["traffic_bytes_per_launch"] == 12345
    assert bench.profile_counters("wl-b") == {}  # no capture of that workload
    src.write_text("/* the kernel */\n\nint v = 1;  // first\n")  # comments only: same code
    assert bench.profile_counters("wl-a")["tensor_pipe_active_pct"] == 70.0
    src.write_text("// kernel\nint v = 2;  // one\n")  # the code changed since the capture
    assert bench.profile_counters("wl-a") == {}


def test_committed_sidecars_are_valid_json():
    d = os.path.join(ROOT, "profiles")
    for name in os.listdir(d):
        if name.endswith(".json"):
            with open(os.path.join(d, name)) as f:
                rec = json.load(f)
            assert len(rec["kernel_code_sha16"]) == 16


def test_algorithm2_loop_calls():
    w = workload("llama8b-128k")
    scr = bench.loop_calls(w, False)
    assert len(scr) == 8 and all(len(u) == 1 for _, u in scr)  # one cluster per outer chunk
    assert scr[0] == ((0, 16384), [(0, 16384)])
    sub = bench.loop_calls(w, True)
    assert len(sub) == 8 and sum(len(u) for _, u in sub) == 64  # one call per sub-chunk
    assert sub[1][1][0] == (16384, 18432)
    ragged = bench.loop_calls(workload("gqa4-4k", n_tokens=3000), True)
    assert ragged[-1][1][-1] == (2816, 3000)  # last sub-chunk ends at N


def test_selection_agreement_counts():
    w = workload("gqa4-4k")
    ref = {"sel": np.array([[1, 2], [3, 4], [5, 6]]), "sel_count": np.array([2, 2, 2]),
           "gap": np.array([0.5, 1e-4, 0.5])}
    gpu = np.array([[1, 2], [3, 7], [5, 6]])
    a = bench.selection_agreement(w, ref, gpu, np.array([2, 2, 2]))
    assert (a["selection_match_units"], a["near_tie_units"], a["selection_mismatch_units"]) == (2, 1, 0)
    gpu[2, 1] = 9
    a = bench.selection_agreement(w, ref, gpu, np.array([2, 2, 2]))
    assert a["selection_mismatch_units"] == 1


def test_launch_counts():
    # step (a): k_block_reps, k_fingerprint, k_cluster (+ k_gram when clusters have > 1 sub-chunk);
    # selection: k_logits + k_select_fused (up to 4096 blocks); attention: k_sparse_attn
    assert bench.launches(workload("llama8b-128k"))["total"] == 7   # 4 + 2 + 1
    assert bench.launches(workload("gqa4-4k", max_cluster_subchunks=1))["total"] == 6
    # more than 4096 blocks: k_logits, k_stats, k_vote, k_topk
    assert bench.launches(workload("llama8b-1m", block_size=128))["total"] == 4 + 4 + 1
    # token level: split, two scoring passes and their merge, then the multi-CTA top-k
    # (init, 4 histogram passes, count, scan, emit)
    assert bench.launches(workload("llama8b-128k-tok"))["total"] == 3 + 4 + 8 + 3
    assert bench.launches(workload("llama8b-32k", block_size=1, top_k=1024))["total"] == 3 + 5 + 3
    # the 1M-token step of Algorithm 2: 16 outer chunks, one unit each (the ncu launch list of that step
    # counted 288 launches of the library's kernels)
    w = workload("llama8b-1m-tok")
    chunks = w.n_tokens // w.outer_chunk
    assert bench.launches(w, chunks, chunks)["total"] == 288
    assert bench.launches(workload("llama8b-64k-32l"), 8)["total"] == 4 + 8 * 3
    assert bench.launches(workload("llama8b-64k-32l"), 8, 8)["total"] == 8 * 4 + 8 * 3  # per-chunk step (a)


def test_other_configs_compacts_each_side_run(monkeypatch):
    """The side runs of the other configs: one process per workload; a layer's
    line (with both modes and the selection check) and a stack's line (no
    batched form) are compacted, a failed run is reported, not raised."""
    import subprocess

    layer = {"config": {"n_tokens": 32768}, "steps": 3, "warmup": 3, "ms_per_step": 6.0, "value": 5.4e6,
             "roofline": {"achieved": 1500.0, "frac": 0.78}, "stages_ms": {"select": 1.1},
             "retrieval_calls": 3, "units": 4, "batched": {"ms_per_step": 2.7},
             "other_mode": {"ms_per_step": 5.0, "tokens_per_s": 6.5e6, "attn_tflops": 1300.0,
                            "stages_ms": {"select": 3.0}, "retrieval_calls": 30, "units": 32,
                            "batched": {"ms_per_step": 2.0}},
             "scr_over_subchunk": 1.2, "attn_flops_ratio": 1.5, "clocks": {"sm_mhz": 2000.0},
             "selection_match_units": 4, "near_tie_units": 0, "selection_mismatch_units": 0}
    stack = {"config": {"n_tokens": 65536, "layers": 32}, "steps": 3, "warmup": 3, "ms_per_step": 200.0,
             "value": 3.3e5, "roofline": {"achieved": 1600.0, "frac": 0.83}, "retrieval_calls": 224,
             "units": 256, "other_mode": {"ms_per_step": 230.0, "tokens_per_s": 2.8e5, "attn_tflops": 1400.0,
                                          "retrieval_calls": 1984, "units": 2048},
             "scr_over_subchunk": 0.87, "attn_flops_ratio": 1.58, "clocks": None}
    calls = []

    def fake_run(cmd, **kw):
        name = cmd[cmd.index("--workload") + 1]
        calls.append(cmd)
        if name == "llama8b-1m":
            return subprocess.CompletedProcess(cmd, 1, "", "RuntimeError: boom\n")
        out = stack if name == "llama8b-64k-32l" else layer
        return subprocess.CompletedProcess(cmd, 0, "log line\n" + json.dumps(out) + "\n", "")

    monkeypatch.setattr(subprocess, "run", fake_run)
    got = bench.other_configs()
    assert [c[c.index("--workload") + 1] for c in calls] == [n for n, _ in bench.OTHER_CONFIGS]
    assert all("--no-other-configs" in c for c in calls)
    assert ("--selection-check" in calls[2]) is False  # the stack runs no oracle check
    assert ("--selection-check" in calls[-1]) is False  # nor 1M tokens at token level
    l32 = got["llama8b-32k"]
    assert l32["cluster"]["ttft_ms"] == 6.0 and l32["subchunk"]["ttft_ms"] == 5.0
    assert l32["cluster"]["batched_ms"] == 2.7 and l32["subchunk"]["select_ms"] == 3.0
    assert l32["selection"]["selection_mismatch_units"] == 0
    st = got["llama8b-64k-32l"]
    assert st["layers"] == 32 and st["cluster"]["batched_ms"] is None and "selection" not in st
    assert got["llama8b-1m"] == {"error": "RuntimeError: boom", "rc": 1}
