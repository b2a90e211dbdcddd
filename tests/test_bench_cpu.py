"""CPU checks of bench.py's bookkeeping: the per-launch DRAM traffic is read
from the committed ncu summary of the same workload only while the kernel
source is unchanged, and the launch counts follow the path's kernels."""

import hashlib
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402
from synth import workload  # noqa: E402


def test_profile_traffic_follows_the_kernel_source(tmp_path, monkeypatch):
    src = tmp_path / "attn.cu"
    src.write_bytes(b"// kernel v1\n")
    sha = hashlib.sha256(src.read_bytes()).hexdigest()[:16]
    summary = tmp_path / "attn_wl-a_ncu.md"
    summary.write_text(f"# title\n\n- attn.cu sha256[:16]: {sha}\n- traffic bytes per full launch: 12345\n")
    monkeypatch.setattr(bench, "KERNEL_SRC", str(src))
    monkeypatch.setattr(bench, "PROFILE_DIR", str(tmp_path))
    assert bench.profile_traffic("wl-a") == 12345.0
    assert bench.profile_traffic("wl-b") is None  # no capture of that workload
    src.write_bytes(b"// kernel v2\n")  # changed since the capture
    assert bench.profile_traffic("wl-a") is None


def test_launch_counts():
    # step (a): k_block_reps, k_fingerprint, k_cluster (+ k_gram when clusters have > 1 sub-chunk)
    assert bench.launches(workload("llama8b-128k"))["total"] == 9   # 4 + 4 + 1
    assert bench.launches(workload("gqa4-4k", max_cluster_subchunks=1))["total"] == 8
    assert bench.launches(workload("llama8b-128k-tok"))["total"] == 3 + 16 + 3  # multi-CTA top-k
    assert bench.launches(workload("llama8b-32k", block_size=1, top_k=1024))["total"] == 3 + 5 + 3
    assert bench.launches(workload("llama8b-64k-32l"), 8)["total"] == 4 + 8 * 5
    assert bench.launches(workload("llama8b-64k-32l"), 8, 8)["total"] == 8 * 4 + 8 * 5  # per-chunk step (a)
