"""CPU checks of bench.py's bookkeeping: the per-launch DRAM traffic is read
from the committed ncu summary only while the kernel source is unchanged, and
the launch counts follow the path's kernels."""

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
    summary = tmp_path / "summary.md"
    summary.write_text(f"# title\n\n- attn.cu sha256[:16]: {sha}\n- traffic bytes per full launch: 12345\n")
    monkeypatch.setattr(bench, "KERNEL_SRC", str(src))
    monkeypatch.setattr(bench, "PROFILE_SUMMARY", str(summary))
    assert bench.profile_traffic() == 12345.0
    src.write_bytes(b"// kernel v2\n")  # changed since the capture
    assert bench.profile_traffic() is None


def test_launch_counts():
    assert bench.launches(workload("llama8b-128k"))["total"] == 10   # 5 + 4 + 1
    assert bench.launches(workload("gqa4-4k", max_cluster_subchunks=1))["total"] == 9
    assert bench.launches(workload("llama8b-128k-tok"))["total"] == 4 + 16 + 3  # multi-CTA top-k
    assert bench.launches(workload("llama8b-32k", block_size=1, top_k=1024))["total"] == 4 + 5 + 3
    assert bench.launches(workload("llama8b-64k-32l"), 8)["total"] == 5 + 8 * 5
