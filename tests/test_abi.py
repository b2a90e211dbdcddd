"""CPU checks of the C ABI: the library builds and loads, exports every symbol
include/scale.h declares, its struct layout matches the binding, and its
host-only entry points validate arguments and count retrieval calls. No
kernel is launched here."""

import ctypes
import os
import subprocess
import tempfile

import numpy as np
import pytest

import paper_2609_31568_gb300 as pkg
from paper_2609_31568_gb300 import scale as S
from synth import workload

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    pkg.build()
    return S.load()


def test_every_declared_symbol_is_exported(lib):
    names = S.declared_functions()
    assert len(names) >= 12
    missing = [n for n in names if not hasattr(lib, n)]
    assert not missing


def test_wait_limit_entry_points_validate(lib):
    """A wait limit of 0 is refused and the default is accepted; the wait
    self-check refuses a missing workspace before launching anything."""
    assert lib.scale_set_wait_timeout_ns(0) == S.SCALE_ERR_INVALID_ARG
    assert lib.scale_set_wait_timeout_ns(4_000_000_000) == S.SCALE_OK  # the default
    assert lib.scale_selftest_wait_timeout(None, 0, 1_000_000, None) == S.SCALE_ERR_INVALID_ARG


def test_params_struct_layout_matches_header():
    src = r"""
#include <stddef.h>
#include <stdio.h>
#include "scale.h"
#define F(x) printf(#x " %zu\n", offsetof(scale_params_t, x));
int main(void) {
  printf("size %zu\n", sizeof(scale_params_t));
  F(num_q_heads) F(num_kv_heads) F(head_dim) F(sub_chunk) F(n_tokens) F(max_cluster_subchunks)
  F(outer_chunk) F(theta) F(block_size) F(top_k) F(n_sink) F(n_local) F(select_scale) F(attn_scale)
  return 0;
}
"""
    with tempfile.TemporaryDirectory() as d:
        c = os.path.join(d, "t.c")
        exe = os.path.join(d, "t")
        with open(c, "w") as f:
            f.write(src)
        subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), c, "-o", exe], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout
    got = dict(line.split() for line in out.strip().splitlines())
    assert int(got.pop("size")) == ctypes.sizeof(S.ScaleParams)
    for name, off in got.items():
        assert getattr(S.ScaleParams, name).offset == int(off), name


def test_status_strings_and_version(lib):
    assert S.scale_version() >= 10000
    for rc in (0, -1, -2, -3, -4, -5, -6):
        assert S.status_string(rc) != "unknown status"


def _p(**over):
    return S.params_for(workload("llama8b-32k"), **over)


@pytest.mark.parametrize("over,rc", [
    (dict(head_dim=64), S.SCALE_ERR_UNSUPPORTED),
    (dict(num_kv_heads=3), S.SCALE_ERR_INVALID_ARG),
    (dict(num_q_heads=0), S.SCALE_ERR_INVALID_ARG),
    (dict(n_tokens=0), S.SCALE_ERR_INVALID_ARG),
    (dict(n_tokens=1 << 31), S.SCALE_ERR_UNSUPPORTED),
    (dict(sub_chunk=0), S.SCALE_ERR_INVALID_ARG),
    (dict(outer_chunk=1000), S.SCALE_ERR_INVALID_ARG),
    (dict(block_size=0), S.SCALE_ERR_INVALID_ARG),
    (dict(top_k=-1), S.SCALE_ERR_INVALID_ARG),
    (dict(n_sink=-1), S.SCALE_ERR_INVALID_ARG),
    (dict(theta=float("nan")), S.SCALE_ERR_INVALID_ARG),
    (dict(attn_scale=-1.0), S.SCALE_ERR_INVALID_ARG),
    (dict(select_scale=float("inf")), S.SCALE_ERR_INVALID_ARG),
])
def test_parameter_validation(lib, over, rc):
    with pytest.raises(S.ScaleError) as e:
        S.scale_workspace_size(_p(**over), S.SCALE_MODE_PER_CLUSTER)
    assert e.value.rc == rc


def test_null_pointers_rejected_without_launch(lib):
    p = _p()
    assert lib.scale_build_reps(ctypes.byref(p), None, None, None, None, None, None, None, 0, None) \
        == S.SCALE_ERR_INVALID_ARG
    assert lib.scale_select(ctypes.byref(p), 0, 0, p.n_tokens, None, None, None, None, None, None,
                            None, None, 0, None) == S.SCALE_ERR_INVALID_ARG
    assert lib.scale_sparse_prefill(ctypes.byref(p), 1, 0, p.n_tokens, None, None, None, None, None,
                                    None, None, None, None, 0, None) == S.SCALE_ERR_INVALID_ARG
    assert lib.scale_select(ctypes.byref(p), 7, 0, p.n_tokens, None, None, None, None, None, None,
                            None, None, 0, None) == S.SCALE_ERR_INVALID_ARG


def test_workspace_grows_with_problem(lib):
    small = S.scale_workspace_size(S.params_for(workload("gqa4-4k")), 0)
    big = S.scale_workspace_size(S.params_for(workload("llama8b-1m")), 0)
    assert 0 < small < big < (1 << 30)


def _golden():
    rows = {}
    with open(os.path.join(ROOT, "tests", "golden", "retrieval_calls.txt")) as f:
        for line in f:
            if line.strip() and not line.startswith("#"):
                n, su, sc, bu, bc = line.split()
                rows[n] = tuple(map(int, (su, sc, bu, bc)))
    return rows


@pytest.mark.parametrize("name", sorted(_golden()))
def test_retrieval_call_count_matches_closed_form(lib, name):
    w = workload(name)
    su, sc, bu, bc = _golden()[name]
    p = S.params_for(w)
    assert S.scale_retrieval_calls(p, S.SCALE_MODE_PER_SUBCHUNK, None, 0) == (bu, bc)
    # fixed-size clusters (theta = -1): anchors every S_max sub-chunks in each outer chunk
    per = w.outer_chunk // w.sub_chunk
    starts = [c + i for c in range(0, w.n_subchunks, per)
              for i in range(0, min(per, w.n_subchunks - c), w.max_cluster_subchunks)]
    assert S.scale_retrieval_calls(p, S.SCALE_MODE_PER_CLUSTER, np.array(starts), len(starts)) == (su, sc)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    monkeypatch.setattr(S, "LIB_PATH", str(tmp_path / "nope.so"))
    monkeypatch.setattr(S, "_lib", None)
    with pytest.raises(S.ScaleLibraryMissing):
        S.load()


def test_block_and_token_selection_entry_points_check_block_size(lib):
    """scale_select serves block sizes > 1, scale_select_tokens block size 1;
    each refuses the other before looking at any pointer."""
    p1 = S.params_for(workload("llama8b-32k", block_size=1, top_k=1024))
    assert lib.scale_select(ctypes.byref(p1), 0, 0, p1.n_tokens, None, None, None, None, None, None,
                            None, None, 0, None) == S.SCALE_ERR_UNSUPPORTED
    pb = _p()
    assert lib.scale_select_tokens(ctypes.byref(pb), 0, 0, pb.n_tokens, None, None, None, None, None,
                                   None, None, None, 0, None) == S.SCALE_ERR_INVALID_ARG
    p16 = S.params_for(workload("llama8b-32k", block_size=1, num_kv_heads=2))  # 16 query heads per KV head
    assert lib.scale_select_tokens(ctypes.byref(p16), 0, 0, p16.n_tokens, None, None, None, None, None,
                                   None, None, None, 0, None) == S.SCALE_ERR_UNSUPPORTED


def test_token_workspace_has_no_logits_plane():
    """Block size 1 keeps no [units][heads][tokens] logits (that would be 32 GB
    at 1M tokens per sub-chunk): the workspace is the [units][tokens] scores
    plus the packed distant keys and values of every unit, plus small parts."""
    w = workload("llama8b-1m-tok")
    p = S.params_for(w)
    n = S.scale_workspace_size(p, S.SCALE_MODE_PER_SUBCHUNK)
    M, N = w.n_subchunks, w.n_tokens
    slots = -(-(w.n_sink + w.top_k) // 128) * 128
    big = M * N * 4 + 2 * M * w.num_kv_heads * slots * 128 * 2
    assert big <= n < big * 1.1
    assert n < M * w.num_q_heads * N * 4  # the logits plane alone would be larger


def test_kv_pages_struct_layout_matches_header():
    src = r"""
#include <stddef.h>
#include <stdio.h>
#include "scale.h"
#define F(x) printf(#x " %zu\n", offsetof(scale_kv_pages_t, x));
int main(void) {
  printf("size %zu\n", sizeof(scale_kv_pages_t));
  F(k_pages) F(v_pages) F(page_table) F(page_size) F(num_pages)
  return 0;
}
"""
    with tempfile.TemporaryDirectory() as d:
        c = os.path.join(d, "t.c")
        exe = os.path.join(d, "t")
        with open(c, "w") as f:
            f.write(src)
        subprocess.run(["gcc", "-I", os.path.join(ROOT, "include"), c, "-o", exe], check=True)
        out = subprocess.run([exe], capture_output=True, text=True, check=True).stdout
    got = dict(line.split() for line in out.strip().splitlines())
    assert int(got.pop("size")) == ctypes.sizeof(S.ScaleKvPages)
    for name, off in got.items():
        assert getattr(S.ScaleKvPages, name).offset == int(off), name


@pytest.mark.parametrize("page_size,over,rc", [
    (100, {}, S.SCALE_ERR_UNSUPPORTED),                 # pages of 64-row boxes only
    (64, dict(n_sink=100), S.SCALE_ERR_UNSUPPORTED),    # sinks must end on a 64-row boundary
    (64, dict(block_size=96), S.SCALE_ERR_UNSUPPORTED),
    (0, {}, S.SCALE_ERR_INVALID_ARG),
    (64, {}, S.SCALE_ERR_INVALID_ARG),                  # valid sizes, null pointers
])
def test_paged_entry_points_validate_before_launch(lib, page_size, over, rc):
    p = _p(**over)
    kv = S.ScaleKvPages(None, None, None, page_size, 16)
    assert lib.scale_sparse_prefill_paged(ctypes.byref(p), 0, 0, p.n_tokens, None, ctypes.byref(kv), None,
                                          None, None, None, None, None, 0, None) == rc
    assert lib.scale_build_reps_paged(ctypes.byref(p), None, ctypes.byref(kv), None, None, None, None,
                                      None, 0, None) == rc
    assert lib.scale_build_reps_range_paged(ctypes.byref(p), 0, p.outer_chunk, None, ctypes.byref(kv), None,
                                            None, None, None, None, 0, None) == rc


@pytest.mark.parametrize("over,tb,te,rc", [
    (dict(head_dim=64), 0, 8192, S.SCALE_ERR_UNSUPPORTED),   # parameters are checked first
    ({}, 0, 8192, S.SCALE_ERR_INVALID_ARG),                  # valid range, null pointers
    ({}, 4096, 8192, S.SCALE_ERR_INVALID_ARG),               # not on an outer-chunk boundary
    ({}, 8192, 4096, S.SCALE_ERR_INVALID_ARG),
])
def test_range_build_validates_before_launch(lib, over, tb, te, rc):
    p = _p(**over)
    assert lib.scale_build_reps_range(ctypes.byref(p), tb, te, None, None, None, None, None, None, None, 0,
                                      None) == rc

