"""ctypes binding of libscale (include/scale.h), one Python function per C entry point.

This module only marshals arguments: torch tensors become raw pointers and
the caller's CUDA stream handle. Every step of the path runs inside
libscale.so's kernels. If the library has not been built, loading raises
``ScaleLibraryMissing``; there is no fallback implementation.
"""

from __future__ import annotations

import ctypes
import dataclasses
import os
import re
import threading

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libscale.so")
HEADER = os.path.join(HERE, "..", "include", "scale.h")

SCALE_OK = 0
SCALE_ERR_INVALID_ARG = -1
SCALE_ERR_UNSUPPORTED = -2
SCALE_ERR_WORKSPACE = -3
SCALE_ERR_CUDA = -4
SCALE_ERR_TIMEOUT = -5
SCALE_ERR_DEVICE = -6
SCALE_MODE_PER_CLUSTER = 0
SCALE_MODE_PER_SUBCHUNK = 1


class ScaleLibraryMissing(RuntimeError):
    pass


class ScaleError(RuntimeError):
    def __init__(self, fn: str, rc: int):
        super().__init__(f"{fn} failed: {rc} ({status_string(rc)})")
        self.rc = rc


class ScaleParams(ctypes.Structure):
    """Mirror of scale_params_t."""

    _fields_ = [
        ("num_q_heads", ctypes.c_int32),
        ("num_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32),
        ("sub_chunk", ctypes.c_int32),
        ("n_tokens", ctypes.c_int64),
        ("max_cluster_subchunks", ctypes.c_int32),
        ("outer_chunk", ctypes.c_int32),
        ("theta", ctypes.c_float),
        ("block_size", ctypes.c_int32),
        ("top_k", ctypes.c_int32),
        ("n_sink", ctypes.c_int32),
        ("n_local", ctypes.c_int32),
        ("select_scale", ctypes.c_float),
        ("attn_scale", ctypes.c_float),
    ]


class ScaleKvPages(ctypes.Structure):
    """scale_kv_pages_t: a paged K/V cache (device pointers)."""

    _fields_ = [("k_pages", ctypes.c_void_p), ("v_pages", ctypes.c_void_p),
                ("page_table", ctypes.c_void_p), ("page_size", ctypes.c_int32),
                ("num_pages", ctypes.c_int64)]


def kv_pages(k_pages, v_pages, page_table, page_size: int) -> ScaleKvPages:
    """Descriptor of torch tensors k_pages / v_pages [num_pages][page_size][H_kv][128]
    and page_table (int32) on the device."""
    return ScaleKvPages(_ptr(k_pages), _ptr(v_pages), _ptr(page_table), page_size, k_pages.shape[0])


def params(*, num_q_heads, num_kv_heads, head_dim=128, sub_chunk, n_tokens, max_cluster_subchunks,
           outer_chunk=0, theta=-1.0, block_size, top_k, n_sink, n_local, select_scale=1.0,
           attn_scale=0.0) -> ScaleParams:
    return ScaleParams(num_q_heads, num_kv_heads, head_dim, sub_chunk, n_tokens,
                       max_cluster_subchunks, outer_chunk, theta, block_size, top_k, n_sink,
                       n_local, select_scale, attn_scale)


def params_for(w, **overrides) -> ScaleParams:
    """scale_params_t for a workload description with the usual field names."""
    kw = dict(num_q_heads=w.num_q_heads, num_kv_heads=w.num_kv_heads, head_dim=w.head_dim,
              sub_chunk=w.sub_chunk, n_tokens=w.n_tokens,
              max_cluster_subchunks=w.max_cluster_subchunks, outer_chunk=w.outer_chunk,
              theta=w.theta, block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink,
              n_local=w.n_local)
    kw.update(overrides)
    return params(**kw)


_lock = threading.Lock()
_lib = None


def declared_functions() -> list[str]:
    """Names of the functions include/scale.h declares."""
    with open(HEADER) as f:
        text = f.read()
    return sorted(set(re.findall(r"\b(scale_[a-z0-9_]+)\s*\(", text)))


def load() -> ctypes.CDLL:
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise ScaleLibraryMissing(
                f"{LIB_PATH} is missing: build it with paper_2609_31568_gb300._build.build()")
        lib = ctypes.CDLL(LIB_PATH)
        P, i32, i64, sz, u64 = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t, ctypes.c_uint64
        pp = ctypes.POINTER(ScaleParams)
        kp = ctypes.POINTER(ScaleKvPages)
        sig = {
            "scale_workspace_size": [pp, i32, ctypes.POINTER(sz)],
            "scale_workspace_init": [P, sz, P],
            "scale_build_reps": [pp, P, P, P, P, P, P, P, sz, P],
            "scale_build_reps_noalloc": [pp, P, P, P, P, P, P, P],
            "scale_select": [pp, i32, i64, i64, P, P, P, P, P, P, P, P, sz, P],
            "scale_select_tokens": [pp, i32, i64, i64, P, P, P, P, P, P, P, P, sz, P],
            "scale_build_reps_paged": [pp, P, kp, P, P, P, P, P, sz, P],
            "scale_build_reps_range": [pp, i64, i64, P, P, P, P, P, P, P, sz, P],
            "scale_build_reps_range_paged": [pp, i64, i64, P, kp, P, P, P, P, P, sz, P],
            "scale_select_tokens_paged": [pp, i32, i64, i64, kp, P, P, P, P, P, P, P, sz, P],
            "scale_sparse_prefill_paged": [pp, i32, i64, i64, P, kp, P, P, P, P, P, P, sz, P],
            "scale_decode_cache_size": [pp, ctypes.POINTER(sz)],
            "scale_decode_cache_init": [P, sz, P],
            "scale_decode_workspace_size": [pp, ctypes.POINTER(sz)],
            "scale_decode_step": [pp, i64, P, P, P, P, sz, P, P, sz, P],
            "scale_sparse_prefill": [pp, i32, i64, i64, P, P, P, P, P, P, P, P, P, sz, P],
            "scale_get_device_status": [P, P, ctypes.POINTER(i32)],
            "scale_retrieval_calls": [pp, i32, P, i32, ctypes.POINTER(i64), ctypes.POINTER(i64)],
            "scale_prefill_host_arena_size": [pp, i32, ctypes.POINTER(sz)],
            "scale_prefill_host": [pp, i32, P, P, P, P, P, sz, P],
            "scale_set_wait_timeout_ns": [u64],
            "scale_selftest_wait_timeout": [P, sz, u64, P],
            "scale_status_string": [ctypes.c_int],
            "scale_version": [],
        }
        for name, args in sig.items():
            f = getattr(lib, name)
            f.argtypes = args
            f.restype = ctypes.c_int
        lib.scale_status_string.restype = ctypes.c_char_p
        _lib = lib
        return lib


def _ptr(x) -> int | None:
    """Device or host address of a tensor / array / int (None for None)."""
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        if not x.is_contiguous():
            raise ValueError("tensors passed to libscale must be contiguous")
        return x.data_ptr()
    if hasattr(x, "ctypes"):
        return x.ctypes.data
    raise TypeError(f"cannot pass {type(x).__name__} as a pointer")


def _nbytes(x) -> int:
    if hasattr(x, "numel"):
        return x.numel() * x.element_size()
    return int(x.nbytes)


def _stream(stream) -> int | None:
    if stream is None:
        import torch

        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def _check(name: str, rc: int) -> None:
    if rc != SCALE_OK:
        raise ScaleError(name, rc)


def status_string(rc: int) -> str:
    return load().scale_status_string(rc).decode()


def scale_version() -> int:
    return load().scale_version()


def scale_status_string(rc: int) -> str:
    return status_string(rc)


def scale_workspace_size(p: ScaleParams, mode: int) -> int:
    n = ctypes.c_size_t()
    _check("scale_workspace_size", load().scale_workspace_size(ctypes.byref(p), mode, ctypes.byref(n)))
    return n.value


def scale_workspace_init(ws, stream=None) -> None:
    _check("scale_workspace_init", load().scale_workspace_init(_ptr(ws), _nbytes(ws), _stream(stream)))


def scale_build_reps(p, q, k, reps, fingerprints, unit_start, n_units, ws, stream=None) -> None:
    _check("scale_build_reps", load().scale_build_reps(
        ctypes.byref(p), _ptr(q), _ptr(k), _ptr(reps), _ptr(fingerprints), _ptr(unit_start),
        _ptr(n_units), _ptr(ws), _nbytes(ws), _stream(stream)))


def scale_build_reps_range(p, tok_begin, tok_end, q, k, reps, fingerprints, unit_start, n_units, ws,
                           stream=None) -> None:
    """Step (a) over the outer chunks covering [tok_begin, tok_end); ranges go in order from 0."""
    _check("scale_build_reps_range", load().scale_build_reps_range(
        ctypes.byref(p), tok_begin, tok_end, _ptr(q), _ptr(k), _ptr(reps), _ptr(fingerprints),
        _ptr(unit_start), _ptr(n_units), _ptr(ws), _nbytes(ws), _stream(stream)))


def scale_build_reps_noalloc(p, q, k, reps, fingerprints, unit_start, n_units, stream=None) -> None:
    """Step (a) with the library's fixed scratch array instead of a workspace."""
    _check("scale_build_reps_noalloc", load().scale_build_reps_noalloc(
        ctypes.byref(p), _ptr(q), _ptr(k), _ptr(reps), _ptr(fingerprints), _ptr(unit_start),
        _ptr(n_units), _stream(stream)))


def scale_select(p, mode, tok_begin, tok_end, reps, fingerprints, unit_start, n_units,
                 sel_blocks, sel_count, sel_scores, ws, stream=None) -> None:
    _check("scale_select", load().scale_select(
        ctypes.byref(p), mode, tok_begin, tok_end, _ptr(reps), _ptr(fingerprints),
        _ptr(unit_start), _ptr(n_units), _ptr(sel_blocks), _ptr(sel_count), _ptr(sel_scores),
        _ptr(ws), _nbytes(ws), _stream(stream)))


def scale_select_tokens(p, mode, tok_begin, tok_end, k, fingerprints, unit_start, n_units,
                        sel_tokens, sel_count, sel_scores, ws, stream=None) -> None:
    _check("scale_select_tokens", load().scale_select_tokens(
        ctypes.byref(p), mode, tok_begin, tok_end, _ptr(k), _ptr(fingerprints),
        _ptr(unit_start), _ptr(n_units), _ptr(sel_tokens), _ptr(sel_count), _ptr(sel_scores),
        _ptr(ws), _nbytes(ws), _stream(stream)))


def scale_sparse_prefill(p, mode, tok_begin, tok_end, q, k, v, unit_start, n_units, sel_blocks,
                         sel_count, out, ws, stream=None) -> None:
    _check("scale_sparse_prefill", load().scale_sparse_prefill(
        ctypes.byref(p), mode, tok_begin, tok_end, _ptr(q), _ptr(k), _ptr(v), _ptr(unit_start),
        _ptr(n_units), _ptr(sel_blocks), _ptr(sel_count), _ptr(out), _ptr(ws), _nbytes(ws),
        _stream(stream)))


def scale_build_reps_paged(p, q, kv: ScaleKvPages, reps, fingerprints, unit_start, n_units, ws,
                           stream=None) -> None:
    _check("scale_build_reps_paged", load().scale_build_reps_paged(
        ctypes.byref(p), _ptr(q), ctypes.byref(kv), _ptr(reps), _ptr(fingerprints), _ptr(unit_start),
        _ptr(n_units), _ptr(ws), _nbytes(ws), _stream(stream)))


def scale_build_reps_range_paged(p, tok_begin, tok_end, q, kv: ScaleKvPages, reps, fingerprints,
                                 unit_start, n_units, ws, stream=None) -> None:
    _check("scale_build_reps_range_paged", load().scale_build_reps_range_paged(
        ctypes.byref(p), tok_begin, tok_end, _ptr(q), ctypes.byref(kv), _ptr(reps), _ptr(fingerprints),
        _ptr(unit_start), _ptr(n_units), _ptr(ws), _nbytes(ws), _stream(stream)))


def scale_select_tokens_paged(p, mode, tok_begin, tok_end, kv: ScaleKvPages, fingerprints, unit_start,
                              n_units, sel_tokens, sel_count, sel_scores, ws, stream=None) -> None:
    _check("scale_select_tokens_paged", load().scale_select_tokens_paged(
        ctypes.byref(p), mode, tok_begin, tok_end, ctypes.byref(kv), _ptr(fingerprints), _ptr(unit_start),
        _ptr(n_units), _ptr(sel_tokens), _ptr(sel_count), _ptr(sel_scores), _ptr(ws), _nbytes(ws),
        _stream(stream)))


def scale_sparse_prefill_paged(p, mode, tok_begin, tok_end, q, kv: ScaleKvPages, unit_start, n_units,
                               sel_blocks, sel_count, out, ws, stream=None) -> None:
    _check("scale_sparse_prefill_paged", load().scale_sparse_prefill_paged(
        ctypes.byref(p), mode, tok_begin, tok_end, _ptr(q), ctypes.byref(kv), _ptr(unit_start),
        _ptr(n_units), _ptr(sel_blocks), _ptr(sel_count), _ptr(out), _ptr(ws), _nbytes(ws),
        _stream(stream)))


def run_path_paged(p: ScaleParams, mode: int, q, kv: ScaleKvPages, buf: "Buffers", stream=None) -> None:
    """Steps (a)-(d) with K and V in a paged cache."""
    scale_build_reps_paged(p, q, kv, buf.reps, buf.fingerprints, buf.unit_start, buf.n_units, buf.ws, stream)
    if p.block_size == 1:
        scale_select_tokens_paged(p, mode, 0, p.n_tokens, kv, buf.fingerprints, buf.unit_start, buf.n_units,
                                  buf.sel_blocks, buf.sel_count, buf.sel_scores, buf.ws, stream)
    else:
        scale_select(p, mode, 0, p.n_tokens, buf.reps, buf.fingerprints, buf.unit_start, buf.n_units,
                     buf.sel_blocks, buf.sel_count, buf.sel_scores, buf.ws, stream)
    scale_sparse_prefill_paged(p, mode, 0, p.n_tokens, q, kv, buf.unit_start, buf.n_units, buf.sel_blocks,
                               buf.sel_count, buf.out, buf.ws, stream)


def scale_decode_cache_size(p) -> int:
    n = ctypes.c_size_t()
    _check("scale_decode_cache_size", load().scale_decode_cache_size(ctypes.byref(p), ctypes.byref(n)))
    return n.value


def scale_decode_cache_init(cache, stream=None) -> None:
    _check("scale_decode_cache_init", load().scale_decode_cache_init(_ptr(cache), _nbytes(cache), _stream(stream)))


def scale_decode_workspace_size(p) -> int:
    n = ctypes.c_size_t()
    _check("scale_decode_workspace_size", load().scale_decode_workspace_size(ctypes.byref(p), ctypes.byref(n)))
    return n.value


def scale_decode_step(p, t: int, q_t, k, v, cache, out_t, ws, stream=None) -> None:
    _check("scale_decode_step", load().scale_decode_step(
        ctypes.byref(p), t, _ptr(q_t), _ptr(k), _ptr(v), _ptr(cache), _nbytes(cache), _ptr(out_t),
        _ptr(ws), _nbytes(ws), _stream(stream)))


def decode_cache_state(cache) -> dict:
    """Host view of a decode cache's header: whether the last step retrieved,
    the anchor position, steps sharing the anchor, and its selection size."""
    import torch

    st = cache[:64].view(torch.int32).cpu().tolist()
    return {"valid": st[0], "steps": st[1], "retrieved": st[2], "anchor": st[4]}


def decode_cache_selection(cache, p) -> tuple:
    """The selection held by a decode cache (ascending tokens) and its size."""
    import torch

    off = 256 + p.num_q_heads * 128 * 4
    k = max(p.top_k, 1)
    raw = cache[off: off + (k + 1) * 4].view(torch.int32).cpu().numpy()
    return raw[:k].copy(), int(raw[k])


def scale_get_device_status(ws, stream=None) -> int:
    st = ctypes.c_int32()
    _check("scale_get_device_status", load().scale_get_device_status(_ptr(ws), _stream(stream),
                                                                     ctypes.byref(st)))
    return st.value


def scale_retrieval_calls(p, mode, unit_start_host, n_units: int) -> tuple[int, int]:
    import numpy as np

    us = None if unit_start_host is None else np.ascontiguousarray(unit_start_host, np.int32)
    units, calls = ctypes.c_int64(), ctypes.c_int64()
    _check("scale_retrieval_calls", load().scale_retrieval_calls(
        ctypes.byref(p), mode, None if us is None else us.ctypes.data, n_units,
        ctypes.byref(units), ctypes.byref(calls)))
    return units.value, calls.value


def scale_prefill_host_arena_size(p, mode) -> int:
    n = ctypes.c_size_t()
    _check("scale_prefill_host_arena_size",
           load().scale_prefill_host_arena_size(ctypes.byref(p), mode, ctypes.byref(n)))
    return n.value


def scale_prefill_host(p, mode, q_host, k_host, v_host, out_host, arena, stream=None) -> None:
    _check("scale_prefill_host", load().scale_prefill_host(
        ctypes.byref(p), mode, _ptr(q_host), _ptr(k_host), _ptr(v_host), _ptr(out_host),
        _ptr(arena), _nbytes(arena), _stream(stream)))


def scale_set_wait_timeout_ns(ns: int) -> None:
    _check("scale_set_wait_timeout_ns", load().scale_set_wait_timeout_ns(ns))


def scale_selftest_wait_timeout(ws, timeout_ns: int, stream=None) -> None:
    _check("scale_selftest_wait_timeout", load().scale_selftest_wait_timeout(
        _ptr(ws), _nbytes(ws), timeout_ns, _stream(stream)))


@dataclasses.dataclass
class Buffers:
    """Device tensors of one layer's path, allocated with torch (plumbing only)."""

    reps: object
    fingerprints: object
    unit_start: object
    n_units: object
    sel_blocks: object
    sel_count: object
    sel_scores: object
    out: object
    ws: object


def allocate(p: ScaleParams, mode: int, device="cuda", want_scores: bool = False) -> Buffers:
    import torch

    N, Hq, Hkv = p.n_tokens, p.num_q_heads, p.num_kv_heads
    M = -(-N // p.sub_chunk)
    nb = -(-N // p.block_size)
    f32, i32 = torch.float32, torch.int32
    ws = torch.empty(scale_workspace_size(p, mode), dtype=torch.uint8, device=device)
    scale_workspace_init(ws)
    return Buffers(
        # block size 1 selects from K itself (scale_select_tokens): no representatives
        reps=None if p.block_size == 1 else torch.empty((Hkv, nb, p.head_dim), dtype=f32, device=device),
        fingerprints=torch.empty((M, Hq * p.head_dim), dtype=f32, device=device),
        unit_start=torch.empty(M + 1, dtype=i32, device=device),
        n_units=torch.empty(1, dtype=i32, device=device),
        sel_blocks=torch.empty((M, max(p.top_k, 1)), dtype=i32, device=device),
        sel_count=torch.empty(M, dtype=i32, device=device),
        sel_scores=torch.empty((M, nb), dtype=f32, device=device) if want_scores else None,
        out=torch.empty((N, Hq, p.head_dim), dtype=torch.bfloat16, device=device),
        ws=ws,
    )


def select(p: ScaleParams, mode: int, tok_begin: int, tok_end: int, k, buf: Buffers, stream=None) -> None:
    """Steps (b)-(c): block-level selection, or token-level when the block size is 1."""
    if p.block_size == 1:
        scale_select_tokens(p, mode, tok_begin, tok_end, k, buf.fingerprints, buf.unit_start,
                            buf.n_units, buf.sel_blocks, buf.sel_count, buf.sel_scores, buf.ws, stream)
    else:
        scale_select(p, mode, tok_begin, tok_end, buf.reps, buf.fingerprints, buf.unit_start,
                     buf.n_units, buf.sel_blocks, buf.sel_count, buf.sel_scores, buf.ws, stream)


def run_path(p: ScaleParams, mode: int, q, k, v, buf: Buffers, tok_begin: int = 0,
             tok_end: int | None = None, stream=None) -> None:
    """Steps (a)-(d) on one layer: build reps and clusters, select, attend."""
    tok_end = p.n_tokens if tok_end is None else tok_end
    scale_build_reps(p, q, k, buf.reps, buf.fingerprints, buf.unit_start, buf.n_units, buf.ws, stream)
    select(p, mode, tok_begin, tok_end, k, buf, stream)
    scale_sparse_prefill(p, mode, tok_begin, tok_end, q, k, v, buf.unit_start, buf.n_units,
                         buf.sel_blocks, buf.sel_count, buf.out, buf.ws, stream)
