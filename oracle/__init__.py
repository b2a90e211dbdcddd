"""CPU fp64 oracle of the Similarity Chunk Rolling prefill path (test infrastructure).

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package. The product package never imports it and
shares no code with it. The arithmetic lives in ``scale_oracle.c`` (plain C,
double precision); this module compiles it with gcc and marshals numpy arrays.

Parity pins: every function here is pinned by CPU tests against the paper's
closed forms, hand cases and library routines (dense causal SDPA); see the
``tests/test_oracle_*.py`` files.
"""

from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "scale_oracle.c")
_LIB = os.path.join(_HERE, "libscale_oracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile scale_oracle.c into libscale_oracle.so (gcc, OpenMP, no fast-math)."""
    if force or not os.path.exists(_LIB) or os.path.getmtime(_LIB) < os.path.getmtime(_SRC):
        tmp = _LIB + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-std=c11", "-fopenmp", "-fPIC", "-shared", "-fno-fast-math",
               _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB)
    return _LIB


def _load():
    global _lib
    with _lock:
        if _lib is None:
            build()
            lib = ctypes.CDLL(_LIB)
            P = ctypes.c_void_p
            i32, i64, dbl = ctypes.c_int32, ctypes.c_int64, ctypes.c_double
            lib.oracle_fingerprints.argtypes = [P, i64, i32, i32, i32, P, P]
            lib.oracle_anchor_clustering.argtypes = [P, P, i64, i64, i32, i64, dbl, P, P, P]
            lib.oracle_block_reps.argtypes = [P, i64, i32, i32, i32, P]
            lib.oracle_select.argtypes = [i32, i32, i32, i64, i32, i32, i32, i32, i32, dbl, i32,
                                          P, P, P, i64, P, P, P, P, P]
            lib.oracle_attention_rows.argtypes = [i32, i32, i32, i64, i32, i32, i32, i32, i32, dbl,
                                                  i32, P, P, P, P, i64, P, P, P, i64, P]
            for f in (lib.oracle_fingerprints, lib.oracle_anchor_clustering, lib.oracle_block_reps,
                      lib.oracle_select, lib.oracle_attention_rows):
                f.restype = ctypes.c_int
            _lib = lib
    return _lib


def _ptr(a: np.ndarray | None):
    return None if a is None else a.ctypes.data_as(ctypes.c_void_p)


def _check(rc: int, what: str):
    if rc != 0:
        raise ValueError(f"oracle {what}: invalid arguments (rc={rc})")


def _u16(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x)
    if x.dtype != np.uint16:
        raise TypeError("oracle inputs are bf16 bit patterns (uint16)")
    return x


def fingerprints(q: np.ndarray, sub_chunk: int):
    """Eq. 6 means of the multi-head queries per sub-chunk; returns (v [M, H_q*d_h], norms [M])."""
    q = _u16(q)
    N, Hq, dh = q.shape
    M = -(-N // sub_chunk)
    v = np.empty((M, Hq * dh), np.float64)
    norms = np.empty(M, np.float64)
    _check(_load().oracle_fingerprints(_ptr(q), N, Hq, dh, sub_chunk, _ptr(v), _ptr(norms)),
           "fingerprints")
    return v, norms


def anchor_clustering(v: np.ndarray, norms: np.ndarray, max_cluster_subchunks: int,
                      subchunks_per_outer: int, theta: float):
    """Algorithm 1 per outer chunk; returns (unit_start [n_units+1], margin)."""
    v = np.ascontiguousarray(v, np.float64)
    norms = np.ascontiguousarray(norms, np.float64)
    M, D = v.shape
    us = np.empty(M + 1, np.int32)
    n = ctypes.c_int32()
    mg = ctypes.c_double()
    _check(_load().oracle_anchor_clustering(_ptr(v), _ptr(norms), M, D, max_cluster_subchunks,
                                            subchunks_per_outer, float(theta), _ptr(us),
                                            ctypes.byref(n), ctypes.byref(mg)), "clustering")
    return us[: n.value + 1].copy(), mg.value


def block_reps(k: np.ndarray, block_size: int) -> np.ndarray:
    """Mean key per block and KV head; returns reps [H_kv, nb, d_h]."""
    k = _u16(k)
    N, Hkv, dh = k.shape
    nb = -(-N // block_size)
    reps = np.empty((Hkv, nb, dh), np.float64)
    _check(_load().oracle_block_reps(_ptr(k), N, Hkv, dh, block_size, _ptr(reps)), "block_reps")
    return reps


def select(*, num_q_heads: int, n_tokens: int, sub_chunk: int, block_size: int, top_k: int,
           n_sink: int, n_local: int, select_scale: float, per_subchunk: bool,
           reps: np.ndarray, v: np.ndarray, unit_start: np.ndarray | None, want_scores=False):
    """Eq. 9 with head soft-voting; returns dict(sel, sel_count, cand_count, gap[, scores])."""
    reps = np.ascontiguousarray(reps, np.float64)
    v = np.ascontiguousarray(v, np.float64)
    Hkv, nb, dh = reps.shape
    M = v.shape[0]
    if per_subchunk:
        n_units = M
        us = None
    else:
        us = np.ascontiguousarray(unit_start, np.int32)
        n_units = us.shape[0] - 1
    kk = max(top_k, 0)
    sel = np.empty((n_units, max(kk, 1)), np.int32)
    sc = np.empty(n_units, np.int32)
    cc = np.empty(n_units, np.int32)
    gap = np.empty(n_units, np.float64)
    scores = np.empty((n_units, nb), np.float64) if want_scores else None
    _check(_load().oracle_select(num_q_heads, Hkv, dh, n_tokens, sub_chunk, block_size, top_k,
                                 n_sink, n_local, float(select_scale), int(per_subchunk),
                                 _ptr(reps), _ptr(v), _ptr(us), n_units, _ptr(sel), _ptr(sc),
                                 _ptr(cc), _ptr(gap), _ptr(scores)), "select")
    out = dict(sel=sel[:, :kk], sel_count=sc, cand_count=cc, gap=gap)
    if want_scores:
        out["scores"] = scores
    return out


def attention_rows(*, q: np.ndarray, k: np.ndarray, v: np.ndarray, sub_chunk: int,
                   block_size: int, top_k: int, n_sink: int, n_local: int, attn_scale: float,
                   per_subchunk: bool, unit_start: np.ndarray | None, sel: np.ndarray,
                   sel_count: np.ndarray, rows: np.ndarray) -> np.ndarray:
    """Eq. 10 for the listed token rows; returns out [n_rows, H_q, d_h] (float64)."""
    q, k, v = _u16(q), _u16(k), _u16(v)
    N, Hq, dh = q.shape
    Hkv = k.shape[1]
    rows = np.ascontiguousarray(rows, np.int64)
    if per_subchunk:
        n_units = -(-N // sub_chunk)
        us = None
    else:
        us = np.ascontiguousarray(unit_start, np.int32)
        n_units = us.shape[0] - 1
    sel = np.ascontiguousarray(sel, np.int32)
    sel = sel.reshape(n_units, top_k) if top_k > 0 else np.zeros((n_units, 0), np.int32)
    if sel.shape[1] != top_k:
        raise ValueError("sel must be [n_units, top_k]")
    sc = np.ascontiguousarray(sel_count, np.int32)
    out = np.empty((rows.shape[0], Hq, dh), np.float64)
    _check(_load().oracle_attention_rows(Hq, Hkv, dh, N, sub_chunk, block_size, top_k, n_sink,
                                         n_local, float(attn_scale), int(per_subchunk), _ptr(q),
                                         _ptr(k), _ptr(v), _ptr(us), n_units,
                                         _ptr(sel) if top_k > 0 else None, _ptr(sc), _ptr(rows),
                                         rows.shape[0], _ptr(out)), "attention_rows")
    return out


def run_path(w, q: np.ndarray, k: np.ndarray, v: np.ndarray, *, per_subchunk: bool,
             rows: np.ndarray | None = None, theta: float | None = None,
             select_scale: float = 1.0, attn_scale: float | None = None):
    """Algorithm 2 over the whole sequence, step by step; returns a dict of every stage."""
    theta = w.theta if theta is None else theta
    attn_scale = 1.0 / np.sqrt(w.head_dim) if attn_scale is None else attn_scale
    fv, norms = fingerprints(q, w.sub_chunk)
    per_outer = w.outer_chunk // w.sub_chunk
    us, margin = anchor_clustering(fv, norms, w.max_cluster_subchunks, per_outer, theta)
    reps = block_reps(k, w.block_size)
    s = select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
               block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
               select_scale=select_scale, per_subchunk=per_subchunk, reps=reps, v=fv,
               unit_start=us)
    out = dict(fingerprints=fv, norms=norms, unit_start=us, margin=margin, reps=reps, **s)
    if rows is not None:
        out["rows"] = np.asarray(rows, np.int64)
        out["attn"] = attention_rows(q=q, k=k, v=v, sub_chunk=w.sub_chunk,
                                     block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink,
                                     n_local=w.n_local, attn_scale=attn_scale,
                                     per_subchunk=per_subchunk, unit_start=us, sel=s["sel"],
                                     sel_count=s["sel_count"], rows=out["rows"])
    return out


def member_selection(w, reps: np.ndarray, v: np.ndarray, unit_start: np.ndarray, j: int,
                     select_scale: float = 1.0):
    """Selection of every cluster scored with its member j's fingerprint in place
    of the anchor's, against the cluster's own candidate blocks (Sec. IV-C's
    per-sub-chunk retrieval "against the same KV cache"); units with at most j
    sub-chunks keep their anchor."""
    v2 = np.array(v, np.float64, copy=True)
    for u in range(len(unit_start) - 1):
        a, b = int(unit_start[u]), int(unit_start[u + 1])
        if b - a > j:
            v2[a] = v[a + j]
    return select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
                  block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                  select_scale=select_scale, per_subchunk=False, reps=reps, v=v2,
                  unit_start=unit_start)


def overlap_ratio(anchor_blocks, member_blocks) -> float:
    """Overlap ratio of one cluster (Sec. IV-C): the share of the anchor's
    selected blocks that at least one other member would also select.
    anchor_blocks: the anchor's selection; member_blocks: one selection per
    other member."""
    anchor = {int(b) for b in anchor_blocks}
    others = set()
    for m in member_blocks:
        others |= {int(b) for b in m}
    return len(anchor & others) / len(anchor)


def _bf16_f64(x: np.ndarray) -> np.ndarray:
    x = np.ascontiguousarray(x, np.uint16)
    return (x.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def decode_select(q_t: np.ndarray, k: np.ndarray, t: int, *, n_sink: int, n_local: int, top_k: int,
                  select_scale: float = 1.0):
    """Eq. 9 for one query token (a unit of C = 1 token, Def. 1) at position t,
    token level: candidates n_sink <= c < W_t = max(0, t - n_local); per-head
    softmax of select_scale * q^(h) . k_c^(h / g) over them, summed over the
    heads; the top_k tokens by (score desc, index asc), returned ascending,
    with the relative gap between the k-th and (k+1)-th scores (inf if none).
      q_t [H_q][d] bf16 bits, k [N][H_kv][d] bf16 bits."""
    Hq = q_t.shape[0]
    Hkv = k.shape[1]
    g = Hq // Hkv
    W = max(0, t - n_local)
    cand = np.arange(n_sink, W, dtype=np.int64)
    if cand.size == 0:
        return np.zeros(0, np.int64), np.inf
    q = _bf16_f64(q_t)
    kc = _bf16_f64(k[cand])  # [n, H_kv, d]
    score = np.zeros(cand.size)
    for h in range(Hq):
        z = select_scale * (kc[:, h // g, :] @ q[h])
        e = np.exp(z - z.max())
        score += e / e.sum()
    order = np.lexsort((cand, -score))
    take = min(top_k, cand.size)
    gap = np.inf
    if cand.size > top_k > 0:
        s_k, s_k1 = score[order[top_k - 1]], score[order[top_k]]
        gap = (s_k - s_k1) / s_k
    return np.sort(cand[order[:take]]), gap


def decode_reuse(queries: np.ndarray, theta: float, max_shared: int):
    """The selection cache across decode steps (Eq. 8 with Algorithm 1's cap,
    applied in time): step 0 retrieves; step i reuses the anchor's selection
    when cos(q_i, anchor) >= theta (all heads together; a zero norm gives 0)
    and fewer than max_shared steps have shared it, else it retrieves and
    becomes the anchor. Returns (retrieve flags, anchor index of every step,
    |cos - theta| of the closest decision).
      queries [T][H_q][d] bf16 bits."""
    qs = [_bf16_f64(q).ravel() for q in queries]
    retrieve, anchor_of, margin = [], [], np.inf
    anchor, shared = None, 0
    for i, q in enumerate(qs):
        if anchor is None:
            reuse = False
        else:
            na, nq = np.linalg.norm(qs[anchor]), np.linalg.norm(q)
            c = float(qs[anchor] @ q / (na * nq)) if na > 0 and nq > 0 else 0.0
            if shared < max_shared:
                margin = min(margin, abs(c - theta))
            reuse = shared < max_shared and c >= theta
        if reuse:
            shared += 1
        else:
            anchor, shared = i, 1
        retrieve.append(not reuse)
        anchor_of.append(anchor)
    return np.array(retrieve), np.array(anchor_of), margin

