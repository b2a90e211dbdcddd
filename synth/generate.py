"""Seeded Gaussian-mixture Q/K/V shaped like the paper's long-context workloads.

The paper measures on InfiniteBench and RULER with Qwen2-7B (Sec. VI-A1);
neither the model nor the data exists here, so these synthetic tensors stand
in for them. The recipe, per layer:

1. centroids: for every KV head, ``C`` directions drawn from N(0, I) and
   scaled to norm 3 (the drifting variant draws two such sets ``a`` and ``b``
   and, at position t, uses ``3 * normalize((1 - t/N) a + (t/N) b)``);
2. keys: a component id per (token, KV head), drawn i.i.d. uniform and used
   in the order drawn, plus N(0, 1) noise per element;
3. queries: a component id per (token, query head) from the centroid set of
   the query head's KV head (``h // (H_q / H_kv)``), plus N(0, 1) noise;
4. values: N(0, 1);
5. optional rotate-half RoPE at absolute positions ``0..N-1`` on Q and K;
6. mixing, noise and RoPE are computed in float32 (the centroids in
   float64), then rounded to bf16 with round-to-nearest-even.

Random streams are counter-keyed by ``(seed, layer, tensor, 4096-token
chunk)`` with numpy's PCG64, so any token range can be regenerated exactly
without generating the tokens before it.
"""

from __future__ import annotations

import dataclasses
import os

import numpy as np

CHUNK = 4096  # tokens per independent random stream


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    num_q_heads: int
    num_kv_heads: int
    head_dim: int
    n_tokens: int
    sub_chunk: int
    max_cluster_subchunks: int
    outer_chunk: int
    block_size: int
    top_k: int
    n_sink: int
    n_local: int
    components: int
    rope_base: float | None
    drift: bool
    layers: int = 1
    seed: int = 0
    theta: float = -1.0

    def replace(self, **kw) -> "Workload":
        return dataclasses.replace(self, **kw)

    @property
    def group(self) -> int:
        return self.num_q_heads // self.num_kv_heads

    @property
    def n_subchunks(self) -> int:
        return -(-self.n_tokens // self.sub_chunk)

    @property
    def n_blocks(self) -> int:
        return -(-self.n_tokens // self.block_size)


WORKLOADS: dict[str, Workload] = {
    # GQA 4:1 single layer, 4K context, no RoPE.
    "gqa4-4k": Workload("gqa4-4k", 4, 1, 128, 4096, 256, 4, 1024, 64, 8, 64, 256, 32, None, False),
    # Llama-3-8B-shaped layer at 32K context.
    "llama8b-32k": Workload("llama8b-32k", 32, 8, 128, 32768, 1024, 8, 8192, 128, 32, 128, 1024, 256,
                            500000.0, False),
    # Same layer at 128K context with slowly drifting mixture components.
    "llama8b-128k": Workload("llama8b-128k", 32, 8, 128, 131072, 2048, 8, 16384, 128, 64, 128, 1024,
                             256, 500000.0, True),
    # 32-layer stack at 64K context, independent inputs per layer (layer l uses seed l).
    "llama8b-64k-32l": Workload("llama8b-64k-32l", 32, 8, 128, 65536, 1024, 8, 8192, 128, 32, 128, 1024,
                                256, 500000.0, False, layers=32),
    # 1M-token single layer.
    "llama8b-1m": Workload("llama8b-1m", 32, 8, 128, 1048576, 4096, 16, 65536, 256, 128, 128, 1024,
                           1024, 500000.0, False),
}


def workload(name: str, **overrides) -> Workload:
    w = WORKLOADS[name]
    return w.replace(**overrides) if overrides else w


def f64_to_bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round to float32 (if wider), then to bf16 (nearest-even); returns uint16 bit patterns."""
    f = np.ascontiguousarray(x, dtype=np.float32)
    u = f.view(np.uint32)
    rounded = (u + np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))) >> np.uint32(16)
    return rounded.astype(np.uint16)


def bf16_bits_to_f32(b: np.ndarray) -> np.ndarray:
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << np.uint32(16)).view(np.float32)


def _unit_rows(x: np.ndarray) -> np.ndarray:
    return x / np.linalg.norm(x, axis=-1, keepdims=True)


def _centroids(w: Workload, layer: int, seed: int):
    rng = np.random.default_rng([seed, layer, 0])
    shape = (w.num_kv_heads, w.components, w.head_dim)
    if not w.drift:
        return (3.0 * _unit_rows(rng.standard_normal(shape))).astype(np.float32), None
    a = _unit_rows(rng.standard_normal(shape)).astype(np.float32)
    b = _unit_rows(rng.standard_normal(shape)).astype(np.float32)
    return a, b


def _mix(w: Workload, cents, heads_kv: np.ndarray, ids: np.ndarray, pos: np.ndarray) -> np.ndarray:
    """Centroid vectors for component ids[t, h] of KV head heads_kv[h] at positions pos[t]."""
    a, b = cents
    if b is None:
        return a[heads_kv[None, :], ids]
    f = (pos.astype(np.float32) / np.float32(w.n_tokens))[:, None, None]
    m = (np.float32(1.0) - f) * a[heads_kv[None, :], ids] + f * b[heads_kv[None, :], ids]
    return np.float32(3.0) * _unit_rows(m)


def _rope(x: np.ndarray, pos: np.ndarray, base: float) -> np.ndarray:
    half = x.shape[-1] // 2
    inv = base ** (-np.arange(half, dtype=np.float64) * 2.0 / x.shape[-1])
    ang = pos.astype(np.float64)[:, None] * inv[None, :]
    c = np.cos(ang).astype(np.float32)[:, None, :]
    s = np.sin(ang).astype(np.float32)[:, None, :]
    lo, hi = x[..., :half], x[..., half:]
    return np.concatenate([lo * c - hi * s, hi * c + lo * s], axis=-1)


def _chunk(w: Workload, layer: int, seed: int, cents, ch: int):
    t0 = ch * CHUNK
    t1 = min(w.n_tokens, t0 + CHUNK)
    T = t1 - t0
    pos = np.arange(t0, t1, dtype=np.int64)
    kvh = np.arange(w.num_kv_heads)
    qkv = np.arange(w.num_q_heads) // w.group

    rk = np.random.default_rng([seed, layer, 1, ch])
    kid = rk.integers(0, w.components, size=(T, w.num_kv_heads))
    k = _mix(w, cents, kvh, kid, pos) + rk.standard_normal((T, w.num_kv_heads, w.head_dim), dtype=np.float32)

    rq = np.random.default_rng([seed, layer, 2, ch])
    qid = rq.integers(0, w.components, size=(T, w.num_q_heads))
    q = _mix(w, cents, qkv, qid, pos) + rq.standard_normal((T, w.num_q_heads, w.head_dim), dtype=np.float32)

    rv = np.random.default_rng([seed, layer, 3, ch])
    v = rv.standard_normal((T, w.num_kv_heads, w.head_dim), dtype=np.float32)

    if w.rope_base:
        q = _rope(q, pos, w.rope_base)
        k = _rope(k, pos, w.rope_base)
    return f64_to_bf16_bits(q), f64_to_bf16_bits(k), f64_to_bf16_bits(v)


def _chunk_job(args):
    w, layer, seed, ch = args
    return _chunk(w, layer, seed, _centroids(w, layer, seed), ch)


def generate_layer(w: Workload, layer: int = 0, seed: int | None = None,
                   t0: int = 0, t1: int | None = None, workers: int | None = None):
    """Q [T, H_q, d_h], K and V [T, H_kv, d_h] as bf16 bit patterns (uint16) for tokens [t0, t1).

    ``workers`` > 1 spreads the independent 4096-token chunks over a process
    pool started with the ``spawn`` method (safe after CUDA initialisation);
    the result does not depend on it.
    """
    if seed is None:
        seed = w.seed + layer if w.layers > 1 else w.seed
    t1 = w.n_tokens if t1 is None else t1
    c0, c1 = t0 // CHUNK, -(-t1 // CHUNK)
    T = t1 - t0
    q = np.empty((T, w.num_q_heads, w.head_dim), np.uint16)
    k = np.empty((T, w.num_kv_heads, w.head_dim), np.uint16)
    v = np.empty((T, w.num_kv_heads, w.head_dim), np.uint16)
    jobs = [(w, layer, seed, ch) for ch in range(c0, c1)]
    if workers is None:
        workers = min(len(jobs), os.cpu_count() or 1) if T * w.num_q_heads >= (1 << 20) else 1
    if workers > 1 and len(jobs) > 1:
        import concurrent.futures as cf
        import multiprocessing as mp

        # A process pool that raises (BrokenProcessPool) if a worker dies,
        # instead of waiting forever for its lost task.
        with cf.ProcessPoolExecutor(max_workers=min(workers, 16),
                                    mp_context=mp.get_context("spawn")) as ex:
            for ch, (cq, ck, cv) in zip(range(c0, c1), ex.map(_chunk_job, jobs)):
                a = max(t0, ch * CHUNK)
                b = min(t1, ch * CHUNK + cq.shape[0])
                s = a - ch * CHUNK
                q[a - t0:b - t0] = cq[s:s + b - a]
                k[a - t0:b - t0] = ck[s:s + b - a]
                v[a - t0:b - t0] = cv[s:s + b - a]
        return q, k, v
    else:
        cents = _centroids(w, layer, seed)
        parts = (_chunk(w, layer, seed, cents, ch) for ch in range(c0, c1))
    for ch, (cq, ck, cv) in zip(range(c0, c1), parts):
        a = max(t0, ch * CHUNK)
        b = min(t1, ch * CHUNK + cq.shape[0])
        s = a - ch * CHUNK
        q[a - t0:b - t0] = cq[s:s + b - a]
        k[a - t0:b - t0] = ck[s:s + b - a]
        v[a - t0:b - t0] = cv[s:s + b - a]
    return q, k, v
