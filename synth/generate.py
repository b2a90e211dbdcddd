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
   With planted topics (``topics`` > 0) the sequence is cut into segments of
   exponentially distributed length (mean ``topic_len`` tokens, boundaries
   at any token), each segment carries one of ``topics`` topics (never the
   same as the segment before), each topic owns a contiguous group of
   ``components / topics`` components, and every key and query of a segment
   draws its component id from that group only. On top of the mixture,
   every query head carries a fixed shared direction of norm
   ``shared_norm`` and every segment adds its topic's direction of norm
   ``topic_norm`` (one per topic and KV head, on the queries of that KV
   head's group and on its keys); both live in the lowest-frequency quarter
   of the rotary pairs, as the large low-frequency query components of
   trained models do, so sub-chunk fingerprints stay close within a topic,
   drift slowly with distance (the slow rotation of those pairs), and jump
   at a boundary. A drift in the same band, shared by all query heads, a stationary
   AR(1) process over knots 1024 tokens apart (stationary norm
   ``wobble_norm``, correlation ``wobble_corr`` from one knot to the next,
   linear between knots, moving in ``wobble_dims`` fixed random directions
   of the band), spreads the similarity of consecutive sub-chunks;
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
    topics: int = 0          # planted topics (0: none)
    topic_len: int = 0       # mean topic segment length in tokens
    topic_norm: float = 0.0  # norm of a topic's low-frequency direction
    shared_norm: float = 0.0  # norm of each query head's shared low-frequency direction
    wobble_norm: float = 0.0  # stationary norm of the low-frequency drift (all query heads)
    wobble_corr: float = 0.0  # its correlation from one 1024-token knot to the next
    wobble_dims: int = 0      # directions the drift moves in (0: the whole band)

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


# Token-level selection (block size 1, the paper's own rule) with the paper's
# k = 8192 tokens, on the 128K and 1M layers.
WORKLOADS["llama8b-128k-tok"] = WORKLOADS["llama8b-128k"].replace(name="llama8b-128k-tok", block_size=1,
                                                                 top_k=8192)
WORKLOADS["llama8b-1m-tok"] = WORKLOADS["llama8b-1m"].replace(name="llama8b-1m-tok", block_size=1, top_k=8192)

# Planted-topic variant for the clustering-threshold sweep: the paper's sub-chunk
# L = 512 and outer chunk 8192, k = 64 blocks of 128 = 8192 tokens, 128K context.
WORKLOADS["llama8b-128k-topics"] = Workload(
    "llama8b-128k-topics", 32, 8, 128, 131072, 512, 8, 8192, 128, 64, 128, 512, 256, 500000.0, False,
    theta=0.95, topics=16, topic_len=16384, topic_norm=3.0, shared_norm=6.0, wobble_norm=4.0,
    wobble_corr=0.96, wobble_dims=2)


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


def topic_segments(w: Workload, layer: int, seed: int):
    """(segment start tokens, topic of each segment) for planted topics."""
    rng = np.random.default_rng([seed, layer, 4])
    starts, topics = [0], [int(rng.integers(0, w.topics))]
    while True:
        nxt = starts[-1] + 1 + int(rng.exponential(w.topic_len))
        if nxt >= w.n_tokens:
            break
        t = int(rng.integers(0, w.topics - 1))
        starts.append(nxt)
        topics.append(t if t < topics[-1] else t + 1)  # a different topic
    return np.array(starts, np.int64), np.array(topics, np.int64)


def _low_band(w: Workload) -> np.ndarray:
    """Dims of the lowest-frequency quarter of the rotate-half rotary pairs."""
    half = w.head_dim // 2
    pairs = np.arange(half - half // 4, half)
    return np.concatenate([pairs, pairs + half])


def _topic_dirs(w: Workload, layer: int, seed: int):
    """(shared [H_q, d_h], topic [topics, H_kv, d_h]) low-frequency directions."""
    rng = np.random.default_rng([seed, layer, 5])
    band = _low_band(w)
    shared = np.zeros((w.num_q_heads, w.head_dim))
    shared[:, band] = _unit_rows(rng.standard_normal((w.num_q_heads, band.size))) * w.shared_norm
    topic = np.zeros((w.topics, w.num_kv_heads, w.head_dim))
    topic[:, :, band] = _unit_rows(rng.standard_normal((w.topics, w.num_kv_heads, band.size))) * w.topic_norm
    return shared.astype(np.float32), topic.astype(np.float32)


WOBBLE_KNOT = 1024


def _wobble(w: Workload, layer: int, seed: int, pos: np.ndarray) -> np.ndarray:
    """Low-frequency drift [T, 1, d_h] (the same for every query head) at positions pos."""
    rng = np.random.default_rng([seed, layer, 6])
    band = _low_band(w)
    r = w.wobble_dims or band.size
    basis = np.linalg.qr(rng.standard_normal((band.size, r)))[0]  # orthonormal columns
    n_knots = w.n_tokens // WOBBLE_KNOT + 2
    sd = w.wobble_norm / np.sqrt(r)
    a = w.wobble_corr
    z = rng.standard_normal((n_knots, 1, r))
    knots = np.empty_like(z)
    knots[0] = sd * z[0]
    for j in range(1, n_knots):
        knots[j] = a * knots[j - 1] + np.sqrt(1.0 - a * a) * sd * z[j]
    j = pos // WOBBLE_KNOT
    f = ((pos % WOBBLE_KNOT) / WOBBLE_KNOT)[:, None, None]
    out = np.zeros((pos.size, 1, w.head_dim), np.float32)
    out[:, :, band] = (((1.0 - f) * knots[j] + f * knots[j + 1]) @ basis.T).astype(np.float32)
    return out


def _component_ids(w: Workload, rng, shape, pos, segs):
    if not w.topics:
        return rng.integers(0, w.components, size=shape)
    group = w.components // w.topics
    starts, topics = segs
    topic = topics[np.searchsorted(starts, pos, side="right") - 1]
    return topic[:, None] * group + rng.integers(0, group, size=shape)


def _chunk(w: Workload, layer: int, seed: int, cents, ch: int):
    t0 = ch * CHUNK
    t1 = min(w.n_tokens, t0 + CHUNK)
    T = t1 - t0
    pos = np.arange(t0, t1, dtype=np.int64)
    kvh = np.arange(w.num_kv_heads)
    qkv = np.arange(w.num_q_heads) // w.group

    segs = topic_segments(w, layer, seed) if w.topics else None
    rk = np.random.default_rng([seed, layer, 1, ch])
    kid = _component_ids(w, rk, (T, w.num_kv_heads), pos, segs)
    k = _mix(w, cents, kvh, kid, pos) + rk.standard_normal((T, w.num_kv_heads, w.head_dim), dtype=np.float32)

    rq = np.random.default_rng([seed, layer, 2, ch])
    qid = _component_ids(w, rq, (T, w.num_q_heads), pos, segs)
    q = _mix(w, cents, qkv, qid, pos) + rq.standard_normal((T, w.num_q_heads, w.head_dim), dtype=np.float32)

    if w.topics:
        shared, topic = _topic_dirs(w, layer, seed)
        starts, tops = segs
        tp = tops[np.searchsorted(starts, pos, side="right") - 1]
        k = k + topic[tp]
        q = q + shared[None] + topic[tp][:, qkv]
        if w.wobble_norm:
            q = q + _wobble(w, layer, seed, pos)

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
