"""GPU parity of every step of the SCR path against the CPU fp64 oracle.

All calls go through the C ABI (libscale.so via the ctypes binding). Inputs
are the seeded synthetic tensors of ``synth``; expected values come from
``oracle`` only.
"""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_31568_gb300 as pkg
from paper_2609_31568_gb300 import scale as S
from _util import (ATTN_MAX_ABS, ATTN_MEAN_ABS, NEAR_TIE_GAP, attn_errors, compare_selection,
                   inputs, last_query_blocks, sample_rows, selection_for_reference, to_f64_bf16)

pytestmark = pytest.mark.gpu

PER_CLUSTER, PER_SUB = S.SCALE_MODE_PER_CLUSTER, S.SCALE_MODE_PER_SUBCHUNK

# Small cases that span several tiles and end in ragged pieces.
RAGGED = dict(n_tokens=3000, block_size=48, n_sink=40, n_local=100, top_k=6)
# Ragged too, with a window of whole 128-row tiles: the host call runs in pieces.
RAGGED_PIECES = dict(n_tokens=3000, block_size=48, n_sink=40, n_local=128, top_k=6)
GQA_SMALL = dict(n_tokens=8192 + 333, sub_chunk=512, max_cluster_subchunks=4, outer_chunk=2048,
                 top_k=8)


@pytest.fixture(scope="session", autouse=True)
def _built():
    pkg.build()
    S.load()


def gpu_path(w, mode, dev, want_scores=True, **over):
    p = S.params_for(w, **over)
    buf = S.allocate(p, mode, want_scores=want_scores)
    S.run_path(p, mode, *dev, buf)
    torch.cuda.synchronize()
    assert S.scale_get_device_status(buf.ws) == S.SCALE_OK
    return p, buf


def oracle_path(w, q, k, v, mode, rows=None, **over):
    ww = w.replace(**over) if over else w
    return oracle.run_path(ww, q, k, v, per_subchunk=(mode == PER_SUB), rows=rows)


def unit_count(buf, mode, w):
    return w.n_subchunks if mode == PER_SUB else int(buf.n_units.item())


# --------------------------------------------------------------------------- step (a)


@pytest.mark.parametrize("name,over", [("gqa4-4k", {}), ("gqa4-4k", RAGGED),
                                       ("llama8b-32k", GQA_SMALL), ("llama8b-32k", {})])
def test_build_reps_parity(name, over):
    w, q, k, v, dev = inputs(name, **over)
    p, buf = gpu_path(w, PER_CLUSTER, dev)
    ref = oracle_path(w, q, k, v, PER_CLUSTER)
    reps = buf.reps.cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(reps, ref["reps"], rtol=0, atol=2e-5)
    fp = buf.fingerprints.cpu().numpy().astype(np.float64)
    np.testing.assert_allclose(fp, ref["fingerprints"], rtol=0, atol=2e-5)
    n = int(buf.n_units.item())
    assert buf.unit_start[: n + 1].cpu().numpy().tolist() == ref["unit_start"].tolist()
    assert np.all(buf.unit_start[n + 1:].cpu().numpy() == w.n_subchunks)


def _robust_theta(fp: np.ndarray, norms: np.ndarray, w) -> float:
    """A threshold between observed anchor-candidate cosines, far (>1e-4) from all of them."""
    vt = fp / norms[:, None]
    per = w.outer_chunk // w.sub_chunk
    cs = []
    for i in range(len(vt)):
        for d in range(1, w.max_cluster_subchunks):
            j = i + d
            if j < len(vt) and j // per == i // per:
                cs.append(float(vt[i] @ vt[j]))
    cs = np.sort(np.array(cs))
    mid = len(cs) // 2
    gaps = np.diff(cs)
    window = range(max(0, mid - len(cs) // 4), min(len(gaps), mid + len(cs) // 4 + 1))
    best = max(window, key=lambda i: gaps[i])
    assert gaps[best] > 2e-4
    return float(cs[best] + gaps[best] / 2)


@pytest.mark.parametrize("name,over", [("gqa4-4k", dict(max_cluster_subchunks=4)),
                                       ("llama8b-32k", GQA_SMALL)])
def test_threshold_clustering_parity(name, over):
    w, q, k, v, dev = inputs(name, **over)
    fp, norms = oracle.fingerprints(q, w.sub_chunk)
    theta = _robust_theta(fp, norms, w)
    ref_us, margin = oracle.anchor_clustering(fp, norms, w.max_cluster_subchunks,
                                              w.outer_chunk // w.sub_chunk, theta)
    assert margin > 1e-4
    p, buf = gpu_path(w, PER_CLUSTER, dev, theta=theta)
    n = int(buf.n_units.item())
    got = buf.unit_start[: n + 1].cpu().numpy()
    assert got.tolist() == ref_us.tolist()
    assert 1 < n < w.n_subchunks or len(ref_us) - 1 == n


# --------------------------------------------------------------------------- steps (b), (c)


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
@pytest.mark.parametrize("name,over", [("gqa4-4k", {}), ("gqa4-4k", RAGGED),
                                       ("llama8b-32k", {}), ("llama8b-128k", {})])
def test_select_parity(name, over, mode):
    w, q, k, v, dev = inputs(name, **over)
    p, buf = gpu_path(w, mode, dev)
    ref = oracle.run_path(w, q, k, v, per_subchunk=(mode == PER_SUB))
    n = unit_count(buf, mode, w)
    assert n == len(ref["sel_count"])
    sel = buf.sel_blocks.cpu().numpy()[:n, : w.top_k]
    cnt = buf.sel_count.cpu().numpy()[:n]
    same, near = compare_selection(sel, cnt, ref)
    # the soft-vote scores themselves, on the candidates
    ref_sc = oracle.select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
                           block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink,
                           n_local=w.n_local, select_scale=1.0, per_subchunk=(mode == PER_SUB),
                           reps=ref["reps"], v=ref["fingerprints"], unit_start=ref["unit_start"],
                           want_scores=True)["scores"]
    got_sc = buf.sel_scores.cpu().numpy()[:n].astype(np.float64)
    cand = ~np.isnan(ref_sc)
    assert np.array_equal(cand, ~np.isnan(got_sc))
    np.testing.assert_allclose(got_sc[cand], ref_sc[cand], rtol=2e-5, atol=1e-6)
    print(f"{name} mode={mode}: {n} units, {int((cnt > 0).sum())} retrievals, "
          f"{near} near-tie units differ (gap < {NEAR_TIE_GAP})")


# --------------------------------------------------------------------------- step (d)


def _prefill_on(w, mode, dev, unit_start, n_units, sel, cnt, **over):
    p = S.params_for(w, **over)
    ws = torch.empty(S.scale_workspace_size(p, mode), dtype=torch.uint8, device="cuda")
    S.scale_workspace_init(ws)
    out = torch.zeros((w.n_tokens, w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
    k = max(w.top_k, 1)
    M = w.n_subchunks
    sel_full = np.full((M, k), -1, np.int32)
    cnt_full = np.zeros(M, np.int32)
    sel_full[: sel.shape[0], : sel.shape[1]] = sel
    cnt_full[: len(cnt)] = cnt
    us = torch.from_numpy(np.ascontiguousarray(unit_start, np.int32)).cuda()
    nu = torch.tensor([n_units], dtype=torch.int32, device="cuda")
    S.scale_sparse_prefill(p, mode, 0, w.n_tokens, *dev, us, nu,
                           torch.from_numpy(sel_full).cuda(), torch.from_numpy(cnt_full).cuda(), out, ws)
    torch.cuda.synchronize()
    assert S.scale_get_device_status(ws) == S.SCALE_OK
    return out


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
@pytest.mark.parametrize("name,over,stride", [
    ("gqa4-4k", {}, 1),
    ("gqa4-4k", RAGGED, 1),
    ("gqa4-4k", dict(top_k=0, n_sink=0), 1),
    ("gqa4-4k", dict(block_size=256, top_k=2, n_sink=128, n_local=0), 1),
    ("llama8b-32k", GQA_SMALL, 5),
    # query-head groups of 2, 8, 3 and 7 (the last head of an odd group runs
    # in a CTA of its own with one query tile)
    ("gqa4-4k", dict(num_q_heads=8, num_kv_heads=4, n_tokens=2048 + 64), 1),
    ("gqa4-4k", dict(num_q_heads=16, num_kv_heads=2, n_tokens=2048 + 64), 1),
    ("gqa4-4k", dict(num_q_heads=6, num_kv_heads=2, n_tokens=2048 + 64), 1),
    ("gqa4-4k", dict(num_q_heads=7, num_kv_heads=1, n_tokens=2048 + 64), 1),
])
def test_attention_parity_on_oracle_selection(name, over, stride, mode):
    """scale_sparse_prefill on the oracle's selection vs the oracle's Eq. 10,
    for every row, including query-head groups of odd size."""
    w, q, k, v, dev = inputs(name, **over)
    rows = np.arange(0, w.n_tokens, stride)
    ref = oracle_path(w, q, k, v, mode, rows=rows)
    us = ref["unit_start"] if mode == PER_CLUSTER else np.arange(w.n_subchunks + 1, dtype=np.int32)
    out = _prefill_on(w, mode, dev, us, len(us) - 1, ref["sel"], ref["sel_count"])
    got = to_f64_bf16(out[torch.from_numpy(rows).cuda()])
    mx, mean = attn_errors(got, ref["attn"])
    print(f"{name} {over} mode={mode}: max {mx:.3e} mean {mean:.3e}")
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
def test_qwen2_7b_head_shape_end_to_end(mode):
    """The head layout of the paper's model (Qwen2-7B: 28 query heads on 4 KV
    heads, groups of 7) through all four steps: unit table, selection (exact
    except near-ties) and every attention row against the oracle."""
    w, q, k, v, dev = inputs("gqa4-4k", num_q_heads=28, num_kv_heads=4, n_tokens=2048 + 96)
    p, buf = gpu_path(w, mode, dev)
    ref = oracle_path(w, q, k, v, mode)
    n = unit_count(buf, mode, w)
    if mode == PER_CLUSTER:
        assert buf.unit_start[: n + 1].cpu().numpy().tolist() == ref["unit_start"].tolist()
    sel = buf.sel_blocks.cpu().numpy()[:n, : w.top_k]
    same, near = compare_selection(sel, buf.sel_count.cpu().numpy()[:n], ref)
    rows = np.arange(w.n_tokens)
    us = ref["unit_start"] if mode == PER_CLUSTER else np.arange(w.n_subchunks + 1, dtype=np.int32)
    ref_attn = oracle.attention_rows(q=q, k=k, v=v, sub_chunk=w.sub_chunk, block_size=w.block_size,
                                     top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                                     attn_scale=1.0 / np.sqrt(w.head_dim), per_subchunk=(mode == PER_SUB),
                                     unit_start=ref["unit_start"], sel=selection_for_reference(sel, ref, same),
                                     sel_count=ref["sel_count"], rows=rows)
    mx, mean = attn_errors(to_f64_bf16(buf.out), ref_attn)
    print(f"28q/4kv mode={mode}: {n} units, {near} near-ties, max {mx:.3e} mean {mean:.3e} ({len(us) - 1} units)")
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


# bf16 spike key values 14.0, 22.0 and 32.0: against a query coordinate of 8
# the spike's logit lies about 12, 20 and 30 log2 units above the rows' other
# logits. The first stays on the softmax's fast path (every p of the tile at
# most 2^16, the running max kept), the others fail its sum test and take the
# exact path (raise, O rescale).
SPIKES = (0x4160, 0x41B0, 0x4200)


@pytest.mark.parametrize("spike", SPIKES)
@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
def test_attention_max_jump_in_alternate_rows(mode, spike):
    """Rows whose running max jumps in a later key tile next to rows whose max
    does not: even rows get a large score against a few spike keys (the online
    softmax of Sec. V-A3 must raise their max and rescale their partial sums,
    or keep a lower max with large terms), odd rows score exactly 0 against
    them. Both kinds of row share each group of 32 consecutive rows."""
    w, q, k, v, _ = inputs("gqa4-4k")
    q = q.copy()
    k = k.copy()
    spikes = np.arange(200, w.n_tokens, 512)
    k[spikes] = 0
    k[spikes, :, 0] = spike
    q[0::2, :, 0] = 0x4100    # bf16 8.0: score 8 x spike against a spike key
    q[1::2, :, 0] = 0         # score 0 against a spike key
    dev = [torch.from_numpy(x).view(torch.bfloat16).cuda() for x in (q, k, v)]
    rows = np.arange(w.n_tokens)
    ref = oracle_path(w, q, k, v, mode, rows=rows)
    us = ref["unit_start"] if mode == PER_CLUSTER else np.arange(w.n_subchunks + 1, dtype=np.int32)
    out = _prefill_on(w, mode, dev, us, len(us) - 1, ref["sel"], ref["sel_count"])
    got = to_f64_bf16(out)
    mx, mean = attn_errors(got, ref["attn"])
    print(f"mode={mode} spike={spike:#x}: max {mx:.3e} mean {mean:.3e}")
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


def _heavy_units(w, mode, n_units):
    """Units whose last query block is checked row by row: every cluster in SCR
    mode; in per-sub-chunk mode the last sub-chunk of every outer chunk."""
    if mode == PER_CLUSTER:
        return list(range(n_units))
    per = w.outer_chunk // w.sub_chunk
    return [u for u in range(n_units) if (u + 1) % per == 0 or u == n_units - 1]


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
@pytest.mark.parametrize("name,n_random,heavy", [("llama8b-32k", 16, False), ("llama8b-128k", 8, True)])
def test_end_to_end_parity_sampled(name, n_random, heavy, mode):
    """All four steps on the GPU at the workload's full size; selection compared
    unit by unit; attention on sampled rows of every unit against the oracle's
    Eq. 10 run on the selection the GPU used (the oracle's own where the two
    agree, the GPU's where they differ at a near-tie). At 128K every row of
    the last 128-row query block of each cluster is added, all heads: those
    rows have the longest window."""
    w, q, k, v, dev = inputs(name)
    p, buf = gpu_path(w, mode, dev)
    ref = oracle_path(w, q, k, v, mode)
    n = unit_count(buf, mode, w)
    sel = buf.sel_blocks.cpu().numpy()[:n, : w.top_k]
    cnt = buf.sel_count.cpu().numpy()[:n]
    same, near = compare_selection(sel, cnt, ref)
    us = ref["unit_start"] if mode == PER_CLUSTER else np.arange(w.n_subchunks + 1, dtype=np.int32)
    rows = sample_rows(w, us, n_random)
    n_heavy = 0
    if heavy:
        extra = last_query_blocks(w, us, _heavy_units(w, mode, n))
        n_heavy = len(extra)
        rows = np.union1d(rows, extra)
    ref_attn = oracle.attention_rows(q=q, k=k, v=v, sub_chunk=w.sub_chunk, block_size=w.block_size,
                                     top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                                     attn_scale=1.0 / np.sqrt(w.head_dim),
                                     per_subchunk=(mode == PER_SUB), unit_start=ref["unit_start"],
                                     sel=selection_for_reference(sel, ref, same),
                                     sel_count=ref["sel_count"], rows=rows)
    got = to_f64_bf16(buf.out[torch.from_numpy(rows).cuda()])
    mx, mean = attn_errors(got, ref_attn)
    print(f"{name} mode={mode}: {len(rows)} rows ({n_heavy} in last query blocks), max {mx:.3e} "
          f"mean {mean:.3e}, {near} near-tie units (checked on the GPU's selection)")
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


# --------------------------------------------------------------------------- token level (B = 1)

TOKEN_CASES = [("gqa4-4k", dict(block_size=1, top_k=64)),
               ("gqa4-4k", dict(block_size=1, n_tokens=3000, n_sink=40, n_local=100, top_k=50)),
               ("llama8b-32k", dict(block_size=1, top_k=1024)),
               # the paper's model and selection: Qwen2-7B heads (28 on 4 KV heads), token level
               ("gqa4-4k", dict(block_size=1, top_k=128, num_q_heads=28, num_kv_heads=4, n_tokens=2048 + 64)),
               ("gqa4-4k", dict(block_size=1, top_k=96, num_q_heads=6, num_kv_heads=2, n_tokens=2048 + 64)),
               ("gqa4-4k", dict(block_size=1, top_k=64, num_q_heads=16, num_kv_heads=2, n_tokens=2048 + 64))]


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
@pytest.mark.parametrize("name,over", TOKEN_CASES + [("llama8b-128k-tok", {})])
def test_token_select_parity(name, over, mode):
    """scale_select_tokens (tensor-core scores from K, per-head softmax, soft
    vote, top-k of tokens) against the oracle's Eq. 9 at block size 1."""
    w, q, k, v, dev = inputs(name, **over)
    p, buf = gpu_path(w, mode, dev)
    ref = oracle.run_path(w, q, k, v, per_subchunk=(mode == PER_SUB))
    n = unit_count(buf, mode, w)
    sel = buf.sel_blocks.cpu().numpy()[:n, : w.top_k]
    cnt = buf.sel_count.cpu().numpy()[:n]
    same, near = compare_selection(sel, cnt, ref)
    ref_sc = oracle.select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
                           block_size=1, top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                           select_scale=1.0, per_subchunk=(mode == PER_SUB), reps=ref["reps"],
                           v=ref["fingerprints"], unit_start=ref["unit_start"], want_scores=True)["scores"]
    got_sc = buf.sel_scores.cpu().numpy()[:n].astype(np.float64)
    cand = ~np.isnan(ref_sc)
    assert np.array_equal(cand, ~np.isnan(got_sc))
    np.testing.assert_allclose(got_sc[cand], ref_sc[cand], rtol=2e-5, atol=1e-10)
    print(f"{name} {over} mode={mode}: {n} units, {near} near-tie units differ")


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
@pytest.mark.parametrize("name,over,stride", [(nm, ov, 1 if nm == "gqa4-4k" else 5) for nm, ov in TOKEN_CASES])
def test_token_attention_parity_on_oracle_selection(name, over, stride, mode):
    """scale_sparse_prefill at block size 1 (distant keys gathered row by row)
    on the oracle's token selection vs the oracle's Eq. 10."""
    w, q, k, v, dev = inputs(name, **over)
    rows = np.arange(0, w.n_tokens, stride)
    ref = oracle_path(w, q, k, v, mode, rows=rows)
    us = ref["unit_start"] if mode == PER_CLUSTER else np.arange(w.n_subchunks + 1, dtype=np.int32)
    out = _prefill_on(w, mode, dev, us, len(us) - 1, ref["sel"], ref["sel_count"])
    got = to_f64_bf16(out[torch.from_numpy(rows).cuda()])
    mx, mean = attn_errors(got, ref["attn"])
    print(f"{name} {over} mode={mode}: max {mx:.3e} mean {mean:.3e}")
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
def test_token_select_range_calls_long_sequence(mode):
    """Token-level selection by range calls, one outer chunk per call as the
    Algorithm 2 loop issues them, on a sequence with 1024 token ranges (128K
    tokens, one query head per KV head): the few-unit scorer then keeps whole
    ranges and all KV heads in each CTA, and the later units have more than
    64K candidates (the multi-CTA top-k). Every unit's scores and selection
    against the oracle's Eq. 9 and top-k."""
    w, q, k, v, dev = inputs("llama8b-128k-tok", num_q_heads=8, num_kv_heads=8)
    p = S.params_for(w)
    buf = S.allocate(p, mode, want_scores=True)
    for t0 in range(0, w.n_tokens, w.outer_chunk):
        t1 = min(w.n_tokens, t0 + w.outer_chunk)
        S.scale_build_reps_range(p, t0, t1, dev[0], dev[1], buf.reps, buf.fingerprints, buf.unit_start,
                                 buf.n_units, buf.ws)
        S.select(p, mode, t0, t1, dev[1], buf)
    torch.cuda.synchronize()
    assert S.scale_get_device_status(buf.ws) == S.SCALE_OK
    ref = oracle.run_path(w, q, k, v, per_subchunk=(mode == PER_SUB))
    n = unit_count(buf, mode, w)
    assert n == len(ref["sel_count"])
    same, near = compare_selection(buf.sel_blocks.cpu().numpy()[:n, : w.top_k], buf.sel_count.cpu().numpy()[:n],
                                   ref)
    ref_sc = oracle.select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
                           block_size=1, top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                           select_scale=1.0, per_subchunk=(mode == PER_SUB), reps=ref["reps"],
                           v=ref["fingerprints"], unit_start=ref["unit_start"], want_scores=True)["scores"]
    got_sc = buf.sel_scores.cpu().numpy()[:n].astype(np.float64)
    cand = ~np.isnan(ref_sc)
    assert np.array_equal(cand, ~np.isnan(got_sc))
    np.testing.assert_allclose(got_sc[cand], ref_sc[cand], rtol=2e-5, atol=1e-10)
    print(f"mode={mode}: {n} units, {near} near-tie units differ")


def test_token_attention_ignores_invalid_entries():
    """Selected tokens outside [n_sink, W_u), repeated or out of order are
    ignored, as scale_sparse_prefill documents: the result equals the one on
    the cleaned selection."""
    w, q, k, v, dev = inputs("gqa4-4k", block_size=1, top_k=64)
    ref = oracle_path(w, q, k, v, PER_CLUSTER)
    us = ref["unit_start"]
    clean = _prefill_on(w, PER_CLUSTER, dev, us, len(us) - 1, ref["sel"], ref["sel_count"])
    dirty = ref["sel"].copy()
    cnt = ref["sel_count"].copy()
    for u in range(len(cnt)):
        c = int(cnt[u])
        if c >= 4:
            dirty[u, 1] = dirty[u, 0]          # repeat (not above its predecessor)
            dirty[u, c - 1] = w.n_tokens + 5   # beyond the window
    bad = _prefill_on(w, PER_CLUSTER, dev, us, len(us) - 1, dirty, cnt)
    cleaned = [[t for i, t in enumerate(dirty[u, : cnt[u]])
                if w.n_sink <= t < max(0, us[u] * w.sub_chunk - w.n_local) and (i == 0 or t > dirty[u, i - 1])]
               for u in range(len(cnt))]
    sel2 = np.full_like(dirty, -1)
    cnt2 = np.array([len(x) for x in cleaned], np.int32)
    for u, x in enumerate(cleaned):
        sel2[u, : len(x)] = x
    ref2 = _prefill_on(w, PER_CLUSTER, dev, us, len(us) - 1, sel2, cnt2)
    assert torch.equal(bad, ref2)
    assert not torch.equal(bad, clean)


def test_1m_tokens_full_size():
    """Token-level selection at 1M tokens with k = 8192 (SCR): every unit's
    selection and sampled attention rows against the oracle."""
    from synth import generate_layer, workload

    w = workload("llama8b-1m-tok")
    q, k, v = generate_layer(w)
    n, mx, mean, near = _full_size_check(w, q, k, v, PER_CLUSTER, n_random=24)
    print(f"1M tokens: {n} rows, max {mx:.3e} mean {mean:.3e}, {near} near-tie units")
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


# --------------------------------------------------------------------------- threshold sweep


@pytest.mark.parametrize("s_max,theta", [(4, 0.97), (8, 0.95), (8, 0.99)])
def test_planted_topic_sweep_parity(s_max, theta):
    """Alg. 1 with a real threshold on planted-topic data (32K tokens, L = 512):
    the GPU's clusters, the anchors' selections, every member's selection
    against the cluster's candidates, and the overlap ratio of Sec. IV-C match
    the oracle."""
    from paper_2609_31568_gb300 import fidelity as F

    w, q, k, v, dev = inputs("llama8b-128k-topics", n_tokens=32768, max_cluster_subchunks=s_max,
                             theta=theta)
    p, buf = gpu_path(w, PER_CLUSTER, dev)
    ref = oracle_path(w, q, k, v, PER_CLUSTER)
    assert ref["margin"] > 1e-5  # every admission decision is far from theta in fp32 terms
    n = int(buf.n_units.item())
    us = buf.unit_start[: n + 1].cpu().numpy()
    assert us.tolist() == ref["unit_start"].tolist()
    assert 1 < n < w.n_subchunks
    sel = buf.sel_blocks.cpu().numpy()[:n, : w.top_k]
    cnt = buf.sel_count.cpu().numpy()[:n]
    same, _ = compare_selection(sel, cnt, ref)
    gpu_m, ref_m = {}, {}
    for j in range(1, s_max):
        fpj = F.member_query_fingerprints(buf.fingerprints, buf.unit_start, n, j)
        sj, cj = torch.empty_like(buf.sel_blocks), torch.empty_like(buf.sel_count)
        S.scale_select(p, PER_CLUSTER, 0, w.n_tokens, buf.reps, fpj, buf.unit_start, buf.n_units,
                       sj, cj, None, buf.ws)
        torch.cuda.synchronize()
        assert S.scale_get_device_status(buf.ws) == S.SCALE_OK
        r = oracle.member_selection(w, ref["reps"], ref["fingerprints"], ref["unit_start"], j)
        gpu_m[j] = (sj.cpu().numpy()[:n, : w.top_k], cj.cpu().numpy()[:n])
        ref_m[j] = r
        ok_j, _ = compare_selection(*gpu_m[j], r)
        same &= ok_j
    rho, units = F.overlap_ratios(us, sel, cnt, lambda u, j: gpu_m[j][0][u, : gpu_m[j][1][u]])
    sizes = np.diff(ref["unit_start"])
    for r_gpu, u in zip(rho, units):
        if not same[u]:
            continue  # a near-tie changed one of the selections involved
        want = oracle.overlap_ratio(ref["sel"][u, : ref["sel_count"][u]],
                                    [ref_m[j]["sel"][u, : ref_m[j]["sel_count"][u]] for j in range(1, sizes[u])])
        assert r_gpu == want
    assert len(units) == int(np.count_nonzero((sizes >= 2) & (ref["sel_count"] > 0)))
    print(f"L_max={s_max}L theta={theta}: {n} units, rho min {rho.min():.3f} median {np.median(rho):.3f}")


# --------------------------------------------------------------------------- invariants


def test_size_one_clusters_equal_per_subchunk_mode():
    w, q, k, v, dev = inputs("gqa4-4k", max_cluster_subchunks=1)
    _, a = gpu_path(w, PER_CLUSTER, dev)
    _, b = gpu_path(w, PER_SUB, dev)
    assert int(a.n_units.item()) == w.n_subchunks
    assert torch.equal(a.sel_blocks, b.sel_blocks) and torch.equal(a.sel_count, b.sel_count)
    assert torch.equal(a.out, b.out)


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
def test_outer_chunk_loop_equals_one_call(mode):
    """Algorithm 2 runs per outer chunk; calling select + attention chunk by chunk
    gives the same bits as one call over all tokens."""
    w, q, k, v, dev = inputs("llama8b-32k", **GQA_SMALL)
    p, whole = gpu_path(w, mode, dev)
    buf = S.allocate(p, mode, want_scores=True)
    S.scale_build_reps(p, dev[0], dev[1], buf.reps, buf.fingerprints, buf.unit_start, buf.n_units, buf.ws)
    buf.out.zero_()
    step = w.outer_chunk
    for t0 in range(0, w.n_tokens, step):
        t1 = min(w.n_tokens, t0 + step)
        S.scale_select(p, mode, t0, t1, buf.reps, buf.fingerprints, buf.unit_start, buf.n_units,
                       buf.sel_blocks, buf.sel_count, buf.sel_scores, buf.ws)
        S.scale_sparse_prefill(p, mode, t0, t1, *dev, buf.unit_start, buf.n_units, buf.sel_blocks,
                               buf.sel_count, buf.out, buf.ws)
    torch.cuda.synchronize()
    n = unit_count(whole, mode, w)
    assert torch.equal(whole.sel_blocks[:n], buf.sel_blocks[:n])
    assert torch.equal(whole.out, buf.out)


def test_deterministic_bits():
    w, q, k, v, dev = inputs("llama8b-32k", **GQA_SMALL)
    _, a = gpu_path(w, PER_CLUSTER, dev)
    _, b = gpu_path(w, PER_CLUSTER, dev)
    n = int(a.n_units.item())
    assert n == int(b.n_units.item())
    # bit patterns (scores hold NaN off the candidates; rows past n_units are unused)
    for x, y in ((a.reps, b.reps), (a.fingerprints, b.fingerprints), (a.unit_start, b.unit_start),
                 (a.sel_blocks[:n], b.sel_blocks[:n]), (a.sel_count[:n], b.sel_count[:n]),
                 (a.sel_scores[:n], b.sel_scores[:n]), (a.out, b.out)):
        assert torch.equal(x.view(torch.int32) if x.dtype == torch.float32 else x,
                           y.view(torch.int32) if y.dtype == torch.float32 else y)


@pytest.mark.parametrize("over", [RAGGED, RAGGED_PIECES, dict(block_size=1, top_k=64)])
def test_prefill_host_matches_device_path(over):
    """scale_prefill_host (host buffers in and out) gives the device path's
    output bit for bit, at block level and at token level, whether it runs as
    one piece (a window that is not whole tiles) or in pieces of outer chunks
    overlapped with the copies."""
    w, q, k, v, dev = inputs("gqa4-4k", **over)
    for mode in (PER_CLUSTER, PER_SUB):
        p, buf = gpu_path(w, mode, dev, want_scores=False)
        arena = torch.empty(S.scale_prefill_host_arena_size(p, mode), dtype=torch.uint8, device="cuda")
        out = np.empty((w.n_tokens, w.num_q_heads, w.head_dim), np.uint16)
        S.scale_prefill_host(p, mode, q, k, v, out, arena)
        assert np.array_equal(out, buf.out.view(torch.int16).cpu().numpy().view(np.uint16))


@pytest.mark.parametrize("over", [RAGGED_PIECES, dict(block_size=1, top_k=64)])
def test_range_calls_read_no_row_past_the_range(over):
    """Chunked prefill (Sec. III-B) with the range calls: the device copies of
    Q, K and V start as NaN and the rows of each outer chunk arrive just before
    its calls. A read of any row past the range would put NaN into the
    representatives, the fingerprints, the scores or (through P = 0 times a NaN
    value row) the output; the results must equal the whole-sequence calls bit
    for bit, including the unit table that the ranges build by appending."""
    w, q, k, v, dev = inputs("gqa4-4k", **over)
    for mode in (PER_CLUSTER, PER_SUB):
        p, whole = gpu_path(w, mode, dev, want_scores=False)
        late = [torch.full_like(x, float("nan")) for x in dev]
        buf = S.allocate(p, mode)
        buf.out.fill_(float("nan"))  # every row must be written by its own range
        for t0 in range(0, w.n_tokens, w.outer_chunk):
            t1 = min(w.n_tokens, t0 + w.outer_chunk)
            for dst, src in zip(late, dev):
                dst[t0:t1].copy_(src[t0:t1])
            S.scale_build_reps_range(p, t0, t1, late[0], late[1], buf.reps, buf.fingerprints,
                                     buf.unit_start, buf.n_units, buf.ws)
            S.select(p, mode, t0, t1, late[1], buf)
            S.scale_sparse_prefill(p, mode, t0, t1, *late, buf.unit_start, buf.n_units, buf.sel_blocks,
                                   buf.sel_count, buf.out, buf.ws)
        torch.cuda.synchronize()
        assert S.scale_get_device_status(buf.ws) == S.SCALE_OK
        n = unit_count(whole, mode, w)
        assert int(buf.n_units.item()) == int(whole.n_units.item())
        assert torch.equal(buf.unit_start, whole.unit_start)
        assert torch.equal(buf.fingerprints.view(torch.int32), whole.fingerprints.view(torch.int32))
        if whole.reps is not None:
            assert torch.equal(buf.reps.view(torch.int32), whole.reps.view(torch.int32))
        assert torch.equal(buf.sel_count[:n], whole.sel_count[:n])
        assert torch.equal(buf.sel_blocks[:n], whole.sel_blocks[:n])
        assert torch.equal(buf.out.view(torch.int16), whole.out.view(torch.int16))


def test_range_calls_reject_ranges_off_the_outer_chunks():
    w, q, k, v, dev = inputs("gqa4-4k")
    p = S.params_for(w)
    buf = S.allocate(p, PER_CLUSTER)
    for t0, t1 in ((256, 2048), (0, 1000), (1024, 512), (0, w.n_tokens + 1024)):
        with pytest.raises(S.ScaleError) as e:
            S.scale_build_reps_range(p, t0, t1, dev[0], dev[1], buf.reps, buf.fingerprints,
                                     buf.unit_start, buf.n_units, buf.ws)
        assert e.value.rc == S.SCALE_ERR_INVALID_ARG


def test_wait_timeout_is_reported_and_context_survives():
    w, q, k, v, dev = inputs("gqa4-4k")
    p = S.params_for(w)
    ws = torch.empty(S.scale_workspace_size(p, PER_CLUSTER), dtype=torch.uint8, device="cuda")
    S.scale_workspace_init(ws)
    S.scale_selftest_wait_timeout(ws, 1_000_000)  # 1 ms on a barrier nothing arrives at
    assert S.scale_get_device_status(ws) == S.SCALE_ERR_TIMEOUT
    S.scale_workspace_init(ws)
    assert S.scale_get_device_status(ws) == S.SCALE_OK
    _, buf = gpu_path(w, PER_CLUSTER, dev)  # the context is still usable
    assert torch.isfinite(buf.out.float()).all()


def test_invalid_arguments_are_rejected_before_launch():
    w, q, k, v, dev = inputs("gqa4-4k")
    p = S.params_for(w)
    buf = S.allocate(p, PER_CLUSTER)
    host_q = torch.from_numpy(q).view(torch.bfloat16)
    with pytest.raises(S.ScaleError) as e:
        S.scale_build_reps(p, host_q, dev[1], buf.reps, buf.fingerprints, buf.unit_start, buf.n_units, buf.ws)
    assert e.value.rc == S.SCALE_ERR_INVALID_ARG
    with pytest.raises(S.ScaleError) as e:
        S.scale_select(p, PER_CLUSTER, 0, w.n_tokens, buf.reps, buf.fingerprints, buf.unit_start,
                       buf.n_units, buf.sel_blocks, buf.sel_count, None, buf.ws[:1024])
    assert e.value.rc == S.SCALE_ERR_WORKSPACE
    with pytest.raises(S.ScaleError) as e:
        S.scale_sparse_prefill(p, PER_CLUSTER, 100, w.n_tokens, *dev, buf.unit_start, buf.n_units,
                               buf.sel_blocks, buf.sel_count, buf.out, buf.ws)
    assert e.value.rc == S.SCALE_ERR_INVALID_ARG
    narrow = S.params_for(w, head_dim=64)  # valid, but the kernels implement head_dim 128 only
    with pytest.raises(S.ScaleError) as e:
        S.scale_sparse_prefill(narrow, PER_SUB, 0, w.n_tokens, *dev, None, None, buf.sel_blocks,
                               buf.sel_count, buf.out, buf.ws)
    assert e.value.rc == S.SCALE_ERR_UNSUPPORTED
    torch.cuda.synchronize()
    assert S.scale_get_device_status(buf.ws) == S.SCALE_OK


# --------------------------------------------------------------------------- full-size stack and 1M


def _full_size_check(w, q, k, v, mode, n_random, seed=7):
    import time

    t0 = time.time()
    log = lambda *a: print(f"  [{time.time() - t0:6.1f}s]", *a, flush=True)  # noqa: E731
    dev = [torch.from_numpy(x).view(torch.bfloat16).cuda() for x in (q, k, v)]
    p, buf = gpu_path(w, mode, dev, want_scores=False)
    log("gpu path done")
    ref = oracle_path(w, q, k, v, mode)
    log("oracle selection done")
    n = unit_count(buf, mode, w)
    sel = buf.sel_blocks.cpu().numpy()[:n, : w.top_k]
    cnt = buf.sel_count.cpu().numpy()[:n]
    same, near = compare_selection(sel, cnt, ref)
    us = ref["unit_start"] if mode == PER_CLUSTER else np.arange(w.n_subchunks + 1, dtype=np.int32)
    rng = np.random.default_rng(seed)
    tok_us = np.minimum(us.astype(np.int64) * w.sub_chunk, w.n_tokens)
    rows = [int(tok_us[u]) for u in range(len(us) - 1)] + [int(tok_us[u + 1]) - 1 for u in range(len(us) - 1)]
    rows += rng.integers(0, w.n_tokens, size=n_random).tolist()
    rows = np.unique(np.array(rows, np.int64))
    log(f"oracle attention on {len(rows)} rows ({near} near-tie units, on the GPU's selection)")
    # near-tie units keep their rows: the oracle runs on the selection the GPU used
    ref_attn = oracle.attention_rows(q=q, k=k, v=v, sub_chunk=w.sub_chunk, block_size=w.block_size,
                                     top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                                     attn_scale=1.0 / np.sqrt(w.head_dim),
                                     per_subchunk=(mode == PER_SUB), unit_start=ref["unit_start"],
                                     sel=selection_for_reference(sel, ref, same),
                                     sel_count=ref["sel_count"], rows=rows)
    log("oracle attention done")
    got = to_f64_bf16(buf.out[torch.from_numpy(rows).cuda()])
    mx, mean = attn_errors(got, ref_attn)
    del buf, dev
    torch.cuda.empty_cache()
    return len(rows), mx, mean, near


@pytest.mark.parametrize("layer", [0, 15, 31])
def test_stack_64k_layers_full_size(layer):
    """The 32-layer 64K stack: independent inputs per layer (seed = layer); layers 0, 15, 31."""
    from synth import generate_layer, workload

    w = workload("llama8b-64k-32l")
    q, k, v = generate_layer(w, layer=layer)
    for mode in (PER_CLUSTER, PER_SUB):
        n, mx, mean, near = _full_size_check(w, q, k, v, mode, n_random=48, seed=layer)
        print(f"layer {layer} mode={mode}: {n} rows, max {mx:.3e} mean {mean:.3e}, {near} near-tie units")
        assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


def test_1m_context_full_size():
    """The 1M-token layer, both modes: selection of every unit, attention on the
    first and last row of every unit plus random rows."""
    from synth import generate_layer, workload

    w = workload("llama8b-1m")
    q, k, v = generate_layer(w)
    for mode in (PER_CLUSTER, PER_SUB):
        n, mx, mean, near = _full_size_check(w, q, k, v, mode, n_random=40)
        print(f"1M mode={mode}: {n} rows, max {mx:.3e} mean {mean:.3e}, {near} near-tie units")
        assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


# --------------------------------------------------------------------------- paged KV cache


def _paged(x, page_size, rng, extra=3):
    """x [N][H][128] on the device -> (pool [n_pages + extra][P][H][128], page table):
    pages in shuffled order, unused pages and the tail of the last page filled
    with large values that a wrong read would expose."""
    N, H, D = x.shape
    n_pages = -(-N // page_size)
    pool = torch.full((n_pages + extra, page_size, H, D), 1000.0, dtype=x.dtype, device=x.device)
    perm = torch.from_numpy(rng.permutation(n_pages + extra)[:n_pages].astype(np.int32)).to(x.device)
    for i in range(n_pages):
        rows = x[i * page_size:(i + 1) * page_size]
        pool[int(perm[i]), : rows.shape[0]] = rows
    return pool, perm


PAGED_CASES = [("gqa4-4k", {}, 64), ("gqa4-4k", dict(n_tokens=3000), 128),
               ("llama8b-32k", {}, 256), ("llama8b-32k", dict(block_size=1, top_k=1024), 128)]


@pytest.mark.parametrize("mode", [PER_CLUSTER, PER_SUB])
@pytest.mark.parametrize("name,over,page", PAGED_CASES)
def test_paged_kv_equals_contiguous(name, over, page, mode):
    """The *_paged entry points on a shuffled page pool against the oracle:
    representatives and fingerprints within the step (a) tolerance, the unit
    table exactly, every unit's selection exactly (near-tie rule), attention on
    every row at 4K and on sampled rows at 32K (the oracle on the selection
    the paged path used). They also give the contiguous path's results bit for
    bit (same keys and values, same arithmetic)."""
    w, q, k, v, dev = inputs(name, **over)
    p, contig = gpu_path(w, mode, dev)
    rng = np.random.default_rng(11)
    kp, table = _paged(dev[1], page, rng)
    vp, _ = _paged(dev[2], page, np.random.default_rng(11))
    kv = S.kv_pages(kp, vp, table, page)
    buf = S.allocate(p, mode)
    S.run_path_paged(p, mode, dev[0], kv, buf)
    torch.cuda.synchronize()
    assert S.scale_get_device_status(buf.ws) == S.SCALE_OK
    # against the oracle
    ref = oracle_path(w, q, k, v, mode)
    if w.block_size > 1:
        np.testing.assert_allclose(buf.reps.cpu().numpy().astype(np.float64), ref["reps"], rtol=0, atol=2e-5)
    np.testing.assert_allclose(buf.fingerprints.cpu().numpy().astype(np.float64), ref["fingerprints"],
                               rtol=0, atol=2e-5)
    n = unit_count(buf, mode, w)
    if mode == PER_CLUSTER:
        assert buf.unit_start[: n + 1].cpu().numpy().tolist() == ref["unit_start"].tolist()
    sel = buf.sel_blocks.cpu().numpy()[:n, : w.top_k]
    cnt = buf.sel_count.cpu().numpy()[:n]
    same, near = compare_selection(sel, cnt, ref)
    us = ref["unit_start"] if mode == PER_CLUSTER else np.arange(w.n_subchunks + 1, dtype=np.int32)
    rows = np.arange(w.n_tokens) if w.n_tokens <= 4096 else sample_rows(w, us, 16)
    ref_attn = oracle.attention_rows(q=q, k=k, v=v, sub_chunk=w.sub_chunk, block_size=w.block_size,
                                     top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                                     attn_scale=1.0 / np.sqrt(w.head_dim),
                                     per_subchunk=(mode == PER_SUB), unit_start=ref["unit_start"],
                                     sel=selection_for_reference(sel, ref, same),
                                     sel_count=ref["sel_count"], rows=rows)
    mx, mean = attn_errors(to_f64_bf16(buf.out[torch.from_numpy(rows).cuda()]), ref_attn)
    print(f"{name} {over} page {page} mode={mode}: {len(rows)} rows, max {mx:.3e} mean {mean:.3e}, "
          f"{near} near-tie units")
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS
    # and bit for bit against the contiguous path
    if w.block_size > 1:
        assert torch.equal(buf.reps, contig.reps)
    assert torch.equal(buf.fingerprints, contig.fingerprints)
    assert torch.equal(buf.sel_count[:n], contig.sel_count[:n])
    assert torch.equal(buf.sel_blocks[:n], contig.sel_blocks[:n])
    assert torch.equal(buf.out, contig.out)


@pytest.mark.parametrize("name,over,page", [("gqa4-4k", dict(n_tokens=3000), 128),
                                            ("llama8b-32k", dict(n_tokens=20000), 256)])
def test_paged_range_build_equals_contiguous(name, over, page):
    """scale_build_reps_range_paged over the outer chunks in order, on a
    shuffled page pool: representatives and fingerprints against the oracle
    (Eq. 6, block means) within the step (a) tolerance and the appended unit
    table against the oracle's Algorithm 1 exactly; and bit for bit against
    the contiguous whole-sequence step (a)."""
    w, q, k, v, dev = inputs(name, **over)
    p, ref = gpu_path(w, PER_CLUSTER, dev, want_scores=False)
    kp, table = _paged(dev[1], page, np.random.default_rng(5))
    vp, _ = _paged(dev[2], page, np.random.default_rng(5))
    kv = S.kv_pages(kp, vp, table, page)
    buf = S.allocate(p, PER_CLUSTER)
    for t0 in range(0, w.n_tokens, w.outer_chunk):
        t1 = min(w.n_tokens, t0 + w.outer_chunk)
        S.scale_build_reps_range_paged(p, t0, t1, dev[0], kv, buf.reps, buf.fingerprints, buf.unit_start,
                                       buf.n_units, buf.ws)
    torch.cuda.synchronize()
    assert S.scale_get_device_status(buf.ws) == S.SCALE_OK
    want = oracle_path(w, q, k, v, PER_CLUSTER)
    np.testing.assert_allclose(buf.reps.cpu().numpy().astype(np.float64), want["reps"], rtol=0, atol=2e-5)
    np.testing.assert_allclose(buf.fingerprints.cpu().numpy().astype(np.float64), want["fingerprints"],
                               rtol=0, atol=2e-5)
    n = int(buf.n_units.item())
    assert buf.unit_start[: n + 1].cpu().numpy().tolist() == want["unit_start"].tolist()
    assert torch.equal(buf.reps.view(torch.int32), ref.reps.view(torch.int32))
    assert torch.equal(buf.fingerprints.view(torch.int32), ref.fingerprints.view(torch.int32))
    assert torch.equal(buf.unit_start, ref.unit_start)
    assert int(buf.n_units.item()) == int(ref.n_units.item())


def test_paged_kv_entry_outside_pool_reads_zeros():
    """A page-table entry outside the pool is not dereferenced; its tokens act
    as zero keys and values: checked against the oracle run on K and V with
    those rows zeroed (every row), and against the contiguous path with those
    rows zeroed (bit for bit)."""
    w, q, k, v, dev = inputs("gqa4-4k")
    page = 64
    kz, vz = dev[1].clone(), dev[2].clone()
    kz[3 * page:4 * page] = 0
    vz[3 * page:4 * page] = 0
    p, ref = gpu_path(w, PER_CLUSTER, [dev[0], kz, vz])
    kp, table = _paged(dev[1], page, np.random.default_rng(5))
    vp, _ = _paged(dev[2], page, np.random.default_rng(5))
    table[3] = kp.shape[0] + 7
    buf = S.allocate(p, PER_CLUSTER)
    S.run_path_paged(p, PER_CLUSTER, dev[0], S.kv_pages(kp, vp, table, page), buf)
    torch.cuda.synchronize()
    assert S.scale_get_device_status(buf.ws) == S.SCALE_OK
    kh, vh = k.copy(), v.copy()
    kh[3 * page:4 * page] = 0
    vh[3 * page:4 * page] = 0
    rows = np.arange(w.n_tokens)
    want = oracle_path(w, q, kh, vh, PER_CLUSTER)
    np.testing.assert_allclose(buf.reps.cpu().numpy().astype(np.float64), want["reps"], rtol=0, atol=2e-5)
    n = int(buf.n_units.item())
    sel = buf.sel_blocks.cpu().numpy()[:n, : w.top_k]
    same, _ = compare_selection(sel, buf.sel_count.cpu().numpy()[:n], want)
    ref_attn = oracle.attention_rows(q=q, k=kh, v=vh, sub_chunk=w.sub_chunk, block_size=w.block_size,
                                     top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local,
                                     attn_scale=1.0 / np.sqrt(w.head_dim), per_subchunk=False,
                                     unit_start=want["unit_start"], sel=selection_for_reference(sel, want, same),
                                     sel_count=want["sel_count"], rows=rows)
    mx, mean = attn_errors(to_f64_bf16(buf.out), ref_attn)
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS
    assert torch.equal(buf.reps, ref.reps)
    assert torch.equal(buf.out, ref.out)


# --------------------------------------------------------------------------- decode with a selection cache


def _decode_queries(q, steps, seed=3):
    """Decode queries as consecutive generated tokens behave: a random walk from
    the query row at the first step (bf16), each step moving by about 7 % of
    its norm, so consecutive queries are close and drift apart with distance."""
    from synth import bf16_bits_to_f32, f64_to_bf16_bits

    rng = np.random.default_rng(seed)
    x = bf16_bits_to_f32(q[steps[0]]).astype(np.float64)
    scale = 0.07 * np.linalg.norm(x) / np.sqrt(x.size)
    out = []
    for _ in steps:
        out.append(f64_to_bf16_bits(x))
        x = x + scale * rng.standard_normal(x.shape)
    return np.stack(out)


def _decode_theta(qd, s_max):
    """A reuse threshold under which the cosine, not only the cap, decides some
    steps, with a mix of decisions and every decision far (> 1e-4) from it."""
    cap_only, _, _ = oracle.decode_reuse(qd, -1.0, s_max)
    best = None
    for theta in np.linspace(0.90, 0.999, 100):
        r, _, margin = oracle.decode_reuse(qd, float(theta), s_max)
        if (not np.array_equal(r, cap_only) and 2 < (~r).sum() < len(r) - 4 and margin > 1e-4
                and (best is None or margin > best[1])):
            best = (float(theta), margin)
    assert best is not None
    return best[0]


@pytest.mark.parametrize("heads", [(6, 2), (8, 1), (4, 4), (16, 8), (34, 17)])
def test_decode_group_sizes(heads):
    """Retrieving decode steps for query-head groups of 3 (the CUDA-core kernel
    for any group size), 8, 1 and 2 query heads per KV head (tensor cores), and
    2 with 17 KV heads (the register-blocked CUDA-core kernel): selection and
    output row against the oracle."""
    hq, hkv = heads
    w, q, k, v, dev = inputs("gqa4-4k", n_tokens=2048, num_q_heads=hq, num_kv_heads=hkv, block_size=1,
                             top_k=128, n_local=256, n_sink=32)
    steps = np.arange(1900, 1906)
    qd = _decode_queries(q, steps)
    p = S.params_for(w, theta=2.0, max_cluster_subchunks=1)  # cos >= 2 never holds: every step retrieves
    cache = torch.empty(S.scale_decode_cache_size(p), dtype=torch.uint8, device="cuda")
    S.scale_decode_cache_init(cache)
    ws = torch.empty(S.scale_decode_workspace_size(p), dtype=torch.uint8, device="cuda")
    S.scale_workspace_init(ws)
    qd_dev = torch.from_numpy(qd).view(torch.bfloat16).cuda()
    sel_full = np.full((w.n_tokens, w.top_k), -1, np.int32)
    cnt_full = np.zeros(w.n_tokens, np.int32)
    outs = []
    for i, t in enumerate(steps):
        out = torch.empty((hq, w.head_dim), dtype=torch.bfloat16, device="cuda")
        S.scale_decode_step(p, int(t), qd_dev[i], dev[1], dev[2], cache, out, ws)
        torch.cuda.synchronize()
        assert S.decode_cache_state(cache)["retrieved"]
        sel, cnt = S.decode_cache_selection(cache, p)
        ref, gap = oracle.decode_select(qd[i], k, int(t), n_sink=w.n_sink, n_local=w.n_local, top_k=w.top_k)
        assert cnt == len(ref)
        if sel[:cnt].tolist() != ref.tolist():
            assert gap < NEAR_TIE_GAP, f"step {t}: selection differs with gap {gap:.3e}"
        sel_full[t, :cnt] = sel[:cnt]
        cnt_full[t] = cnt
        outs.append(to_f64_bf16(out))
    assert S.scale_get_device_status(ws) == S.SCALE_OK
    q_rows = q.copy()
    q_rows[steps] = qd
    ref_attn = oracle.attention_rows(q=q_rows, k=k, v=v, sub_chunk=1, block_size=1, top_k=w.top_k,
                                     n_sink=w.n_sink, n_local=w.n_local,
                                     attn_scale=1.0 / np.sqrt(w.head_dim), per_subchunk=True,
                                     unit_start=None, sel=sel_full, sel_count=cnt_full, rows=steps)
    mx, mean = attn_errors(np.stack(outs), ref_attn)
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS


@pytest.mark.parametrize("theta", [-1.0, None])
def test_decode_steps_with_selection_cache(theta):
    """scale_decode_step over 40 consecutive positions: reuse decisions, the
    selection of every retrieving step and every output row against the oracle."""
    w, q, k, v, dev = inputs("llama8b-32k", n_tokens=4096, block_size=1, top_k=256, n_local=512)
    steps = np.arange(3000, 3040)
    s_max = 8
    qd = _decode_queries(q, steps)
    if theta is None:
        theta = _decode_theta(qd, s_max)
    p = S.params_for(w, theta=theta, max_cluster_subchunks=s_max)
    cache = torch.empty(S.scale_decode_cache_size(p), dtype=torch.uint8, device="cuda")
    S.scale_decode_cache_init(cache)
    ws = torch.empty(S.scale_decode_workspace_size(p), dtype=torch.uint8, device="cuda")
    S.scale_workspace_init(ws)
    qd_dev = torch.from_numpy(qd).view(torch.bfloat16).cuda()
    want_r, anchor_of, margin = oracle.decode_reuse(qd, theta, s_max)
    assert margin > 1e-5
    sel_full = np.full((w.n_tokens, w.top_k), -1, np.int32)
    cnt_full = np.zeros(w.n_tokens, np.int32)
    outs, near = [], 0
    for i, t in enumerate(steps):
        out = torch.empty((w.num_q_heads, w.head_dim), dtype=torch.bfloat16, device="cuda")
        S.scale_decode_step(p, int(t), qd_dev[i], dev[1], dev[2], cache, out, ws)
        torch.cuda.synchronize()
        st = S.decode_cache_state(cache)
        assert bool(st["retrieved"]) == bool(want_r[i]), f"step {t}"
        assert st["anchor"] == steps[anchor_of[i]]
        sel, cnt = S.decode_cache_selection(cache, p)
        if want_r[i]:
            ref, gap = oracle.decode_select(qd[i], k, int(t), n_sink=w.n_sink, n_local=w.n_local,
                                            top_k=w.top_k)
            assert cnt == len(ref)
            if sel[:cnt].tolist() != ref.tolist():
                assert gap < NEAR_TIE_GAP, f"step {t}: selection differs with gap {gap:.3e}"
                near += 1
        sel_full[t, :cnt] = sel[:cnt]
        cnt_full[t] = cnt
        outs.append(to_f64_bf16(out))
    q_rows = q.copy()
    q_rows[steps] = qd
    ref_attn = oracle.attention_rows(q=q_rows, k=k, v=v, sub_chunk=1, block_size=1, top_k=w.top_k,
                                     n_sink=w.n_sink, n_local=w.n_local,
                                     attn_scale=1.0 / np.sqrt(w.head_dim), per_subchunk=True,
                                     unit_start=None, sel=sel_full, sel_count=cnt_full, rows=steps)
    assert S.scale_get_device_status(ws) == S.SCALE_OK
    mx, mean = attn_errors(np.stack(outs), ref_attn)
    print(f"theta={theta:.4f}: {int(want_r.sum())} retrievals in {len(steps)} steps, {near} near-ties, "
          f"attention max {mx:.3e} mean {mean:.3e}")
    assert mx <= ATTN_MAX_ABS and mean <= ATTN_MEAN_ABS
