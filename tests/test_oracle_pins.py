"""Pins of the CPU oracle against what the paper and the mathematics fix.

Nothing here retypes the oracle's formulas: each test checks a closed form, a
hand-worked case, an invariant, or a special case that reduces to a library
routine (torch's dense causal SDPA, numpy's lexsort).
"""

import math
import os

import numpy as np
import pytest
import torch

import oracle
from synth import bf16_bits_to_f32, f64_to_bf16_bits, generate_layer, workload

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def bf16(x):
    return f64_to_bf16_bits(np.asarray(x, np.float64))


# --------------------------------------------------------------------------- Eq. 6


def test_fingerprint_is_mean_with_ragged_last_subchunk():
    # q[t, h, d] = t + h  (small integers, exact in bf16). Sub-chunk i covers
    # [iL, min(N, (i+1)L)); its mean is (t0 + t1 - 1) / 2 + h.
    N, Hq, dh, L = 37, 2, 3, 8
    t = np.arange(N)[:, None, None]
    h = np.arange(Hq)[None, :, None]
    q = bf16(np.broadcast_to(t + h, (N, Hq, dh)))
    v, norms = oracle.fingerprints(q, L)
    assert v.shape == (5, Hq * dh)
    for i in range(5):
        t0, t1 = i * L, min(N, (i + 1) * L)
        expect = np.repeat((t0 + t1 - 1) / 2.0 + np.arange(Hq), dh)
        np.testing.assert_allclose(v[i], expect, rtol=0, atol=1e-12)
        assert norms[i] == pytest.approx(math.sqrt(float((expect ** 2).sum())), rel=1e-14)


def test_fingerprint_concatenates_heads_in_order():
    # Head h filled with the constant h+1: v must list head 0's d_h values first.
    N, Hq, dh, L = 8, 3, 4, 8
    q = bf16(np.broadcast_to(np.arange(1, Hq + 1)[None, :, None], (N, Hq, dh)))
    v, _ = oracle.fingerprints(q, L)
    np.testing.assert_array_equal(v[0], np.repeat(np.arange(1, Hq + 1), dh).astype(float))


# --------------------------------------------------------------------------- block reps


def test_block_reps_mean_and_ragged_last_block():
    N, Hkv, dh, B = 21, 2, 2, 4
    t = np.arange(N)[:, None, None]
    j = 100 * np.arange(Hkv)[None, :, None]
    k = bf16(np.broadcast_to(t + j, (N, Hkv, dh)))
    reps = oracle.block_reps(k, B)
    assert reps.shape == (Hkv, 6, dh)
    for jj in range(Hkv):
        for b in range(6):
            t0, t1 = b * B, min(N, (b + 1) * B)
            assert np.all(reps[jj, b] == (t0 + t1 - 1) / 2.0 + 100 * jj)


def test_block_size_one_reps_are_the_keys():
    # With B = 1 the representative of block b is key b itself, so block selection
    # is the paper's token-level selection exactly.
    w = workload("gqa4-4k", n_tokens=256)
    _, k, _ = generate_layer(w)
    reps = oracle.block_reps(k, 1)
    np.testing.assert_array_equal(reps, bf16_bits_to_f32(k).transpose(1, 0, 2).astype(np.float64))


# --------------------------------------------------------------------------- Algorithm 1


def _angles(deg):
    a = np.deg2rad(np.asarray(deg, np.float64))
    v = np.stack([np.cos(a), np.sin(a)], axis=1)
    return v, np.linalg.norm(v, axis=1)


def test_anchor_clustering_resists_drift():
    # Fingerprints 10 degrees apart, threshold cos(25 deg): every consecutive pair
    # passes, but the anchor comparison closes the cluster at 30 degrees
    # (the drift case that motivates Algorithm 1).
    v, n = _angles([0, 10, 20, 30, 40, 50, 60])
    us, margin = oracle.anchor_clustering(v, n, 8, 7, math.cos(math.radians(25)))
    assert us.tolist() == [0, 3, 6, 7]
    assert margin > 0.01


def test_anchor_clustering_threshold_is_inclusive():
    v = np.array([[1.0, 0.0], [3.0, 4.0]])
    n = np.array([1.0, 5.0])
    us, margin = oracle.anchor_clustering(v, n, 8, 2, 3.0 / 5.0)
    assert us.tolist() == [0, 2]  # cos == theta admits (Eq. 8 uses >=)
    assert margin == 0.0
    us, _ = oracle.anchor_clustering(v, n, 8, 2, np.nextafter(3.0 / 5.0, 1.0))
    assert us.tolist() == [0, 1, 2]


def test_anchor_clustering_cap_and_outer_chunks():
    M = 10
    v = np.ones((M, 3))
    n = np.linalg.norm(v, axis=1)
    us, _ = oracle.anchor_clustering(v, n, 4, 10, 0.5)
    assert us.tolist() == [0, 4, 8, 10]  # |C_a| L < L_max caps clusters at S_max = 4
    us, _ = oracle.anchor_clustering(v, n, 4, 5, 0.5)
    assert us.tolist() == [0, 4, 5, 9, 10]  # clusters never cross an outer chunk
    us, _ = oracle.anchor_clustering(v, n, 1, 10, 0.5)
    assert us.tolist() == list(range(11))  # S_max = 1: every sub-chunk alone


@pytest.mark.parametrize("M,S,per", [(16, 4, 4), (64, 8, 8), (37, 8, 16), (256, 16, 16), (9, 3, 4)])
def test_cluster_count_closed_form_when_all_admitted(M, S, per):
    rng = np.random.default_rng(M)
    v = rng.standard_normal((M, 5))
    us, _ = oracle.anchor_clustering(v, np.linalg.norm(v, axis=1), S, per, -1.0)
    expect = sum(-(-min(per, M - c) // S) for c in range(0, M, per))
    assert len(us) - 1 == expect
    assert us[0] == 0 and us[-1] == M and np.all(np.diff(us) >= 1) and np.all(np.diff(us) <= S)


def test_zero_norm_fingerprint_has_zero_cosine():
    v = np.array([[1.0, 0.0], [0.0, 0.0], [1.0, 0.0]])
    n = np.linalg.norm(v, axis=1)
    assert oracle.anchor_clustering(v, n, 8, 3, 0.5)[0].tolist() == [0, 1, 2, 3]
    assert oracle.anchor_clustering(v, n, 8, 3, -0.5)[0].tolist() == [0, 3]


# --------------------------------------------------------------------------- Eq. 9 soft voting


def _select_hand(logits_per_head, *, g=None, k=1, sigma=1.0):
    """Selection for one unit whose candidate blocks are 0..nc-1 and whose
    per-head logits are given directly: reps are one-hot rows, the anchor
    fingerprint slice of head h is logits_per_head[h]."""
    z = np.asarray(logits_per_head, np.float64)
    Hq, nc = z.shape
    Hkv = 1 if g is None else Hq // g
    dh = nc
    L = nc  # two sub-chunks of nc tokens, B = 1: unit 1 starts at s = nc
    N = 2 * nc
    reps = np.zeros((Hkv, N, dh))
    for j in range(Hkv):
        reps[j, :nc, :] = np.eye(nc)
    v = np.zeros((2, Hq * dh))
    v[1] = z.reshape(-1)
    return oracle.select(num_q_heads=Hq, n_tokens=N, sub_chunk=L, block_size=1, top_k=k,
                         n_sink=0, n_local=0, select_scale=sigma, per_subchunk=True, reps=reps,
                         v=v, unit_start=None, want_scores=True)


def test_soft_voting_normalises_each_head():
    # Head 0 has one huge logit on block 0; heads 1-3 moderately prefer block 1.
    # A raw logit sum would pick block 0; the per-head softmax of Sec. V-A3 keeps
    # head 0 from dominating, and block 1 wins.
    z = [[100, 0, 0, 0], [0, 2, 0, 0], [0, 2, 0, 0], [0, 2, 0, 0]]
    r = _select_hand(z, k=1)
    assert r["sel"][1].tolist() == [1]
    assert r["cand_count"].tolist() == [0, 4]
    # each head contributes a probability distribution: scores sum to H_q
    assert np.nansum(r["scores"][1]) == pytest.approx(4.0, rel=1e-13)


def test_soft_voting_ties_go_to_lower_index():
    r = _select_hand(np.zeros((4, 6)), k=3)
    assert r["sel"][1].tolist() == [0, 1, 2]
    assert r["gap"][1] == 0.0
    np.testing.assert_allclose(r["scores"][1][:6], 4.0 / 6.0, rtol=1e-14)


def test_soft_voting_shift_invariance_per_head():
    rng = np.random.default_rng(3)
    z = rng.standard_normal((4, 9)) * 3
    base = _select_hand(z, k=4)
    shifted = _select_hand(z + rng.standard_normal((4, 1)) * 50, k=4)
    assert base["sel"][1].tolist() == shifted["sel"][1].tolist()
    np.testing.assert_allclose(base["scores"][1][:9], shifted["scores"][1][:9], rtol=1e-12)


def test_select_scale_extremes():
    rng = np.random.default_rng(4)
    z = rng.standard_normal((4, 7))
    flat = _select_hand(z, k=7, sigma=0.0)
    np.testing.assert_allclose(flat["scores"][1][:7], 4.0 / 7.0, rtol=1e-14)
    hard = _select_hand(z, k=7, sigma=1e4)
    votes = np.bincount(np.argmax(z, axis=1), minlength=7).astype(float)
    np.testing.assert_allclose(hard["scores"][1][:7], votes, atol=1e-12)


def test_gqa_mapping_is_grouped_not_interleaved():
    # H_q = 4, H_kv = 2. KV head 0 prefers block 3, KV head 1 prefers block 1.
    # Only query heads 0 and 1 carry a signal. With the grouped mapping
    # (h -> h // 2) both read KV head 0 and block 3 wins; an interleaved mapping
    # (h -> h % 2) would tie blocks 1 and 3 and the tie rule would pick block 1.
    Hq, Hkv, nc = 4, 2, 4
    N, L = 2 * nc, nc
    dh = 2
    reps = np.zeros((Hkv, N, dh))
    reps[0, 3] = [10.0, 0.0]
    reps[1, 1] = [10.0, 0.0]
    v = np.zeros((2, Hq * dh))
    v[1, 0 * dh] = 1.0
    v[1, 1 * dh] = 1.0
    r = oracle.select(num_q_heads=Hq, n_tokens=N, sub_chunk=L, block_size=1, top_k=1, n_sink=0,
                      n_local=0, select_scale=1.0, per_subchunk=True, reps=reps, v=v,
                      unit_start=None)
    assert r["sel"][1].tolist() == [3]


def test_topk_matches_library_sort():
    w = workload("gqa4-4k")
    q, k, _ = generate_layer(w)
    fv, norms = oracle.fingerprints(q, w.sub_chunk)
    reps = oracle.block_reps(k, w.block_size)
    for per in (True, False):
        us = None if per else np.arange(0, w.n_subchunks + 1, w.max_cluster_subchunks, dtype=np.int32)
        r = oracle.select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
                          block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink,
                          n_local=w.n_local, select_scale=1.0, per_subchunk=per, reps=reps, v=fv,
                          unit_start=us, want_scores=True)
        for u in range(r["sel"].shape[0]):
            s = r["scores"][u]
            cand = np.flatnonzero(~np.isnan(s))
            assert r["cand_count"][u] == len(cand)
            order = cand[np.lexsort((cand, -s[cand]))]
            expect = np.sort(order[: w.top_k])
            n = r["sel_count"][u]
            assert n == min(w.top_k, len(cand))
            assert r["sel"][u][:n].tolist() == expect.tolist()
            assert np.all(r["sel"][u][n:] == -1)


def test_candidates_are_distant_blocks():
    # Hand counts of R4 (blocks with a token in [n_sink, W_u), W_u = s_u - n_local):
    #  B=64, n_sink=64, n_local=256, unit at s=512: W=256 -> blocks 1, 2, 3;
    #  B=256, n_sink=128, n_local=1024, unit at s=4096: W=3072 -> blocks 0..11;
    #  B=128, n_sink=128, n_local=1024, unit at s=1024: W=0 -> none.
    for B, ns, nl, s, expect in [(64, 64, 256, 512, [1, 2, 3]),
                                 (256, 128, 1024, 4096, list(range(12))),
                                 (128, 128, 1024, 1024, []),
                                 (100, 150, 30, 400, [1, 2, 3])]:
        N = s + 8
        L = s
        nb = -(-N // B)
        reps = np.zeros((1, nb, 1))
        v = np.zeros((2, 1))
        r = oracle.select(num_q_heads=1, n_tokens=N, sub_chunk=L, block_size=B, top_k=nb,
                          n_sink=ns, n_local=nl, select_scale=1.0, per_subchunk=True, reps=reps,
                          v=v, unit_start=None)
        assert r["sel"][1][: r["sel_count"][1]].tolist() == expect


def _golden_calls():
    rows = {}
    with open(os.path.join(GOLDEN, "retrieval_calls.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            name, su, sc, bu, bc = line.split()
            rows[name] = (int(su), int(sc), int(bu), int(bc))
    return rows


@pytest.mark.parametrize("name", sorted(_golden_calls()))
def test_retrieval_call_counts_match_closed_form(name):
    w = workload(name)
    su, sc, bu, bc = _golden_calls()[name]
    M = w.n_subchunks
    v = np.ones((M, w.num_q_heads))  # head_dim 1 keeps this cheap; counts need no data
    us, _ = oracle.anchor_clustering(v, np.linalg.norm(v, axis=1), w.max_cluster_subchunks,
                                     w.outer_chunk // w.sub_chunk, w.theta)
    reps = np.zeros((w.num_kv_heads, w.n_blocks, 1))
    for per, units, calls in ((False, su, sc), (True, bu, bc)):
        r = oracle.select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
                          block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink,
                          n_local=w.n_local, select_scale=1.0, per_subchunk=per, reps=reps, v=v,
                          unit_start=us)
        assert len(r["cand_count"]) == units
        assert int((r["cand_count"] > 0).sum()) == calls


def test_size_one_clusters_equal_per_subchunk_baseline():
    w = workload("gqa4-4k", max_cluster_subchunks=1)
    q, k, v = generate_layer(w)
    rows = np.arange(0, w.n_tokens, 13)
    a = oracle.run_path(w, q, k, v, per_subchunk=False, rows=rows)
    b = oracle.run_path(w, q, k, v, per_subchunk=True, rows=rows)
    assert a["unit_start"].tolist() == list(range(w.n_subchunks + 1))
    np.testing.assert_array_equal(a["sel"], b["sel"])
    np.testing.assert_array_equal(a["attn"], b["attn"])


# --------------------------------------------------------------------------- Eq. 10


def _sdpa(qf, kf, vf, scale, segments=None):
    """torch's dense causal SDPA in float64 (optionally per segment of rows)."""
    N, Hq, dh = qf.shape
    Hkv = kf.shape[1]
    out = np.empty((N, Hq, dh))
    segs = segments or [(0, N)]
    for s, e in segs:
        Q = torch.from_numpy(qf[s:e].transpose(1, 0, 2).copy())[None]
        K = torch.from_numpy(kf[s:e].transpose(1, 0, 2).copy())[None]
        V = torch.from_numpy(vf[s:e].transpose(1, 0, 2).copy())[None]
        o = torch.nn.functional.scaled_dot_product_attention(Q, K, V, is_causal=True, scale=scale,
                                                             enable_gqa=Hq != Hkv)
        out[s:e] = o[0].numpy().transpose(1, 0, 2)
    return out


def _f64(x):
    return bf16_bits_to_f32(x).astype(np.float64)


@pytest.mark.parametrize("per_subchunk", [False, True])
def test_full_selection_equals_dense_causal_sdpa(per_subchunk):
    # k >= number of blocks: every distant block is selected, so every key at or
    # before the row is attended: dense causal attention (Eq. 1).
    w = workload("gqa4-4k", n_tokens=448, sub_chunk=32, outer_chunk=128, block_size=16,
                 top_k=64, n_sink=16, n_local=32, num_q_heads=4, num_kv_heads=2)
    q, k, v = generate_layer(w)
    rows = np.arange(w.n_tokens)
    r = oracle.run_path(w, q, k, v, per_subchunk=per_subchunk, rows=rows)
    assert np.all(r["sel_count"] == r["cand_count"])
    ref = _sdpa(_f64(q), _f64(k), _f64(v), 1.0 / math.sqrt(w.head_dim))
    np.testing.assert_allclose(r["attn"], ref, rtol=0, atol=1e-12)


def test_no_sinks_no_selection_no_window_is_blockwise_causal():
    # n_sink = 0, k = 0, n_local = 0: every row sees only [s_u, p] of its own unit,
    # i.e. causal SDPA restricted to each cluster.
    w = workload("gqa4-4k", n_tokens=300, sub_chunk=32, outer_chunk=96, max_cluster_subchunks=3,
                 block_size=16, top_k=0, n_sink=0, n_local=0)
    q, k, v = generate_layer(w)
    r = oracle.run_path(w, q, k, v, per_subchunk=False, rows=np.arange(w.n_tokens))
    us = r["unit_start"] * w.sub_chunk
    segs = [(int(us[i]), int(min(w.n_tokens, us[i + 1]))) for i in range(len(us) - 1)]
    assert segs[-1] == (288, 300)
    ref = _sdpa(_f64(q), _f64(k), _f64(v), 1.0 / math.sqrt(w.head_dim), segs)
    np.testing.assert_allclose(r["attn"], ref, rtol=0, atol=1e-12)


def test_key_set_revealed_by_uniform_attention():
    # q = 0 makes the softmax uniform over the key set, and one-hot values v_t = e_t
    # make the output reveal that set: o[d] = 1/|K(p)| for d in K(p), else 0.
    # Hand configuration: N=64, L=8, clusters of 2 sub-chunks (16 tokens), B=4,
    # n_sink=4, n_local=6. Key sets written out from Sec. V-A3 by hand.
    N, L, B = 64, 8, 4
    q = np.zeros((N, 1, N), np.uint16)
    k = np.zeros((N, 1, N), np.uint16)
    v = bf16(np.eye(N)[:, None, :])
    us = np.array([0, 2, 4, 6, 8], np.int32)
    sel = np.array([[-1, -1], [-1, -1], [1, 5], [0, 10]], np.int32)
    cnt = np.array([0, 0, 2, 2], np.int32)
    rows = np.array([0, 5, 20, 32, 40, 48, 50, 63])
    out = oracle.attention_rows(q=q, k=k, v=v, sub_chunk=L, block_size=B, top_k=2, n_sink=4,
                                n_local=6, attn_scale=1.0, per_subchunk=False, unit_start=us,
                                sel=sel, sel_count=cnt, rows=rows)
    R = range
    expect = {
        0: [0],
        5: list(R(0, 6)),
        20: list(R(0, 4)) + list(R(10, 21)),             # unit 1: s=16, W=10
        32: list(R(0, 8)) + list(R(20, 24)) + list(R(26, 33)),  # unit 2: W=26, blocks 1, 5
        40: list(R(0, 8)) + list(R(20, 24)) + list(R(26, 41)),
        48: list(R(0, 4)) + list(R(40, 49)),             # unit 3: W=42, block 0 is inside the sinks,
        50: list(R(0, 4)) + list(R(40, 51)),             #   block 10 {40..43} overlaps the window
        63: list(R(0, 4)) + list(R(40, 64)),
    }
    for i, p in enumerate(rows):
        ks = expect[int(p)]
        want = np.zeros(N)
        want[ks] = 1.0 / len(ks)
        np.testing.assert_allclose(out[i, 0], want, rtol=0, atol=1e-15, err_msg=f"row {p}")


def test_member_selection_uses_member_j_against_the_cluster_candidates():
    """Sec. IV-C's per-member retrieval by construction: block b's
    representative is the unit vector e_b, and a sub-chunk's fingerprint
    points at one block with a large weight in every head, so with top_k = 1
    the selection is that block. Member j of the cluster [8, 12) must pick the
    block its own fingerprint names (not the anchor's, nor a neighbour's), from
    the cluster's candidates (blocks before W_u = 8 * 64 - 64 = 448, i.e. 0..27,
    not the member's own later range); clusters of one sub-chunk keep their
    anchor."""
    from types import SimpleNamespace

    L, B, nb, Hq = 64, 16, 64, 2
    w = SimpleNamespace(num_q_heads=Hq, n_tokens=16 * L, sub_chunk=L, block_size=B, top_k=1, n_sink=0,
                        n_local=L)
    reps = np.zeros((1, nb, 128))
    for b in range(nb):
        reps[0, b, b] = 1.0
    v = np.zeros((16, Hq * 128))
    target = {8: 5, 9: 20, 10: 17, 11: 30, 3: 2}  # sub-chunk -> block its fingerprint names
    for i, b in target.items():
        for h in range(Hq):
            v[i, h * 128 + b] = 50.0
    unit_start = np.array(list(range(9)) + [12, 13, 14, 15, 16], np.int32)  # cluster [8, 12) is unit 8
    anchor = oracle.member_selection(w, reps, v, unit_start, 0)
    assert anchor["sel"][8].tolist() == [5]
    assert oracle.member_selection(w, reps, v, unit_start, 1)["sel"][8].tolist() == [20]
    assert oracle.member_selection(w, reps, v, unit_start, 2)["sel"][8].tolist() == [17]
    # member 3 names block 30: inside its own per-sub-chunk range (blocks < 40) but
    # not the cluster's (blocks < 28), so it must not be selected
    m3 = oracle.member_selection(w, reps, v, unit_start, 3)
    assert m3["cand_count"][8] == 28 and 0 <= m3["sel"][8][0] < 28
    for j in (1, 2, 3):  # singleton units keep their anchor's selection
        r = oracle.member_selection(w, reps, v, unit_start, j)
        assert r["sel"][3].tolist() == anchor["sel"][3].tolist() == [2]
        assert r["sel"][0].tolist() == anchor["sel"][0].tolist()
