"""CPU pins of the decode oracle: one-token selection equals the per-sub-chunk
rule of the C oracle with sub-chunks of one token (Def. 1 with C = 1), and the
selection cache follows the anchor rule on hand-made query sequences."""

import numpy as np

import oracle
from synth import f64_to_bf16_bits, generate_layer, workload


def test_decode_select_equals_one_token_units():
    w = workload("gqa4-4k", n_tokens=300, block_size=1, sub_chunk=1, max_cluster_subchunks=1,
                 outer_chunk=1, n_sink=8, n_local=32, top_k=16)
    q, k, v = generate_layer(w)
    reps = oracle.block_reps(k, 1)
    fp, _ = oracle.fingerprints(q, 1)
    ref = oracle.select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=1, block_size=1,
                        top_k=w.top_k, n_sink=w.n_sink, n_local=w.n_local, select_scale=1.0,
                        per_subchunk=True, reps=reps, v=fp, unit_start=None)
    for t in (0, 39, 40, 41, 120, 299):
        sel, gap = oracle.decode_select(q[t], k, t, n_sink=w.n_sink, n_local=w.n_local, top_k=w.top_k)
        c = int(ref["sel_count"][t])
        assert sel.tolist() == ref["sel"][t, :c].tolist()
        if np.isfinite(gap) or np.isfinite(ref["gap"][t]):
            assert abs(gap - ref["gap"][t]) <= 1e-9 * max(1.0, abs(gap))


def _q(rows):
    return f64_to_bf16_bits(np.array(rows, np.float64).reshape(len(rows), 1, -1))


def test_decode_reuse_hand_cases():
    same = _q([[1.0, 2.0, 3.0, 4.0]] * 7)
    r, a, _ = oracle.decode_reuse(same, theta=0.99, max_shared=3)
    assert r.tolist() == [True, False, False, True, False, False, True]  # capped at 3 steps per anchor
    assert a.tolist() == [0, 0, 0, 3, 3, 3, 6]
    ortho = _q([[1, 0, 0, 0], [0, 1, 0, 0], [0, 0, 1, 0]])
    r, _, _ = oracle.decode_reuse(ortho, theta=0.5, max_shared=8)
    assert r.tolist() == [True, True, True]
    r, _, _ = oracle.decode_reuse(ortho, theta=-1.0, max_shared=2)  # theta -1 admits everything
    assert r.tolist() == [True, False, True]
    drift = _q([[1, 0, 0, 0], [1, 0.1, 0, 0], [1, 0.6, 0, 0], [1, 0.7, 0, 0]])
    r, a, _ = oracle.decode_reuse(drift, theta=0.9, max_shared=8)
    # step 2 compares with the anchor (step 0), not with step 1: cos = 0.857 < 0.9
    assert r.tolist() == [True, False, True, False] and a.tolist() == [0, 0, 2, 2]
    zero = _q([[1, 0, 0, 0], [0, 0, 0, 0]])
    r, _, _ = oracle.decode_reuse(zero, theta=-0.5, max_shared=8)  # zero norm: cosine 0 >= -0.5
    assert r.tolist() == [True, False]
