"""CPU checks of the planted-topic inputs and of the overlap ratio (Sec. IV-C).

The overlap ratio's definition is pinned by hand cases on the oracle's
function; the package's host helpers (which the benchmark uses on GPU
selections) are checked against the oracle's independent code.
"""

import numpy as np
import pytest
import torch

import oracle
from paper_2609_31568_gb300 import fidelity as F
from synth import generate_layer, topic_segments, workload

SMALL = dict(n_tokens=12288 + 100, topic_len=2048)


def test_topic_segments_are_ordered_and_change_topic():
    w = workload("llama8b-128k-topics")
    starts, topics = topic_segments(w, 0, w.seed)
    assert starts[0] == 0 and np.all(np.diff(starts) > 0) and starts[-1] < w.n_tokens
    assert np.all((topics >= 0) & (topics < w.topics))
    assert np.all(topics[1:] != topics[:-1])
    assert 3 <= len(starts) <= 30  # mean segment 16384 tokens over 131072


def test_topic_generation_is_chunk_invariant():
    w = workload("llama8b-128k-topics", **SMALL)
    q, k, v = generate_layer(w, workers=1)
    q2, k2, v2 = generate_layer(w, t0=5000, t1=9000, workers=1)
    assert np.array_equal(q[5000:9000], q2)
    assert np.array_equal(k[5000:9000], k2)
    assert np.array_equal(v[5000:9000], v2)


def test_topic_boundaries_lower_fingerprint_similarity():
    """At every planted boundary one of the two consecutive pairs around the
    sub-chunk that holds it is less similar than every pair inside a topic
    (the property the clustering threshold detects)."""
    w = workload("llama8b-128k-topics", n_tokens=65536, topic_len=8192)
    q, _, _ = generate_layer(w)
    fp, norms = oracle.fingerprints(q, w.sub_chunk)
    vt = fp / norms[:, None]
    c = np.sum(vt[1:] * vt[:-1], axis=1)  # c[i] = cos(v_i, v_{i+1})
    starts, _ = topic_segments(w, 0, w.seed)
    held = sorted({int(b) // w.sub_chunk for b in starts[1:]})  # sub-chunk i holds a boundary
    near = sorted({j for i in held for j in (i - 1, i) if 0 <= j < len(c)})
    inside = np.setdiff1d(np.arange(len(c)), near)
    assert len(held) >= 3
    assert np.median(c[inside]) > 0.98
    for i in held:
        assert min(c[j] for j in (i - 1, i) if 0 <= j < len(c)) < c[inside].min()


def test_overlap_ratio_hand_cases():
    assert oracle.overlap_ratio([1, 2, 3, 4], [[1, 2], [3, 9]]) == 0.75
    assert oracle.overlap_ratio([5, 6], [[5, 6]]) == 1.0
    assert oracle.overlap_ratio([5, 6], [[7], [8]]) == 0.0
    assert oracle.overlap_ratio([5, 6, 7], [[5], [], [7]]) == pytest.approx(2 / 3)


def test_fidelity_helper_matches_oracle_on_random_selections():
    rng = np.random.default_rng(3)
    n_units, k = 12, 6
    sizes = rng.integers(1, 5, size=n_units)
    us = np.concatenate([[0], np.cumsum(sizes)])
    sel = np.sort(rng.choice(50, size=(n_units, k)), axis=1)
    cnt = rng.integers(0, k + 1, size=n_units)
    members = {(u, j): np.unique(rng.choice(50, size=rng.integers(0, k + 1)))
               for u in range(n_units) for j in range(1, int(sizes[u]))}
    rho, units = F.overlap_ratios(us, sel, cnt, lambda u, j: members[(u, j)])
    want = [(u, oracle.overlap_ratio(sel[u, : cnt[u]], [members[(u, j)] for j in range(1, sizes[u])]))
            for u in range(n_units) if sizes[u] >= 2 and cnt[u] > 0]
    assert units.tolist() == [u for u, _ in want]
    np.testing.assert_array_equal(rho, [r for _, r in want])


def test_member_query_fingerprints_substitutes_anchor_rows():
    rng = np.random.default_rng(4)
    fp = torch.from_numpy(rng.standard_normal((10, 8)).astype(np.float32))
    us = torch.tensor([0, 3, 4, 8, 10, 10, 10], dtype=torch.int32)  # padded past n_units
    got = F.member_query_fingerprints(fp, us, 4, 2)
    want = fp.clone()
    want[0] = fp[2]  # unit [0, 3) has a member 2
    want[4] = fp[6]  # unit [4, 8)
    assert torch.equal(got, want)
