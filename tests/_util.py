"""Helpers shared by the GPU tests: inputs on the device, oracle references,
selection comparison under the near-tie rule, attention error metrics."""

from __future__ import annotations

import functools

import numpy as np

from synth import generate_layer, workload

# Tolerances of the attention output (bf16 inputs, fp32 accumulation) against
# the fp64 oracle, and the relative k-th / (k+1)-th score gap under which two
# correct selections may differ.
ATTN_MAX_ABS = 2e-2
ATTN_MEAN_ABS = 2e-3
NEAR_TIE_GAP = 1e-3


@functools.lru_cache(maxsize=4)
def host_inputs(name: str, **overrides):
    w = workload(name, **dict(overrides)) if overrides else workload(name)
    q, k, v = generate_layer(w)
    return w, q, k, v


def inputs(name: str, **overrides):
    """(workload, host q/k/v as uint16, device q/k/v as bf16)."""
    import torch

    w, q, k, v = host_inputs(name, **overrides)
    dev = [torch.from_numpy(x).view(torch.bfloat16).cuda() for x in (q, k, v)]
    return w, q, k, v, dev


def to_f64_bf16(t) -> np.ndarray:
    import torch

    return t.to(torch.float32).cpu().numpy().astype(np.float64)


def compare_selection(gpu_sel: np.ndarray, gpu_cnt: np.ndarray, ref: dict):
    """Exact match of every unit's selected blocks, except units whose oracle
    k-th / (k+1)-th relative score gap is below NEAR_TIE_GAP.

    Returns (identical_units mask, number of near-tie units that differ)."""
    n = len(ref["sel_count"])
    assert gpu_cnt[:n].tolist() == ref["sel_count"].tolist(), "selection counts differ"
    same = np.zeros(n, bool)
    differ_near = 0
    for u in range(n):
        c = int(ref["sel_count"][u])
        a = gpu_sel[u, :c]
        b = ref["sel"][u, :c]
        same[u] = np.array_equal(a, b)
        if not same[u]:
            assert ref["gap"][u] < NEAR_TIE_GAP, (
                f"unit {u}: selection differs with oracle gap {ref['gap'][u]:.3e}")
            differ_near += 1
        assert np.all(gpu_sel[u, c:] == -1)
    return same, differ_near


def selection_for_reference(gpu_sel: np.ndarray, ref: dict, same: np.ndarray) -> np.ndarray:
    """The selection the attention reference runs on: the oracle's for every
    unit whose GPU selection matches it, the GPU's own for the units that
    differ at a near-tie (both are correct selections there, and the
    attention must be right for the one the path actually used)."""
    k = ref["sel"].shape[1]
    merged = np.array(ref["sel"], np.int32, copy=True)
    merged[~same] = gpu_sel[~same, :k]
    return merged


def attn_errors(gpu: np.ndarray, ref: np.ndarray):
    d = np.abs(gpu - ref)
    return float(d.max()), float(d.mean())


def rows_of_units(unit_start_tokens: np.ndarray, units) -> np.ndarray:
    return np.concatenate([np.arange(unit_start_tokens[u], unit_start_tokens[u + 1]) for u in units])


def last_query_blocks(w, unit_start: np.ndarray, units, rows: int = 128) -> np.ndarray:
    """Every row of the last `rows`-row query block of each listed unit: the
    rows with the longest cluster-spanning window, the attention kernel's
    heaviest work items."""
    tok = np.minimum(np.asarray(unit_start, np.int64) * w.sub_chunk, w.n_tokens)
    out = [np.arange(max(tok[u], tok[u + 1] - rows), tok[u + 1]) for u in units]
    return np.concatenate(out) if out else np.zeros(0, np.int64)


def sample_rows(w, unit_start: np.ndarray, n_random: int, seed: int = 1234) -> np.ndarray:
    """First and last row of every sub-chunk plus seeded random rows per unit."""
    rng = np.random.default_rng(seed)
    rows = set()
    for i in range(w.n_subchunks):
        rows.add(i * w.sub_chunk)
        rows.add(min(w.n_tokens, (i + 1) * w.sub_chunk) - 1)
    us = np.minimum(np.asarray(unit_start, np.int64) * w.sub_chunk, w.n_tokens)
    for u in range(len(us) - 1):
        rows.update(rng.integers(us[u], us[u + 1], size=n_random).tolist())
    return np.array(sorted(rows), np.int64)
