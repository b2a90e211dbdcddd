"""Selection fidelity of cluster-level retrieval: the overlap ratio of Sec. IV-C.

A cluster C = {X_a, ..., X_{a+|C|-1}} shares the selection I_C made with its
anchor's fingerprint v_a. The overlap ratio compares I_C with the selections
the other members would have made with their own fingerprints:

    rho(C) = |I_C n U| / |I_C|,   U = union over j = 1 .. |C|-1 of I_{a+j}.

The anchor's own per-sub-chunk selection is I_C itself (same query, same
candidate blocks), so U leaves it out; with it rho would be 1 by
construction. I_{a+j} is either member j's query scored against the
cluster's candidate blocks (the same KV cache as the anchor's retrieval;
``member_query_fingerprints`` prepares the input of ``scale_select`` for it)
or the member's own per-sub-chunk selection (``scale_select`` in per-sub-chunk
mode). Selections are computed on the GPU; this module only prepares inputs
and counts set members on the host.
"""

from __future__ import annotations

import numpy as np


def member_query_fingerprints(fingerprints, unit_start, n_units: int, j: int):
    """Copy of the device fingerprints [M, D] in which the anchor row of every
    unit with more than j sub-chunks holds the fingerprint of its member j;
    ``scale_select`` in per-cluster mode on it scores member j's query against
    that unit's own candidate blocks (units with at most j sub-chunks keep
    their anchor's row)."""
    us = unit_start[: n_units + 1].long()
    a = us[:-1]
    idx = a[(us[1:] - a) > j]
    out = fingerprints.clone()
    out[idx] = fingerprints[idx + j]
    return out


def overlap_ratios(unit_start, sel, cnt, member):
    """rho(C) for every unit with two or more sub-chunks and a non-empty selection.

    unit_start: host ints [n_units + 1]; sel, cnt: host selections of the
    units (ascending block indices, counts); member(u, j): host ints, the
    selection of member j (1 <= j < |C|) of unit u. Returns (rho, units)."""
    rho, units = [], []
    for u in range(len(unit_start) - 1):
        size = int(unit_start[u + 1]) - int(unit_start[u])
        n = int(cnt[u])
        if size < 2 or n == 0:
            continue
        anchor = np.asarray(sel[u, :n], np.int64)
        union = np.unique(np.concatenate([np.asarray(member(u, j), np.int64) for j in range(1, size)]))
        rho.append(np.count_nonzero(np.isin(anchor, union)) / n)
        units.append(u)
    return np.array(rho, np.float64), np.array(units, np.int64)


def summary(x) -> dict:
    """min / median / mean / max, as the paper's overlap table reports them."""
    x = np.asarray(x, np.float64)
    if x.size == 0:
        return {"n": 0}
    return {"n": int(x.size), "min": float(x.min()), "median": float(np.median(x)),
            "mean": float(x.mean()), "max": float(x.max())}
