"""Two gloo ranks on the CPU: the head-sharded split of step (b).

With KV heads (and their query heads) split across ranks, every rank can form
the per-head softmax votes of its own heads; the soft-vote score of Sec. V-A3
is a sum over heads, so one all-reduce (sum) of the partial scores before the
top-k reproduces the single-device selection exactly (up to fp64 summation
order). The arithmetic on each rank is the oracle's, restricted to its heads.
"""

import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, result_path):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import oracle
    from synth import generate_layer, workload

    w = workload("llama8b-32k", n_tokens=8192, sub_chunk=512, outer_chunk=2048,
                 max_cluster_subchunks=4, top_k=8)
    q, k, v = generate_layer(w)
    kv_per = w.num_kv_heads // world
    kv = slice(rank * kv_per, (rank + 1) * kv_per)
    qh = slice(rank * kv_per * w.group, (rank + 1) * kv_per * w.group)
    fp, norms = oracle.fingerprints(q, w.sub_chunk)
    us, _ = oracle.anchor_clustering(fp, norms, w.max_cluster_subchunks,
                                     w.outer_chunk // w.sub_chunk, w.theta)
    reps = oracle.block_reps(k[:, kv], w.block_size)
    fp_local = fp.reshape(fp.shape[0], w.num_q_heads, w.head_dim)[:, qh].reshape(fp.shape[0], -1)
    part = oracle.select(num_q_heads=kv_per * w.group, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
                         block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink,
                         n_local=w.n_local, select_scale=1.0, per_subchunk=False, reps=reps,
                         v=fp_local, unit_start=us, want_scores=True)["scores"]
    t = torch.from_numpy(np.nan_to_num(part, nan=0.0))
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    total = t.numpy()
    if rank == 0:
        np.save(result_path, total)
    dist.barrier()
    dist.destroy_process_group()


def test_head_sharded_votes_allreduce_to_full_selection(tmp_path):
    import oracle
    from synth import generate_layer, workload

    world = 2
    out = str(tmp_path / "scores.npy")
    mp.start_processes(_rank_main, args=(world, _free_port(), out), nprocs=world, join=True,
                       start_method="spawn")
    total = np.load(out)

    w = workload("llama8b-32k", n_tokens=8192, sub_chunk=512, outer_chunk=2048,
                 max_cluster_subchunks=4, top_k=8)
    q, k, v = generate_layer(w)
    ref = oracle.run_path(w, q, k, v, per_subchunk=False)
    full = oracle.select(num_q_heads=w.num_q_heads, n_tokens=w.n_tokens, sub_chunk=w.sub_chunk,
                         block_size=w.block_size, top_k=w.top_k, n_sink=w.n_sink,
                         n_local=w.n_local, select_scale=1.0, per_subchunk=False, reps=ref["reps"],
                         v=ref["fingerprints"], unit_start=ref["unit_start"], want_scores=True)
    cand = ~np.isnan(full["scores"])
    np.testing.assert_allclose(total[cand], full["scores"][cand], rtol=1e-12, atol=1e-12)
    for u in range(total.shape[0]):
        c = np.flatnonzero(cand[u])
        order = c[np.lexsort((c, -total[u, c]))][: w.top_k]
        n = int(full["sel_count"][u])
        assert np.sort(order).tolist() == full["sel"][u, :n].tolist()
