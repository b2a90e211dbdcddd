"""scale_build_reps_noalloc: step (a) for callers that cannot allocate.

Such callers (a plugin interface that passes only input and output buffers, a
serving loop whose device memory is fully reserved) cannot give the library a
workspace; this entry point keeps its scratch in a fixed array inside the
library instead. The test calls it through the C ABI twice in a row, on two
different inputs (so the second call starts from the first call's leftover
scratch), and checks each result against scale_build_reps, the entry point
with a caller-provided workspace. Both run the same kernels with the same
launch on the same inputs, so the results must be equal bit for bit (which is
within any tolerance of the step (a) parity tests). It also checks that a
problem needing more scratch than the fixed array is refused before anything
is launched.
"""

import pytest
import torch

import paper_2609_31568_gb300 as pkg
from paper_2609_31568_gb300 import scale as S
from synth import generate_layer, workload

pytestmark = pytest.mark.gpu


def _bits(x):
    return x.view(torch.int32) if x.dtype == torch.float32 else x


def _outputs(p):
    M = -(-p.n_tokens // p.sub_chunk)
    nb = -(-p.n_tokens // p.block_size)
    return (torch.empty((p.num_kv_heads, nb, 128), dtype=torch.float32, device="cuda"),
            torch.empty((M, p.num_q_heads * 128), dtype=torch.float32, device="cuda"),
            torch.empty(M + 1, dtype=torch.int32, device="cuda"),
            torch.empty(1, dtype=torch.int32, device="cuda"))


def _case(name, seed, **over):
    w = workload(name, **over)
    q, k, _ = generate_layer(w, seed=seed)
    return w, torch.from_numpy(q).view(torch.bfloat16).cuda(), torch.from_numpy(k).view(torch.bfloat16).cuda()


def test_noalloc_build_reps_matches_workspace_entry_point_twice():
    pkg.build()
    S.load()
    cases = [_case("llama8b-32k", 3, n_tokens=16384 + 77, sub_chunk=1024, outer_chunk=4096,
                   max_cluster_subchunks=4),
             _case("gqa4-4k", 5, n_tokens=3000)]
    for w, q, k in cases:
        p = S.params_for(w)
        ref = _outputs(p)
        ws = torch.empty(S.scale_workspace_size(p, S.SCALE_MODE_PER_CLUSTER), dtype=torch.uint8, device="cuda")
        S.scale_workspace_init(ws)
        S.scale_build_reps(p, q, k, *ref, ws)
        got = _outputs(p)
        for x in got:
            x.fill_(-7)  # any stale value must be overwritten
        S.scale_build_reps_noalloc(p, q, k, *got)
        torch.cuda.synchronize()
        # The no-workspace entry point has no device status of its own (step
        # (a) records none), so only the outputs are compared: bit for bit.
        assert torch.equal(_bits(got[0]), _bits(ref[0]))
        assert torch.equal(_bits(got[1]), _bits(ref[1]))
        assert torch.equal(got[3], ref[3])
        n = int(ref[3].item())
        assert torch.equal(got[2][: n + 1], ref[2][: n + 1])


def test_noalloc_refuses_problems_beyond_its_scratch():
    pkg.build()
    S.load()
    # 128M tokens in 512-token sub-chunks: M = 262144 sub-chunks, whose norm
    # sums and banded cosine rows need about 34 MB of step (a) scratch
    p = S.params_for(workload("llama8b-1m"), n_tokens=1 << 27, sub_chunk=512)
    small = torch.zeros(1024, dtype=torch.float32, device="cuda")
    ints = torch.zeros(1024, dtype=torch.int32, device="cuda")
    with pytest.raises(S.ScaleError) as e:
        S.scale_build_reps_noalloc(p, small, small, small, small, ints, ints)
    assert e.value.rc == S.SCALE_ERR_WORKSPACE
    torch.cuda.synchronize()


def test_noalloc_without_representatives_at_block_size_1():
    """At block size 1 the representatives may be skipped (reps = NULL), as for
    scale_build_reps; fingerprints and clusters are still written."""
    pkg.build()
    S.load()
    w, q, k = _case("gqa4-4k", 9, block_size=1, top_k=64)
    p = S.params_for(w)
    _, fp, us, n = _outputs(S.params_for(w.replace(block_size=64)))
    S.scale_build_reps_noalloc(p, q, k, None, fp, us, n)
    ref = _outputs(S.params_for(w.replace(block_size=64)))
    ws = torch.empty(S.scale_workspace_size(p, S.SCALE_MODE_PER_CLUSTER), dtype=torch.uint8, device="cuda")
    S.scale_workspace_init(ws)
    S.scale_build_reps(p, q, k, None, ref[1], ref[2], ref[3], ws)
    torch.cuda.synchronize()
    assert torch.equal(_bits(fp), _bits(ref[1]))
    assert torch.equal(n, ref[3])
    assert torch.equal(us[: int(n.item()) + 1], ref[2][: int(n.item()) + 1])

