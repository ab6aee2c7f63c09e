"""Row sharding of one refresh over several ranks (no GPU): the host-side
plan (cc_partition_rows) and, with world size 2 over gloo, the plan, the
per-rank scoring, the MAX exchange and the keep-set, with the oracle scoring
each rank's rows in place of the GPU pass.  The GPU side (cc_score_rows,
bit-identical rows) is tested in test_gpu_shard.py."""
import os
import socket

import numpy as np
import pytest
import torch
import torch.multiprocessing as mp

import synth
from synth.configs import LLAMA3_8B, ModelShape

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

SHAPE = ModelShape(n_layers=2, d_model=48, n_q_heads=4, n_kv_heads=2, head_dim=16, d_ff=80,
                   vocab=50, rope_theta=1e4, rms_eps=1e-5)


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


def _cost(shape, n, lo, hi):
    """Estimated cost of rows [lo, hi) of a sequence of n: per row the
    projections plus 4 dh Hq per later slot (brute force)."""
    g = 4.0 * shape.d_model * shape.n_q_heads * shape.head_dim + 6.0 * shape.d_model * shape.d_ff
    a = 4.0 * shape.head_dim * shape.n_q_heads
    i = np.arange(lo, hi, dtype=np.float64)
    return float(np.sum(g + a * (n - 1 - i)))


@pytest.mark.parametrize("world", [1, 2, 3, 4, 8])
@pytest.mark.parametrize("seq_lens", [[16384], [32768, 24576, 16384, 8192], [131072],
                                      [1, 0, 127, 129, 5000]])
def test_partition_covers_each_sequence_in_ascending_blocks(cc, world, seq_lens):
    lo, hi = cc.cc_partition_rows(LLAMA3_8B, True, seq_lens, world, 128)
    assert lo.shape == hi.shape == (world, len(seq_lens))
    for b, n in enumerate(seq_lens):
        assert lo[0, b] == 0 and hi[-1, b] == n
        for r in range(world):
            assert 0 <= lo[r, b] <= hi[r, b] <= n
            if r + 1 < world:
                assert hi[r, b] == lo[r + 1, b]                    # contiguous, disjoint
                assert hi[r, b] % 128 == 0 or hi[r, b] == n        # interior boundaries aligned


@pytest.mark.parametrize("world", [2, 3, 4, 8])
def test_partition_balances_the_estimated_cost(cc, world):
    """Every block's cost is within one alignment unit's cost of the equal
    share; early rows (more later slots) get the shorter blocks."""
    n = 131072
    lo, hi = cc.cc_partition_rows(LLAMA3_8B, False, [n], world, 128)
    total = _cost(LLAMA3_8B, n, 0, n)
    unit = _cost(LLAMA3_8B, n, 0, 128)       # the costliest 128 rows
    for r in range(world):
        c = _cost(LLAMA3_8B, n, lo[r, 0], hi[r, 0])
        assert abs(c - total / world) <= unit, (r, c / total)
    sizes = hi[:, 0] - lo[:, 0]
    assert np.all(np.diff(sizes) >= 0)


def test_partition_rejects_bad_arguments(cc):
    with pytest.raises(cc.CCError):
        cc.cc_partition_rows(LLAMA3_8B, True, [100], 0, 128)
    with pytest.raises(cc.CCError):
        cc.cc_partition_rows(LLAMA3_8B, True, [100], 2, 0)
    with pytest.raises(cc.CCError):
        cc.cc_partition_rows(LLAMA3_8B, True, [-1], 2, 128)


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _inputs():
    from tests._util import causal_cache, small_model
    w = small_model(SHAPE, seed=3)
    c = causal_cache(SHAPE, w, [300, 171, 1, 64], 320, seed=4)
    return w, c


def _rank(rank, world, port, full, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import torch.distributed as dist
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import oracle
        from paper_2607_27600_gb300 import cc, shard
        cc.load_library()
        w, c = _inputs()
        plan = shard.RowShard(SHAPE, full, c["seq_len"].tolist(), rank, world, align=16)
        rows = [list(range(plan.lo[rank, b], plan.hi[rank, b])) for b in range(len(c["seq_len"]))]
        fn = oracle.score_full if full else oracle.score_layer
        mine = fn(SHAPE, w, c, rows=rows).astype(np.float32)   # -inf outside the rank's rows
        scores = torch.from_numpy(mine.copy())
        shard.merge_scores(scores)
        idx, cnt = oracle.select_keep(scores.numpy(), c["seq_len"], [75, 40, 1, 16])
        out[rank] = (mine, scores.numpy().copy(), idx, cnt)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("full", [False, True])
def test_two_gloo_ranks_merge_to_the_single_rank_refresh(full):
    """World size 2: each rank scores its planned rows (oracle stand-in for
    the GPU pass), the MAX all-reduce assembles the scores, and both ranks
    hold exactly the merged buffer whose entries are their owners' values,
    the single-process scores (to fp64 summation order) and the same
    keep-set."""
    import oracle
    world = 2
    ctx = mp.get_context("spawn")
    with ctx.Manager() as m:
        out = m.dict()
        port = _free_port()
        ps = [ctx.Process(target=_rank, args=(r, world, port, full, out)) for r in range(world)]
        for p in ps:
            p.start()
        for p in ps:
            p.join(300)
            assert p.exitcode == 0
        res = dict(out)
    w, c = _inputs()
    fn = oracle.score_full if full else oracle.score_layer
    want = fn(SHAPE, w, c).astype(np.float32)
    (mine0, merged0, idx0, cnt0), (mine1, merged1, idx1, cnt1) = res[0], res[1]
    np.testing.assert_array_equal(merged0, merged1)
    # every entry is exactly its owner's value (the other rank holds -inf there)
    own0 = mine0 != -np.inf
    own1 = mine1 != -np.inf
    assert not np.any(own0 & own1)
    np.testing.assert_array_equal(merged0[own0], mine0[own0])
    np.testing.assert_array_equal(merged0[own1], mine1[own1])
    for b, n in enumerate(c["seq_len"]):
        assert np.all(own0[b, :n] | own1[b, :n])             # every row scored once
        np.testing.assert_allclose(merged0[b, :n], want[b, :n], rtol=1e-6, atol=0)
    wi, wc = oracle.select_keep(want, c["seq_len"], [75, 40, 1, 16])
    assert np.array_equal(cnt0, wc) and np.array_equal(idx0, wi)
    assert np.array_equal(idx0, idx1) and np.array_equal(cnt0, cnt1)
