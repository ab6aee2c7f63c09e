"""The seeded generators are deterministic and stream-independent (no GPU)."""
import torch

import synth
from tests._util import SMALL


def test_streams_are_deterministic_and_independent():
    a = synth.normal((4, 5), 0.02, 7, "x")
    b = synth.normal((4, 5), 0.02, 7, "x")
    c = synth.normal((4, 5), 0.02, 7, "y")
    assert torch.equal(a, b) and not torch.equal(a, c)
    assert a.dtype == torch.bfloat16


def test_cache_shapes_and_positions():
    c = synth.synthetic_cache(SMALL, [5, 3], 8, seed=1)
    assert c["k"][0].shape == (2, 8, SMALL.n_kv_heads, SMALL.head_dim)
    assert c["pos"][1].tolist() == list(range(8))
    assert c["seq_len"].tolist() == [5, 3]
    assert int(c["tokens"].max()) < SMALL.vocab


def test_append_continues_positions():
    c = synth.synthetic_cache(SMALL, [5, 3], 12, seed=1)
    c["pos"][0, :5] = torch.tensor([0, 2, 3, 7, 9], dtype=torch.int32)
    synth.append_chunk(SMALL, c, 4, seed=1, cycle=1)
    assert c["seq_len"].tolist() == [9, 7]
    assert c["pos"][0, 5:9].tolist() == [10, 11, 12, 13]
    assert c["pos"][1, 3:7].tolist() == [3, 4, 5, 6]
