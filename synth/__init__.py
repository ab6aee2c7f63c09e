"""Seeded synthetic inputs for the counter-causal refresh.

This module draws every input of a refresh (weights, tokens, positions,
cached K/V and last-layer hidden states) from named, seeded streams.  It
holds none of the method's arithmetic: it only draws numbers.  Both the
CPU oracle's tests and the CUDA path's tests and bench take their inputs
from here.

Every tensor is drawn from its own stream, keyed by (seed, name), so a
tensor does not depend on which other tensors were drawn before it.  A
stream lives on one torch device; draws on CPU and CUDA differ, so a test
draws each tensor once and copies it to wherever it is needed.

Value recipe (all matrices and the embedding as random-init Llama/Qwen
weights):
  * weight matrices and embedding: N(0, 0.02^2), rounded to bf16;
  * RMSNorm gains: 1;
  * q/k/v projection biases (shapes with qkv_bias, as Qwen2.5): N(0, 0.5^2),
    rounded to bf16 -- comparable to the projected values, whose standard
    deviation is 0.02 sqrt(d) (about 1.2 at d = 3584);
  * token ids: uniform on [0, vocab);
  * positions: 0, 1, ..., n-1 (original positions of a never-evicted cache);
  * synthetic cached K and V (post-RoPE): N(0, (0.02 sqrt(d))^2), the law of a
    projection of a unit-RMS normalised hidden state by N(0, 0.02^2) weights
    (RoPE rotates coordinate pairs, which leaves an isotropic Gaussian's law
    unchanged);
  * synthetic last-layer input hidden states H^(L-1): N(0, 1).
"""
import hashlib

import torch

from .configs import ModelShape, Workload, WORKLOADS, HEADLINE, RECORDS  # noqa: F401

WEIGHT_STD = 0.02
BIAS_STD = 0.5


def stream_seed(seed: int, name: str) -> int:
    """63-bit seed of the stream named `name` under the master seed."""
    h = hashlib.blake2b(f"{seed}:{name}".encode(), digest_size=8).digest()
    return int.from_bytes(h, "little") & ((1 << 63) - 1)


def _gen(seed: int, name: str, device) -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(stream_seed(seed, name))
    return g


def normal(shape, std: float, seed: int, name: str, device="cpu",
           dtype=torch.bfloat16) -> torch.Tensor:
    """N(0, std^2) draws, computed in fp32 and rounded to `dtype`."""
    g = _gen(seed, name, device)
    x = torch.randn(*shape, generator=g, device=device, dtype=torch.float32)
    x.mul_(std)
    return x.to(dtype)


def tokens(shape, vocab: int, seed: int, name: str = "tokens", device="cpu") -> torch.Tensor:
    g = _gen(seed, name, device)
    return torch.randint(0, vocab, tuple(shape), generator=g, device=device,
                         dtype=torch.int64).to(torch.int32)


def model_weights(shape: ModelShape, seed: int, device="cpu", with_kv_proj: bool = False,
                  layers=None, with_embed: bool = True) -> dict:
    """Random-init weights in nn.Linear layout: a [out, in] matrix per projection.

    `layers` restricts which layers are drawn (others are None); the fast
    single-layer refresh needs only the last one.  `with_kv_proj` also draws
    the K/V projections, which only a causal forward (cache builder) uses.
    """
    d, q, kv, f, v = shape.d_model, shape.q_dim, shape.kv_dim, shape.d_ff, shape.vocab
    ones = torch.ones(d, dtype=torch.bfloat16, device=device)
    want = range(shape.n_layers) if layers is None else layers
    out = {"embed": normal((v, d), WEIGHT_STD, seed, "embed", device) if with_embed else None,
           "final_norm": ones.clone(),
           "lm_head": normal((v, d), WEIGHT_STD, seed, "lm_head", device),
           "layers": [None] * shape.n_layers}
    for l in want:
        lw = {"attn_norm": ones.clone(), "mlp_norm": ones.clone(),
              "wq": normal((q, d), WEIGHT_STD, seed, f"l{l}.wq", device),
              "wo": normal((d, q), WEIGHT_STD, seed, f"l{l}.wo", device),
              "w_gate": normal((f, d), WEIGHT_STD, seed, f"l{l}.w_gate", device),
              "w_up": normal((f, d), WEIGHT_STD, seed, f"l{l}.w_up", device),
              "w_down": normal((d, f), WEIGHT_STD, seed, f"l{l}.w_down", device)}
        if with_kv_proj:
            lw["wk"] = normal((kv, d), WEIGHT_STD, seed, f"l{l}.wk", device)
            lw["wv"] = normal((kv, d), WEIGHT_STD, seed, f"l{l}.wv", device)
        if shape.qkv_bias:
            lw["bq"] = normal((q,), BIAS_STD, seed, f"l{l}.bq", device)
            if with_kv_proj:
                lw["bk"] = normal((kv,), BIAS_STD, seed, f"l{l}.bk", device)
                lw["bv"] = normal((kv,), BIAS_STD, seed, f"l{l}.bv", device)
        out["layers"][l] = lw
    return out


def kv_std(shape: ModelShape) -> float:
    return WEIGHT_STD * shape.d_model ** 0.5


def synthetic_cache(shape: ModelShape, seq_lens, cap: int, seed: int, device="cpu",
                    layers=None, with_h_last: bool = True) -> dict:
    """Synthetic KV cache of `len(seq_lens)` sequences in `cap`-slot buffers.

    Slots >= seq_len are filled too (with draws of the same law), so stale
    cache contents beyond a sequence's end are finite, as after a compaction.
    """
    b = len(seq_lens)
    hk, dh, d = shape.n_kv_heads, shape.head_dim, shape.d_model
    want = range(shape.n_layers) if layers is None else layers
    std = kv_std(shape)
    ks, vs = [None] * shape.n_layers, [None] * shape.n_layers
    for l in want:
        ks[l] = normal((b, cap, hk, dh), std, seed, f"cache.k{l}", device)
        vs[l] = normal((b, cap, hk, dh), std, seed, f"cache.v{l}", device)
    pos = torch.arange(cap, dtype=torch.int32, device=device).repeat(b, 1)
    out = {"k": ks, "v": vs,
           "tokens": tokens((b, cap), shape.vocab, seed, "cache.tokens", device),
           "pos": pos.contiguous(),
           "seq_len": torch.tensor(list(seq_lens), dtype=torch.int32, device=device),
           "h_last": None}
    if with_h_last:
        out["h_last"] = normal((b, cap, d), 1.0, seed, "cache.h_last", device)
    return out


def append_chunk(shape: ModelShape, cache: dict, count: int, seed: int, cycle: int):
    """Synthetic inference cycle between refreshes: append `count` new slots
    after each sequence's current end (K, V, H, token, next positions), in place.

    Positions continue from the largest position the sequence holds
    (Algorithm DoInference appends k_t, v_t, x_t in time order).  The host
    reads `seq_len` (a device sync) to find each sequence's end."""
    dev = cache["tokens"].device
    hk, dh, d = shape.n_kv_heads, shape.head_dim, shape.d_model
    std = kv_std(shape)
    lens = [int(x) for x in cache["seq_len"].tolist()]
    for b, start in enumerate(lens):
        sl = slice(start, start + count)
        tag = f"append{cycle}.b{b}"
        for l, (kl, vl) in enumerate(zip(cache["k"], cache["v"])):
            if kl is None:
                continue
            kl[b, sl] = normal((count, hk, dh), std, seed, f"{tag}.k{l}", dev)
            vl[b, sl] = normal((count, hk, dh), std, seed, f"{tag}.v{l}", dev)
        if cache.get("h_last") is not None:
            cache["h_last"][b, sl] = normal((count, d), 1.0, seed, f"{tag}.h", dev)
        cache["tokens"][b, sl] = tokens((count,), shape.vocab, seed, f"{tag}.tokens", dev)
        last = int(cache["pos"][b, :start].max()) if start > 0 else -1
        cache["pos"][b, sl] = torch.arange(last + 1, last + 1 + count, dtype=torch.int32,
                                           device=dev)
    cache["seq_len"].add_(count)
