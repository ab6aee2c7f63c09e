"""Model shapes and refresh workloads.

Each workload is one refresh of a KV cache: score every cached position,
select a keep-set of the given budget, compact the cache.  The shapes are
Llama-3-8B and Qwen2.5-7B layer shapes with random weights; the refresh
itself follows Sec. 3.1 (counter-causal surprise, fast single-layer
approximation) and Algorithm DoMemRefresh of arXiv 2607.27600.
"""
from dataclasses import dataclass, field
from typing import List, Optional, Tuple


@dataclass(frozen=True)
class ModelShape:
    n_layers: int
    d_model: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    d_ff: int
    vocab: int
    rope_theta: float
    rms_eps: float
    # Qwen2-style biases on the q/k/v projections (the scorer uses the q bias;
    # k/v biases live inside the cached K/V)
    qkv_bias: bool = False
    # Llama-3.1 RoPE frequency scaling: (factor, low_freq_factor,
    # high_freq_factor, original_max_position); None = plain RoPE
    rope_scaling: Optional[Tuple[float, float, float, int]] = None

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def q_dim(self) -> int:
        return self.n_q_heads * self.head_dim

    @property
    def kv_dim(self) -> int:
        return self.n_kv_heads * self.head_dim


@dataclass(frozen=True)
class Workload:
    name: str
    shape: ModelShape
    mode: str                 # "layer" (fast single-layer) or "full" (all layers)
    seq_lens: List[int]
    budgets: List[int]
    cap: int                  # slots per sequence in the cache buffers
    seed: int
    cache_from_causal_pass: bool   # tiny case: cache built by a causal forward
    cycles: int = 1                # refresh cycles (appends of `append` slots between them)
    append: int = 0
    n_sink: int = 0
    # the paper's own figure for this exact workload, as scored positions/s
    # (n / refresh latency), if it reports one; another GPU's number: context
    paper_positions_per_s: float = 0.0

    @property
    def batch(self) -> int:
        return len(self.seq_lens)

    @property
    def positions(self) -> int:
        return sum(self.seq_lens)


TINY = ModelShape(n_layers=1, d_model=512, n_q_heads=8, n_kv_heads=2, head_dim=64,
                  d_ff=1408, vocab=4096, rope_theta=1e4, rms_eps=1e-5)
LLAMA3_8B = ModelShape(n_layers=32, d_model=4096, n_q_heads=32, n_kv_heads=8, head_dim=128,
                       d_ff=14336, vocab=128256, rope_theta=5e5, rms_eps=1e-5)
QWEN25_7B = ModelShape(n_layers=28, d_model=3584, n_q_heads=28, n_kv_heads=4, head_dim=128,
                       d_ff=18944, vocab=152064, rope_theta=1e6, rms_eps=1e-6, qkv_bias=True)

WORKLOADS = {
    # tiny single-layer scoring, cache from a causal pass of the same random model
    "tiny-512": Workload("tiny-512", TINY, "layer", [512], [128], 512, seed=0,
                         cache_from_causal_pass=True),
    # Llama-3-8B last layer, one sequence of 8192 cached positions
    "llama8b-layer-8k": Workload("llama8b-layer-8k", LLAMA3_8B, "layer", [8192], [2048], 8192,
                                 seed=1, cache_from_causal_pass=False),
    # Llama-3-8B last layer, ragged batch of 4, budget 25 % of each sequence
    "llama8b-layer-32k-ragged": Workload(
        "llama8b-layer-32k-ragged", LLAMA3_8B, "layer", [32768, 24576, 16384, 8192],
        [8192, 6144, 4096, 2048], 32768, seed=2, cache_from_causal_pass=False),
    # Llama-3-8B full 32-layer counter-causal pass
    "llama8b-full-16k": Workload("llama8b-full-16k", LLAMA3_8B, "full", [16384], [4096], 16384,
                                 seed=3, cache_from_causal_pass=False),
    # Qwen2.5-7B-like last layer at 131072 positions, then 3 more cycles of +4096
    "qwen7b-layer-128k": Workload("qwen7b-layer-128k", QWEN25_7B, "layer", [131072], [8192],
                                  131072 + 4096, seed=4, cache_from_causal_pass=False,
                                  cycles=4, append=4096),
    # profiling case of the decode kernels: Qwen2.5-7B layer shapes, two layers
    # (about 1.6 GB of weights with the LM head), 8192 memory slots
    "qwen7b-2layer-8k": Workload("qwen7b-2layer-8k",
                                 ModelShape(**{**QWEN25_7B.__dict__, "n_layers": 2}), "layer",
                                 [8192], [8192], 8192 + 4096, seed=6,
                                 cache_from_causal_pass=False, append=4096),
}

# The paper's efficiency benchmark (Table 1): Qwen2.5-7B, a synthetic KV cache
# of n = 512 or 4096 slots, full L-layer pass and fast single-layer pass
# (RTX 4090, fp16: 54 / 496 ms full, 7.9 / 52.6 ms fast).  The table does not
# state the budget; these keep half the slots.
for _n, _full_ms, _fast_ms in ((512, 54.0, 7.9), (4096, 496.0, 52.6)):
    for _mode, _ms in (("full", _full_ms), ("layer", _fast_ms)):
        _name = f"qwen7b-table1-{'full' if _mode == 'full' else 'fast'}-{_n}"
        WORKLOADS[_name] = Workload(_name, QWEN25_7B, _mode, [_n], [_n // 2], _n, seed=5,
                                    cache_from_causal_pass=False,
                                    paper_positions_per_s=_n / (_ms * 1e-3))

# The bench's headline: the full-model pass over all 32 layers of the Llama-3-8B
# shape (the largest single-GPU workload with a full pass); the same line
# carries these workloads as records (the ragged 32k single-layer batch and
# the long-context refresh cycles).
HEADLINE = "llama8b-full-16k"
RECORDS = ["llama8b-layer-32k-ragged", "qwen7b-layer-128k"]
