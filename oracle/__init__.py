"""CPU oracle of the counter-causal refresh (arXiv 2607.27600) -- TEST INFRASTRUCTURE.

Plain fp64 numpy restatement of the scoring, keep-set selection and
compaction the paper defines.  Only tests/, __graft_entry__.smoke() and the
CPU legs of bench.py may import it.  It shares no code with the CUDA path.

Parity status per function (what pins it, in tests/test_oracle_*.py):
  rms_norm                 torch rms_norm (library routine)
  rope                     complex-multiplication identity; relative-position property
  rope_inv_freq (scaled)   band structure of Llama-3.1 scaling: unchanged short
                           wavelengths, factor-slowed long ones, an affine blend
                           between that meets both edges
  project (q/k/v biases)   closed form with Wq = 0 (queries = rotated bias);
                           RoPE-shift invariance of a biased, scaled model
  counter_causal_attention torch SDPA with an explicit mask (library routine);
                           closed forms (row n-2 -> V[n-1], K = 0 -> mean of later V,
                           last row -> 0); brute force on tiny inputs
  causal_attention         torch SDPA is_causal (library routine)
  swiglu_mlp               hand-computed scalar case
  score_head               closed form; scipy log_softmax (library routine)
  score_layer/score_full   closed-form special cases, mask-leakage, prefix-drop,
                           batch/ragged, GQA-permutation, RoPE-shift and L=1
                           (full == single-layer) invariants
  select_keep              brute-force sort on tiny inputs; forced keeps; identity
  compact                  sequential in-place loop; order preservation
  memory_causal_attention  torch SDPA with an explicit mask (memory all visible,
                           chunk causal); n0 = 0 is causal_attention
  recency_scores           the position itself (keep-set = most recent slots)
  key_attention_colsums    column sums = sum of the attention matrix's entries;
                           each query row sums to 1; torch SDPA weights (library
                           routine) with keys as queries
  importance/h2o scores    closed forms (one head, equal keys -> uniform); H2O
                           over two refreshes = one update with both layer sets
  decode_step              = the causal forward's next-token argmax at the last
                           position, step by step over a greedy continuation
  e4m3_decode/e4m3_encode  values the format's definition names (1, 2, -1, 448,
                           2^-6, 2^-9, NaN); encode(decode(c)) = c for every finite
                           code; ties to the even code; saturation; torch's
                           float8_e4m3fn cast (library routine) in range
  append_chunk             into an empty cache = causal_forward; chunk-by-chunk
                           appends = one append (no refresh between); the layer's
                           attention after a compaction by scalar brute force
The paper prints no worked example with score values, so no pin is a
printed number; every step of the score is pinned by the checks above.
"""
from .refresh import (rms_norm, rope, rope_angles, rope_inv_freq, project, softmax,  # noqa: F401
                      counter_causal_attention,
                      causal_attention, silu, swiglu_mlp, counter_causal_layer, score_head,
                      score_layer, score_full, select_keep, compact, causal_forward,
                      memory_causal_attention, append_chunk, recency_scores,
                      key_attention_colsums, importance_scores, h2o_update, h2o_scores,
                      decode_step)
from .fp8 import e4m3_decode, e4m3_encode, kv_quantize  # noqa: F401
