"""How far does bf16 arithmetic move the exact counter-causal score of a deep
random model?  A study over the oracle (test infrastructure, not collected by
pytest: the file name does not start with test_).

The oracle computes the full counter-causal pass (Sec. 3.1) in fp64.  A GPU
pass rounds some intermediates to use the bf16 tensor cores.  This script
re-runs the oracle's layer with rounding inserted at chosen points and
reports, per layer, the score's max relative error against the exact fp64
pass (the parity metric: |g - o| / max(|o|, rms(o))).  A "split" operand is
carried as the bf16 pair hi = bf16(x), lo = bf16(x - hi) (hi + lo is x to
about 2^-17 relative; a tensor-core product then runs once per half):

  queries      only the queries entering Q K^T rounded (every other step exact)
  activations  every GEMM input (normalised inputs, attention output, SwiGLU
               output) and the queries rounded
  bf16-pass    as `activations`, plus the attention probabilities P rounded
               before P V and the residual stream kept in fp32: every
               rounding point of a bf16 tensor-core pass
  split-act    GEMM inputs split; queries and P single bf16; fp32 residual
  split-q      GEMM inputs and queries split; P single bf16; fp32 residual
  split-all    GEMM inputs, queries and P split; fp32 residual
  split-qp     queries and P split, every GEMM input single bf16
  split-qp-attn  queries, P and the attention-side GEMM inputs (the Q
               projection's normalised input, the attention output) split
  split-qp-mlp   queries, P and the MLP's GEMM inputs (the gate/up
               projection's normalised input, the SwiGLU output) split
  fp16-pass    every rounding point of `bf16-pass` in fp16 instead, with the
               weights and cached K/V converted to fp16 as well

The drift measured here is a property of the arithmetic and of the random
model, not of any kernel; the full-pass tolerances of the parity tests are
derived from it.  It imports only the oracle and the seeded input
generators, never the CUDA path.

    python -m tests.study_fullpass_precision --layers 32 --n 16384 --rows 96
"""
import argparse
import sys

import numpy as np

from oracle import refresh as R


def bf16(x):
    """Round to the nearest bf16 value (ties to even), kept in fp64."""
    a = np.asarray(x, np.float64).astype(np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


def split(x):
    """x carried as the bf16 pair (hi, lo): the value hi + lo, computed from
    the fp32 rounding of x as a GPU epilogue would."""
    x32 = np.asarray(x, np.float64).astype(np.float32).astype(np.float64)
    hi = bf16(x32)
    return hi + bf16(x32 - hi)


def exact(x):
    return x


def f16(x):
    """Round to the nearest fp16 value (ties to even; subnormals below
    2^-14), kept in fp64."""
    return np.asarray(x, np.float64).astype(np.float32).astype(np.float16).astype(np.float64)


def attention_rounded_p(q, k, v, rows, n, rp):
    """Counter-causal attention with the probabilities passed through `rp`
    before P V (the row sum taken from the unrounded values)."""
    out = np.zeros(q.shape)
    group = q.shape[1] // k.shape[1]
    for r, i in enumerate(rows):
        if i + 1 >= n:
            continue
        for g in range(k.shape[1]):
            hs = slice(g * group, (g + 1) * group)
            s = q[r, hs] @ R.f64(k[i + 1:n, g]).T / np.sqrt(q.shape[-1])
            p = np.exp(s - s.max(axis=1, keepdims=True))
            out[r, hs] = (rp(p) @ R.f64(v[i + 1:n, g])) / p.sum(axis=1, keepdims=True)
    return out


def fp32(x):
    return x.astype(np.float32).astype(np.float64)


# name -> (query rounding, GEMM-input rounding, P rounding, residual rounding);
# a GEMM-input entry may be a pair (attention-side inputs: normalised input of
# the Q projection and the attention output; MLP inputs: normalised input of
# gate/up and the SwiGLU output)
VARIANTS = {
    "exact": (exact, exact, exact, exact),
    "queries": (bf16, exact, exact, exact),
    "activations": (bf16, bf16, exact, exact),
    "bf16-pass": (bf16, bf16, bf16, fp32),
    "split-act": (bf16, split, bf16, fp32),
    "split-q": (split, split, bf16, fp32),
    "split-all": (split, split, split, fp32),
    "split-qp": (split, bf16, split, fp32),                  # attention operands only
    "split-qp-attn": (split, (split, bf16), split, fp32),    # + the attention-side GEMM inputs
    "split-qp-mlp": (split, (bf16, split), split, fp32),     # + the MLP GEMM inputs
    # every tensor-core operand in fp16: the bf16 weights and cached K/V
    # converted (exact but for magnitudes below 2^-14), the activations,
    # queries and P rounded to fp16
    "fp16-pass": (f16, f16, f16, fp32, f16),
}


def layer(h, rows, pos, lw, k, v, n, shape, rounding):
    rq, ra, rp, rh = rounding[:4]
    if len(rounding) > 4:   # the weights and the cached K/V as the tensor cores see them
        rw = rounding[4]
        lw = {name: rw(w) for name, w in lw.items()}
        k, v = rw(k), rw(v)
    ra, rm = ra if isinstance(ra, tuple) else (ra, ra)   # attention-side, MLP GEMM inputs
    a = ra(R.rms_norm(h, lw["attn_norm"], shape.rms_eps))
    q = (a @ R.f64(lw["wq"]).T).reshape(len(rows), shape.n_q_heads, shape.head_dim)
    q = rq(R.rope(q, pos, shape.rope_theta))
    if rp is exact:
        o = ra(R.counter_causal_attention(q, k, v, rows, n))
    else:
        o = ra(attention_rounded_p(q, k, v, rows, n, rp))
    h = rh(h + o.reshape(len(rows), -1) @ R.f64(lw["wo"]).T)
    m = rm(R.rms_norm(h, lw["mlp_norm"], shape.rms_eps))
    act = rm(R.silu(m @ R.f64(lw["w_gate"]).T) * (m @ R.f64(lw["w_up"]).T))
    return rh(h + act @ R.f64(lw["w_down"]).T)


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--n", type=int, default=16384)
    ap.add_argument("--rows", type=int, default=4)
    ap.add_argument("--seed", type=int, default=3)
    ap.add_argument("--variants", type=str, default=",".join(v for v in VARIANTS if v != "exact"))
    ap.add_argument("--row-list", type=str, default="",
                    help="comma-separated slots to follow (default: --rows evenly spaced)")
    args = ap.parse_args(argv)
    import synth
    from synth.configs import LLAMA3_8B
    shape = LLAMA3_8B
    n, seed = args.n, args.seed
    names = [v for v in args.variants.split(",") if v]
    rows = (np.array([int(x) for x in args.row_list.split(",")]) if args.row_list
            else np.unique(np.linspace(0, n - 3, args.rows).astype(np.int64)))
    toks = synth.tokens((n,), shape.vocab, seed, "study.tokens").numpy()
    emb = synth.normal((shape.vocab, shape.d_model), 0.02, seed, "embed").float().numpy()
    lm = synth.normal((shape.vocab, shape.d_model), 0.02, seed, "lm_head").float().numpy()
    pos = np.arange(n)[rows]
    hs = {v: R.f64(emb[toks[rows]]) for v in ["exact"] + names}
    ones = np.ones(shape.d_model)
    print("layer  " + "  ".join(f"{v:>11s}" for v in names), flush=True)
    for l in range(args.layers):
        lw = {name: synth.normal(shp, 0.02, seed, f"l{l}.{name}").float().numpy() for name, shp in
              (("wq", (shape.q_dim, shape.d_model)), ("wo", (shape.d_model, shape.q_dim)),
               ("w_gate", (shape.d_ff, shape.d_model)), ("w_up", (shape.d_ff, shape.d_model)),
               ("w_down", (shape.d_model, shape.d_ff)))}
        lw["attn_norm"] = lw["mlp_norm"] = ones
        std = synth.kv_std(shape)
        k = synth.normal((n, shape.n_kv_heads, shape.head_dim), std, seed, f"study.k{l}").float().numpy()
        v = synth.normal((n, shape.n_kv_heads, shape.head_dim), std, seed, f"study.v{l}").float().numpy()
        for name in hs:
            hs[name] = layer(hs[name], rows, pos, lw, k, v, n, shape, VARIANTS[name])
        sc = {name: R.score_head(hs[name], toks[rows], ones, lm, "logit", shape.rms_eps)
              for name in hs}
        ref = sc["exact"]
        rms = np.sqrt(np.mean(ref * ref))
        err = {name: float(np.max(np.abs(sc[name] - ref) / np.maximum(np.abs(ref), rms)))
               for name in names}
        print(f"{l:5d}  " + "  ".join(f"{err[v]:11.5f}" for v in names), flush=True)
    # per-row errors after the last layer: the tail of the drift's distribution
    print("after the last layer, per-row error quantiles (50 / 90 / 99 / max):")
    for name in names:
        e = np.abs(sc[name] - ref) / np.maximum(np.abs(ref), rms)
        q = np.quantile(e, [0.5, 0.9, 0.99, 1.0])
        print(f"  {name:12s} " + "  ".join(f"{x:.5f}" for x in q), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
