"""How far does bf16 arithmetic move the exact counter-causal score of a deep
random model?  -- TEST INFRASTRUCTURE (a study script over the oracle).

The oracle computes the full counter-causal pass (Sec. 3.1) in fp64.  A GPU
pass must round some intermediates to bf16 to use the tensor cores.  This
script re-runs the oracle's layer with bf16 rounding inserted at chosen
points and reports, per layer, the score's max relative error against the
exact fp64 pass (the parity metric: |g - o| / max(|o|, rms(o))):

  queries      only the queries entering QK^T are rounded (every other step exact)
  activations  every GEMM input (normalised inputs, attention output,
               SwiGLU output) and the queries are rounded
  bf16-pass    as `activations`, plus the attention probabilities P rounded
               before P V and the residual stream kept in fp32: every rounding
               point of a bf16 tensor-core pass

The drift measured here is a property of the arithmetic and of the random
model, not of any kernel; the 32-layer full-pass tolerances of the parity
tests are derived from it.  It imports only the oracle and the seeded input
generators, never the CUDA path.

    python -m oracle.sensitivity --layers 32 --n 16384 --rows 4
"""
import argparse
import sys

import numpy as np

from . import refresh as R


def bf16(x):
    """Round to the nearest bf16 value (ties to even), kept in fp64."""
    a = np.asarray(x, np.float64).astype(np.float32)
    u = a.view(np.uint32).astype(np.uint64)
    u = (u + 0x7FFF + ((u >> 16) & 1)) & 0xFFFF0000
    return u.astype(np.uint32).view(np.float32).astype(np.float64)


def attention_rounded_p(q, k, v, rows, n):
    """Counter-causal attention with the probabilities rounded to bf16 before
    P V (the row sum taken from the unrounded values)."""
    out = np.zeros(q.shape)
    group = q.shape[1] // k.shape[1]
    for r, i in enumerate(rows):
        if i + 1 >= n:
            continue
        for g in range(k.shape[1]):
            hs = slice(g * group, (g + 1) * group)
            s = q[r, hs] @ R.f64(k[i + 1:n, g]).T / np.sqrt(q.shape[-1])
            p = np.exp(s - s.max(axis=1, keepdims=True))
            out[r, hs] = (bf16(p) @ R.f64(v[i + 1:n, g])) / p.sum(axis=1, keepdims=True)
    return out


def layer(h, rows, pos, lw, k, v, n, shape, round_q, round_act, round_p=False):
    rq = bf16 if round_q else (lambda x: x)
    ra = bf16 if round_act else (lambda x: x)
    rh = (lambda x: x.astype(np.float32).astype(np.float64)) if round_p else (lambda x: x)
    a = ra(R.rms_norm(h, lw["attn_norm"], shape.rms_eps))
    q = (a @ R.f64(lw["wq"]).T).reshape(len(rows), shape.n_q_heads, shape.head_dim)
    q = rq(R.rope(q, pos, shape.rope_theta))
    if round_p:
        o = ra(attention_rounded_p(q, k, v, rows, n))
    else:
        o = ra(R.counter_causal_attention(q, k, v, rows, n))
    h = rh(h + o.reshape(len(rows), -1) @ R.f64(lw["wo"]).T)
    m = ra(R.rms_norm(h, lw["mlp_norm"], shape.rms_eps))
    act = ra(R.silu(m @ R.f64(lw["w_gate"]).T) * (m @ R.f64(lw["w_up"]).T))
    return rh(h + act @ R.f64(lw["w_down"]).T)


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--n", type=int, default=16384)
    ap.add_argument("--rows", type=int, default=4)
    ap.add_argument("--seed", type=int, default=3)
    ap.add_argument("--row-list", type=str, default="",
                    help="comma-separated slots to follow (default: --rows evenly spaced)")
    args = ap.parse_args(argv)
    import synth
    from synth.configs import LLAMA3_8B
    shape = LLAMA3_8B
    n, seed = args.n, args.seed
    rows = (np.array([int(x) for x in args.row_list.split(",")]) if args.row_list
            else np.unique(np.linspace(0, n - 3, args.rows).astype(np.int64)))
    toks = synth.tokens((n,), shape.vocab, seed, "study.tokens").numpy()
    emb = synth.normal((shape.vocab, shape.d_model), 0.02, seed, "embed").float().numpy()
    lm = synth.normal((shape.vocab, shape.d_model), 0.02, seed, "lm_head").float().numpy()
    pos = np.arange(n)[rows]
    variants = {"exact": (False, False, False), "queries": (True, False, False),
                "activations": (True, True, False), "bf16-pass": (True, True, True)}
    hs = {v: R.f64(emb[toks[rows]]) for v in variants}
    ones = np.ones(shape.d_model)
    print("layer  queries  activations  bf16-pass", flush=True)
    for l in range(args.layers):
        lw = {name: synth.normal(shp, 0.02, seed, f"l{l}.{name}").float().numpy() for name, shp in
              (("wq", (shape.q_dim, shape.d_model)), ("wo", (shape.d_model, shape.q_dim)),
               ("w_gate", (shape.d_ff, shape.d_model)), ("w_up", (shape.d_ff, shape.d_model)),
               ("w_down", (shape.d_model, shape.d_ff)))}
        lw["attn_norm"] = lw["mlp_norm"] = ones
        std = synth.kv_std(shape)
        k = synth.normal((n, shape.n_kv_heads, shape.head_dim), std, seed, f"study.k{l}").float().numpy()
        v = synth.normal((n, shape.n_kv_heads, shape.head_dim), std, seed, f"study.v{l}").float().numpy()
        for name, (rq, ra, rp) in variants.items():
            hs[name] = layer(hs[name], rows, pos, lw, k, v, n, shape, rq, ra, rp)
        sc = {name: R.score_head(hs[name], toks[rows], ones, lm, "logit", shape.rms_eps)
              for name in variants}
        ref = sc["exact"]
        rms = np.sqrt(np.mean(ref * ref))
        err = {name: float(np.max(np.abs(sc[name] - ref) / np.maximum(np.abs(ref), rms)))
               for name in ("queries", "activations", "bf16-pass")}
        print(f"{l:5d}  {err['queries']:.4f}   {err['activations']:.4f}       {err['bf16-pass']:.4f}",
              flush=True)
    # per-row errors after the last layer: the tail of the drift's distribution
    print("after the last layer, per-row error quantiles (50 / 90 / 99 / max):")
    for name in ("queries", "activations", "bf16-pass"):
        e = np.abs(sc[name] - ref) / np.maximum(np.abs(ref), rms)
        q = np.quantile(e, [0.5, 0.9, 0.99, 1.0])
        print(f"  {name:12s} " + "  ".join(f"{x:.4f}" for x in q), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
