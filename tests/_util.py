"""Shared test helpers: numpy views of synthetic inputs and tiny caches built
by the oracle's causal forward."""
import numpy as np
import torch

import synth
from synth.configs import ModelShape

# small shape with d != Hq*dh != d_ff so that a transposed operand fails loudly
SMALL = ModelShape(n_layers=2, d_model=48, n_q_heads=4, n_kv_heads=2, head_dim=16, d_ff=80,
                   vocab=50, rope_theta=1e4, rms_eps=1e-5)


def to_np(x):
    """torch tensors (any nesting of dict/list) -> numpy (bf16 widened to fp32)."""
    if x is None:
        return None
    if isinstance(x, dict):
        return {k: to_np(v) for k, v in x.items()}
    if isinstance(x, (list, tuple)):
        return [to_np(v) for v in x]
    if isinstance(x, torch.Tensor):
        t = x.detach().cpu()
        if t.dtype in (torch.bfloat16, torch.float16):
            t = t.float()
        return t.numpy()
    return x


def bf16_round(a):
    """Round an fp64/fp32 numpy array to the nearest bf16 value (kept as fp32)."""
    return torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.bfloat16).float().numpy()


def causal_cache(shape, weights_np, seq_lens, cap, seed, round_bf16=True):
    """Cache left by a causal forward of the random model over seeded tokens
    (the tiny workload's recipe).  Slots past a sequence's end hold zeros."""
    import oracle
    b = len(seq_lens)
    toks = synth.tokens((b, cap), shape.vocab, seed, "cache.tokens").numpy()
    pos = np.tile(np.arange(cap, dtype=np.int32), (b, 1))
    k = [np.zeros((b, cap, shape.n_kv_heads, shape.head_dim), np.float32)
         for _ in range(shape.n_layers)]
    v = [np.zeros_like(k[0]) for _ in range(shape.n_layers)]
    h_last = np.zeros((b, cap, shape.d_model), np.float32)
    rnd = bf16_round if round_bf16 else (lambda a: np.asarray(a, np.float32))
    for bi, n in enumerate(seq_lens):
        if n == 0:
            continue
        fw = oracle.causal_forward(shape, weights_np, toks[bi, :n], pos[bi, :n])
        for l in range(shape.n_layers):
            k[l][bi, :n] = rnd(fw["k"][l])
            v[l][bi, :n] = rnd(fw["v"][l])
        h_last[bi, :n] = rnd(fw["h_last"])
    return {"k": k, "v": v, "tokens": toks.astype(np.int32), "pos": pos,
            "seq_len": np.asarray(seq_lens, np.int32), "h_last": h_last}


def small_model(shape=SMALL, seed=0, with_kv_proj=True):
    return to_np(synth.model_weights(shape, seed, with_kv_proj=with_kv_proj))


def rel_err(got, want):
    """max |g - o| / max(|o|, rms(o)) over entries where want is finite; infinite
    entries must match exactly (returns inf otherwise)."""
    got, want = np.asarray(got, np.float64), np.asarray(want, np.float64)
    fin = np.isfinite(want)
    if not np.array_equal(got[~fin], want[~fin]):
        return np.inf
    if not fin.any():
        return 0.0
    g, o = got[fin], want[fin]
    rms = np.sqrt(np.mean(o * o))
    return float(np.max(np.abs(g - o) / np.maximum(np.abs(o), rms)))


def to_device(x, device="cuda"):
    """numpy tree -> torch tree on `device`: floats as bf16, integers as int32."""
    if x is None:
        return None
    if isinstance(x, dict):
        return {k: to_device(v, device) for k, v in x.items()}
    if isinstance(x, (list, tuple)):
        return [to_device(v, device) for v in x]
    a = np.ascontiguousarray(x)
    t = torch.from_numpy(a)
    t = t.to(torch.bfloat16) if a.dtype.kind == "f" else t.to(torch.int32)
    return t.to(device)


def keep_set_ok(got_idx, got_cnt, want_idx, want_cnt, oracle_scores, seq_lens, budgets, tol=2e-2,
                min_overlap=0.995):
    """Keep-set bar (the keep-set is the top-J slots by score): identical
    where the oracle's score gap at the budget boundary exceeds `tol`
    (relative to the scores' rms); otherwise at least `min_overlap` of the
    oracle's kept slots kept (99.5 %: at J < 200 that allows no swap at all),
    and every slot kept by one side only a near tie -- its oracle score within
    `tol` x rms of the oracle's J-th score, where rounding of scores within the
    bar may order them either way.  Returns (ok, details): per sequence
    (b, gap, overlap, slots kept by one side only)."""
    details = []
    ok = True
    for b, (n, j) in enumerate(zip(seq_lens, budgets)):
        jj = min(j, n)
        g = set(np.asarray(got_idx[b, :got_cnt[b]]).tolist())
        w = set(np.asarray(want_idx[b, :want_cnt[b]]).tolist())
        if got_cnt[b] != want_cnt[b]:
            return False, f"count {got_cnt[b]} != {want_cnt[b]}"
        s = np.asarray(oracle_scores[b, :n], np.float64)
        fin = s[np.isfinite(s)]
        rms = np.sqrt(np.mean(fin * fin)) if fin.size else 1.0
        srt = np.sort(s)[::-1]
        gap = (srt[jj - 1] - srt[jj]) / rms if jj < n else np.inf
        diff = sorted(g ^ w)
        overlap = len(g & w) / max(1, len(w))
        if gap > tol:
            ok &= g == w
        else:
            thr = srt[jj - 1]
            ok &= overlap >= min_overlap
            ok &= all(np.isfinite(s[i]) and abs(s[i] - thr) <= tol * rms for i in diff)
        details.append((b, gap, overlap, len(diff)))
    return bool(ok), details
