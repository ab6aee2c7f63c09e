"""Counter-causal refresh oracle for arXiv 2607.27600 -- TEST INFRASTRUCTURE.

A plain, slow, obviously correct fp64 CPU restatement of what one memory
refresh computes: the counter-causal surprise score of every cached token
(Sec. 3.1, full L-layer pass and fast single-layer approximation), the
keep-set (Algorithm DoMemRefresh: argsort, keep the J highest) and the
compaction of the cache to the kept entries.

Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline and
reference legs may import this module.  It shares no code with the CUDA
path and never imports it; the CUDA path never imports this.

Conventions (readings of the paper where it is silent or ambiguous):
  * mask: row i attends keys j with i < j < n (strictly later slots, Sec. 3.1);
  * the score of row i is -(logit of its own token x_i) in the default
    "logit" mode (Sec. 3.1 takes the logit of x_i as the score; keeping the
    highest-surprise tokens means a low logit must rank high), or
    -log P(x_i | x_{i+1:t}) in "logprob" mode (Eq. 5 ranks the same as 1 - P);
  * the last cached slot gets +inf (maximum surprise, Sec. 3.1);
  * a row with no later key (the last one) has attention output 0;
  * layer = Llama/Qwen pre-norm block: RMSNorm -> counter-causal attention ->
    residual -> RMSNorm -> SwiGLU MLP -> residual; final RMSNorm; untied LM head;
  * RoPE: rotate-half pairs (k, k + dh/2), inv_freq_k = theta^(-2k/dh)
    (optionally Llama-3.1 frequency scaling), angles pos * inv_freq_k in
    fp64; attention scale 1/sqrt(head_dim);
  * projections: no biases, except the Qwen2-style q/k/v biases where a
    layer holds them (bq, bk, bv), added before RoPE;
  * GQA: query head t reads KV head t // (Hq / Hkv);
  * keep-set ties are broken toward the later slot; NaN scores rank as -inf;
    sink slots [0, n_sink) are always kept (Sec. 3.2, frozen system prompt);
  * compaction keeps the kept entries in ascending slot (time) order.

Array conventions: weights follow nn.Linear ([out, in]); a cache holds, per
layer, K and V of shape [B, cap, Hkv, dh] (post-RoPE), tokens and pos
[B, cap], seq_len [B] and, for the fast mode, h_last [B, cap, d] = H^(L-1).
Any float dtype is accepted and widened to fp64.
"""
import numpy as np

from .fp8 import kv_quantize

NEG_INF = -np.inf
POS_INF = np.inf


def f64(x):
    return np.asarray(x, dtype=np.float64)


# ----------------------------------------------------------------------------
# Layer pieces (the "standard" transformer layer the paper re-runs, Sec. 3.1)
# ----------------------------------------------------------------------------

def rms_norm(x, gain, eps):
    """x * gain / sqrt(mean(x^2) + eps) over the last axis."""
    x = f64(x)
    return x / np.sqrt(np.mean(x * x, axis=-1, keepdims=True) + eps) * f64(gain)


def rope_inv_freq(head_dim, theta, scaling=None):
    """Rotation frequencies inv_freq_k = theta^(-2k/dh), k < dh/2.

    scaling = (factor, low_freq_factor, high_freq_factor, original_max_pos)
    applies Llama-3.1's frequency scaling (a published model property, not
    part of the paper's method): with wavelength w_k = 2 pi / inv_freq_k,
    pairs whose w_k is shorter than original_max_pos / high_freq_factor keep
    their frequency, pairs longer than original_max_pos / low_freq_factor
    turn factor times slower, and in between the frequency is the blend
    (1 - a) inv_freq_k / factor + a inv_freq_k with a rising linearly in
    original_max_pos / w_k from 0 (at the long edge) to 1 (at the short edge).
    """
    k = np.arange(head_dim // 2, dtype=np.float64)
    inv_freq = float(theta) ** (-2.0 * k / head_dim)
    if scaling is None:
        return inv_freq
    factor, low, high, orig = (float(x) for x in scaling)
    wavelen = 2.0 * np.pi / inv_freq
    a = (orig / wavelen - low) / (high - low)
    blended = (1.0 - a) * inv_freq / factor + a * inv_freq
    out = np.where(wavelen > orig / low, inv_freq / factor, blended)
    return np.where(wavelen < orig / high, inv_freq, out)


def rope_angles(pos, head_dim, theta, scaling=None):
    """Rotation angle pos * inv_freq_k of pair k, for every position in `pos`."""
    return f64(pos)[..., None] * rope_inv_freq(head_dim, theta, scaling)


def rope(x, pos, theta, scaling=None):
    """Rotate-half RoPE of x [..., H, dh] at positions pos [...] (one per row)."""
    x = f64(x)
    dh = x.shape[-1]
    half = dh // 2
    ang = rope_angles(pos, dh, theta, scaling)[..., None, :]      # broadcast over heads
    c, s = np.cos(ang), np.sin(ang)
    x1, x2 = x[..., :half], x[..., half:]
    return np.concatenate([x1 * c - x2 * s, x2 * c + x1 * s], axis=-1)


def project(a, lw, name):
    """a @ W^T for the projection `name` (wq, wk, wv), plus its bias (bq, bk,
    bv) where the layer has one (Qwen2-style attention projections)."""
    y = a @ f64(lw[name]).T
    b = lw.get("b" + name[1:])
    return y if b is None else y + f64(b)


def softmax(s):
    s = f64(s)
    e = np.exp(s - np.max(s, axis=-1, keepdims=True))
    return e / np.sum(e, axis=-1, keepdims=True)


def counter_causal_attention(q, k, v, rows, n):
    """Counter-causal scaled dot-product attention (Sec. 3.1, Eq. 2 with the
    upper-triangular mask).

    q: [R, Hq, dh] fresh queries of cache rows `rows`; k, v: [cap, Hkv, dh]
    cached (post-RoPE) keys and values of one sequence, of which the first n
    are valid.  Row i attends only keys j with i < j < n; a row with no such
    key returns 0.  Returns [R, Hq, dh].
    """
    q, rows = f64(q), np.asarray(rows)
    n_rows, hq, dh = q.shape
    hkv = k.shape[1]
    group = hq // hkv
    out = np.zeros((n_rows, hq, dh))
    for r in range(n_rows):
        i = int(rows[r])
        if i + 1 >= n:
            continue
        for g in range(hkv):
            kj = f64(k[i + 1:n, g])                     # [n-i-1, dh]
            vj = f64(v[i + 1:n, g])
            heads = slice(g * group, (g + 1) * group)
            s = q[r, heads] @ kj.T / np.sqrt(dh)       # [group, n-i-1]
            out[r, heads] = softmax(s) @ vj
    return out


def causal_attention(q, k, v):
    """Standard causal attention (row i attends j <= i), used only to build a
    cache by a causal forward.  q [n, Hq, dh], k, v [n, Hkv, dh]."""
    q = f64(q)
    n, hq, dh = q.shape
    hkv = k.shape[1]
    group = hq // hkv
    out = np.zeros((n, hq, dh))
    for i in range(n):
        for g in range(hkv):
            heads = slice(g * group, (g + 1) * group)
            s = q[i, heads] @ f64(k[:i + 1, g]).T / np.sqrt(dh)
            out[i, heads] = softmax(s) @ f64(v[:i + 1, g])
    return out


def silu(x):
    return x / (1.0 + np.exp(-x))


def swiglu_mlp(m, lw):
    """SwiGLU MLP: (silu(m Wg^T) * (m Wu^T)) Wd^T."""
    g = m @ f64(lw["w_gate"]).T
    u = m @ f64(lw["w_up"]).T
    return (silu(g) * u) @ f64(lw["w_down"]).T


def counter_causal_layer(h, rows, pos_rows, lw, k, v, n, shape):
    """One transformer layer re-run under the counter-causal mask (Sec. 3.1):
    fresh queries from the rows' own hidden states at their original
    positions, cached K/V reused (not recomputed).  h: [R, d] -> [R, d]."""
    a = rms_norm(h, lw["attn_norm"], shape.rms_eps)
    q = project(a, lw, "wq").reshape(len(rows), shape.n_q_heads, shape.head_dim)
    q = rope(q, pos_rows, shape.rope_theta, getattr(shape, "rope_scaling", None))
    o = counter_causal_attention(q, k, v, rows, n)
    h = h + o.reshape(len(rows), -1) @ f64(lw["wo"]).T
    m = rms_norm(h, lw["mlp_norm"], shape.rms_eps)
    return h + swiglu_mlp(m, lw)


def logsumexp_rows(x):
    m = np.max(x, axis=-1)
    return m + np.log(np.sum(np.exp(x - m[:, None]), axis=-1))


def score_head(h, tok, final_norm, lm_head, mode, eps, vocab_chunk=16384):
    """Surprise score of each row from its final hidden state (Sec. 3.1).

    logit mode: -z_i[x_i] with z_i = RMSNorm(h_i) W_U^T; logprob mode:
    -(z_i[x_i] - logsumexp(z_i)) = -log P(x_i | later context)."""
    u = rms_norm(h, final_norm, eps)
    z_tgt = np.sum(u * f64(lm_head[np.asarray(tok)]), axis=-1)
    if mode == "logit":
        return -z_tgt
    if mode != "logprob":
        raise ValueError(f"unknown score mode {mode!r}")
    vocab = lm_head.shape[0]
    logits = np.empty((u.shape[0], vocab))
    for c0 in range(0, vocab, vocab_chunk):
        c1 = min(vocab, c0 + vocab_chunk)
        logits[:, c0:c1] = u @ f64(lm_head[c0:c1]).T
    return -(z_tgt - logsumexp_rows(logits))


# ----------------------------------------------------------------------------
# Scoring (Sec. 3.1; Algorithm DoMemRefresh, its surprise loop)
# ----------------------------------------------------------------------------

def _rows_of(rows, b, n):
    if rows is None or rows[b] is None:
        return np.arange(n)
    r = np.asarray(rows[b], dtype=np.int64)
    if r.size and (r.min() < 0 or r.max() >= n):
        raise ValueError("row outside the sequence")
    return r


def _finish(scores_b, r, n):
    s = scores_b.copy()
    s[r == n - 1] = POS_INF          # last slot: no future context, maximum surprise
    return s


def score_layer(shape, weights, cache, mode="logit", rows=None):
    """Fast single-layer approximation (Sec. 3.1, 'Fast single-layer
    approximation'): queries from the stored H^(L-1), counter-causal attention
    over the last layer's cached K/V, the rest of the last layer, the head.

    rows: optional per-sequence list of slot indices to score (None = all).
    Returns scores [B, cap]: scored rows hold their score, others -inf.
    """
    last = shape.n_layers - 1
    lw = weights["layers"][last]
    seq_len = np.asarray(cache["seq_len"])
    bsz, cap = cache["tokens"].shape
    out = np.full((bsz, cap), NEG_INF)
    for b in range(bsz):
        n = int(seq_len[b])
        r = _rows_of(rows, b, n)
        if r.size == 0:
            continue
        h = f64(cache["h_last"][b][r])
        h = counter_causal_layer(h, r, cache["pos"][b][r], lw, cache["k"][last][b],
                                 cache["v"][last][b], n, shape)
        s = score_head(h, cache["tokens"][b][r], weights["final_norm"], weights["lm_head"],
                       mode, shape.rms_eps)
        out[b, r] = _finish(s, r, n)
    return out


def score_full(shape, weights, cache, mode="logit", rows=None):
    """Full counter-causal pass (Sec. 3.1): the model re-run on the cached
    tokens in original order, every layer with fresh queries over its own
    cached K/V, then the head.  Same returns as score_layer."""
    seq_len = np.asarray(cache["seq_len"])
    bsz, cap = cache["tokens"].shape
    out = np.full((bsz, cap), NEG_INF)
    for b in range(bsz):
        n = int(seq_len[b])
        r = _rows_of(rows, b, n)
        if r.size == 0:
            continue
        h = f64(weights["embed"][np.asarray(cache["tokens"][b][r])])
        for l in range(shape.n_layers):
            h = counter_causal_layer(h, r, cache["pos"][b][r], weights["layers"][l],
                                     cache["k"][l][b], cache["v"][l][b], n, shape)
        s = score_head(h, cache["tokens"][b][r], weights["final_norm"], weights["lm_head"],
                       mode, shape.rms_eps)
        out[b, r] = _finish(s, r, n)
    return out


# ----------------------------------------------------------------------------
# Keep-set selection and compaction (Algorithm DoMemRefresh)
# ----------------------------------------------------------------------------

def select_keep(scores, seq_len, budget, n_sink=0):
    """Keep the min(budget_b, n_b) highest-scoring slots of each sequence.

    Order: descending score, ties toward the later slot; NaN ranks as -inf;
    slots [0, n_sink) rank as +inf (frozen).  The kept slots are returned in
    ascending slot order.  scores are taken as given (fp32 in, compared
    exactly).  Returns keep_idx [B, cap] (-1 past the count), keep_count [B].
    """
    scores = np.asarray(scores)
    bsz, cap = scores.shape
    keep_idx = np.full((bsz, cap), -1, dtype=np.int32)
    keep_count = np.zeros(bsz, dtype=np.int32)
    for b in range(bsz):
        n = int(seq_len[b])
        j = min(int(budget[b]), n)
        s = scores[b, :n].astype(np.float64)   # exact widening of the fp32 values
        s = np.where(np.isnan(s), NEG_INF, s)
        s[:min(n_sink, n)] = POS_INF
        slot = np.arange(n)
        order = np.lexsort((-slot, -s))        # primary: score desc; then slot desc
        kept = np.sort(order[:j])
        keep_idx[b, :j] = kept
        keep_count[b] = j
    return keep_idx, keep_count


def compact(buf, keep_idx, keep_count):
    """Compaction K' <- (K' (+) K)_sigma[1:J] along the slot axis (axis 1) of
    buf [B, cap, ...]: slot k of sequence b receives old slot keep_idx[b, k]
    for k < keep_count[b]; the other slots keep their old contents."""
    buf = np.asarray(buf)
    out = buf.copy()
    for b in range(buf.shape[0]):
        j = int(keep_count[b])
        out[b, :j] = buf[b, np.asarray(keep_idx[b, :j], dtype=np.int64)]
    return out


# ----------------------------------------------------------------------------
# Causal forward: builds a cache the way the inference cycle fills it
# (Algorithm DoInference: k_t, v_t, x_t appended as tokens are processed)
# ----------------------------------------------------------------------------

def causal_forward(shape, weights, tokens, pos):
    """Standard causal forward of one sequence.  Returns the cache it leaves:
    K, V per layer (post-RoPE, [n, Hkv, dh]), H^(L-1) ([n, d], the input of
    the last layer, recorded for the fast approximation) and the final hidden
    states ([n, d])."""
    n = len(tokens)
    h = f64(weights["embed"][np.asarray(tokens)])
    ks, vs, h_last = [], [], None
    for l in range(shape.n_layers):
        lw = weights["layers"][l]
        if l == shape.n_layers - 1:
            h_last = h.copy()
        a = rms_norm(h, lw["attn_norm"], shape.rms_eps)
        sc = getattr(shape, "rope_scaling", None)
        q = rope(project(a, lw, "wq").reshape(n, shape.n_q_heads, shape.head_dim), pos,
                 shape.rope_theta, sc)
        k = rope(project(a, lw, "wk").reshape(n, shape.n_kv_heads, shape.head_dim), pos,
                 shape.rope_theta, sc)
        v = project(a, lw, "wv").reshape(n, shape.n_kv_heads, shape.head_dim)
        ks.append(k)
        vs.append(v)
        o = causal_attention(q, k, v)
        h = h + o.reshape(n, -1) @ f64(lw["wo"]).T
        m = rms_norm(h, lw["mlp_norm"], shape.rms_eps)
        h = h + swiglu_mlp(m, lw)
    return {"k": ks, "v": vs, "h_last": h_last, "h_final": h}


# ----------------------------------------------------------------------------
# Inference cycle in pre-fill (Algorithm CacheManagedInference / DoInference,
# chunked mode): a chunk of new tokens runs causally through every layer over
# the memory the cache holds, and their K, V, tokens, positions and H^(L-1)
# are appended
# ----------------------------------------------------------------------------

def memory_causal_attention(q, k, v, n0):
    """Memory-augmented causal attention (Eq. 3 with the causal mask): chunk
    row r (cache slot n0 + r) attends every memory slot j < n0 and the chunk
    slots up to and including its own, i.e. keys j <= n0 + r of the
    concatenation [K' ; K].  q [h, Hq, dh]; k, v [>= n0 + h, Hkv, dh]."""
    q = f64(q)
    h, hq, dh = q.shape
    hkv = k.shape[1]
    group = hq // hkv
    out = np.zeros((h, hq, dh))
    for r in range(h):
        last = n0 + r
        for g in range(hkv):
            heads = slice(g * group, (g + 1) * group)
            s = q[r, heads] @ f64(k[:last + 1, g]).T / np.sqrt(dh)
            out[r, heads] = softmax(s) @ f64(v[:last + 1, g])
    return out


def append_chunk(shape, weights, cache, b, tokens, pos=None):
    """Append a chunk of tokens to sequence b of `cache` (modified in place):
    the inference cycle of Algorithm DoInference run over a chunk in batch, as
    in pre-fill.  Per layer the chunk's queries, keys and values come from its
    own hidden states (keys and queries rotated at the chunk's positions), the
    keys and values are written after the sequence's current slots
    (K <- K (+) k_t, V <- V (+) v_t; in an e4m3 cache, one with
    cache["kv_scale"][l] = (K scale, V scale), as the cache stores them:
    fp8.kv_quantize), and attention sees the memory slots
    already cached plus the chunk causally (memory_causal_attention).  The
    tokens (X <- X (+) x_t), positions and H^(L-1) (the input of the last
    layer, recorded for the fast approximation) are written too, and
    seq_len[b] grows by the chunk length.  pos defaults to the positions
    following the last cached one.  Returns the chunk's final hidden states."""
    n0 = int(cache["seq_len"][b])
    tokens = np.asarray(tokens)
    h = len(tokens)
    if pos is None:
        start = int(cache["pos"][b][n0 - 1]) + 1 if n0 > 0 else 0
        pos = np.arange(start, start + h)
    pos = np.asarray(pos)
    sl = slice(n0, n0 + h)
    x = f64(weights["embed"][tokens])
    sc = getattr(shape, "rope_scaling", None)
    for l in range(shape.n_layers):
        lw = weights["layers"][l]
        if l == shape.n_layers - 1 and cache.get("h_last") is not None:
            cache["h_last"][b][sl] = x
        a = rms_norm(x, lw["attn_norm"], shape.rms_eps)
        q = rope(project(a, lw, "wq").reshape(h, shape.n_q_heads, shape.head_dim), pos,
                 shape.rope_theta, sc)
        k = rope(project(a, lw, "wk").reshape(h, shape.n_kv_heads, shape.head_dim), pos,
                 shape.rope_theta, sc)
        v = project(a, lw, "wv").reshape(h, shape.n_kv_heads, shape.head_dim)
        if cache.get("kv_scale") is not None:   # e4m3 cache: rows stored as code * scale
            k = kv_quantize(k, cache["kv_scale"][l][0])
            v = kv_quantize(v, cache["kv_scale"][l][1])
        cache["k"][l][b][sl] = k
        cache["v"][l][b][sl] = v
        o = memory_causal_attention(q, cache["k"][l][b], cache["v"][l][b], n0)
        x = x + o.reshape(h, -1) @ f64(lw["wo"]).T
        m = rms_norm(x, lw["mlp_norm"], shape.rms_eps)
        x = x + swiglu_mlp(m, lw)
    cache["tokens"][b][sl] = tokens
    cache["pos"][b][sl] = pos
    cache["seq_len"][b] = n0 + h
    return x


# ----------------------------------------------------------------------------
# The paper's comparison scorers (Sec. 4): sliding window, importance, H2O.
# They rank the same cached slots for the same keep-set selection and
# compaction; the attention-based ones use cached keys as proxy queries.
# ----------------------------------------------------------------------------

def recency_scores(cache):
    """Sliding window (first in, first out): the score of a slot is its
    original position, so the keep-set is the most recent slots."""
    pos = np.asarray(cache["pos"])
    seq_len = np.asarray(cache["seq_len"])
    out = np.full(pos.shape, NEG_INF)
    for b in range(pos.shape[0]):
        n = int(seq_len[b])
        out[b, :n] = pos[b, :n]
    return out


def key_attention_colsums(k, n, q_lo):
    """Attention received by each key under the causal mask when the keys of
    slots [q_lo, n) act as queries (proxy queries, Sec. 4): for each KV head
    g, A_g = softmax over j <= i of K_g[i] . K_g[j] / sqrt(dh); returns
    c[j] = sum_g sum_{i in [q_lo, n), i >= j} A_g[i, j] for j < n.
    k: [>= n, Hkv, dh]."""
    k = f64(k)
    hkv, dh = k.shape[1], k.shape[2]
    c = np.zeros(n)
    for g in range(hkv):
        for i in range(q_lo, n):
            s = k[:i + 1, g] @ k[i, g] / np.sqrt(dh)
            c[:i + 1] += softmax(s)
    return c


def importance_scores(shape, cache):
    """Importance (Sec. 4, after TOVA): the mean attention a token receives in
    the last layer, with the layer's cached keys as proxy queries and the
    causal mask: score_j = c[j] / (Hkv * (n - j)), c from
    key_attention_colsums over every query slot (the n - j queries that see
    slot j, in each KV head).  Low mean attention is evicted first."""
    seq_len = np.asarray(cache["seq_len"])
    kl = cache["k"][shape.n_layers - 1]
    bsz, cap = kl.shape[0], kl.shape[1]
    out = np.full((bsz, cap), NEG_INF)
    for b in range(bsz):
        n = int(seq_len[b])
        if n == 0:
            continue
        c = key_attention_colsums(kl[b], n, 0)
        out[b, :n] = c / (shape.n_kv_heads * (n - np.arange(n)))
    return out


def h2o_update(shape, cache, acc, recent):
    """Heavy-hitter (H2O, Sec. 4): adds to the running total acc [B, cap] the
    attention each slot receives from the `recent` most recent keys as proxy
    queries (causal mask), summed over KV heads and every layer."""
    seq_len = np.asarray(cache["seq_len"])
    for b in range(acc.shape[0]):
        n = int(seq_len[b])
        q_lo = max(0, n - int(recent))
        for l in range(shape.n_layers):
            acc[b, :n] += key_attention_colsums(cache["k"][l][b], n, q_lo)
    return acc


def h2o_scores(acc, seq_len, recent):
    """Refresh scores of H2O: the accumulated attention, with the `recent`
    most recent slots always kept (+inf); only older slots are evicted."""
    out = np.full(np.shape(acc), NEG_INF)
    for b in range(out.shape[0]):
        n = int(seq_len[b])
        out[b, :n] = acc[b, :n]
        out[b, max(0, n - int(recent)):n] = POS_INF
    return out


def decode_step(shape, weights, cache, tokens):
    """One decode step of the inference cycle (Algorithm DoInference for a
    single token, greedy sampling as in the paper's experiments): each
    sequence's current token x_t is appended (append_chunk with one token:
    its K, V and H^(L-1) through every layer, attending the memory and
    itself), and the final norm and LM head give the logits of the next
    token.  Returns (next tokens [B], their logits [B], all logits [B, V]);
    ties go to the lowest token id."""
    bsz = len(tokens)
    nxt = np.zeros(bsz, dtype=np.int64)
    best = np.zeros(bsz)
    logits = np.zeros((bsz, shape.vocab))
    for b in range(bsz):
        x = append_chunk(shape, weights, cache, b, [int(tokens[b])])
        u = rms_norm(x, weights["final_norm"], shape.rms_eps)
        logits[b] = (u @ f64(weights["lm_head"]).T)[0]
        nxt[b] = int(np.argmax(logits[b]))
        best[b] = logits[b, nxt[b]]
    return nxt, best, logits
