"""Benchmark of one counter-causal memory refresh (arXiv 2607.27600,
Sec. 3.1 and Algorithm DoMemRefresh) on GB300.

A step = one refresh of one synthetic cache: counter-causal scores of every
cached position (fast single-layer approximation, or the full L-layer pass),
keep-set selection at the budget, in-place compaction of every layer's K/V,
H^(L-1), tokens and positions.  Metric: scored KV positions per second.
The scoring pass runs with fp16 tensor-core operands (CC_SCORE_F16: the
fastest mode that holds the full 32-layer pass to the stated tolerance; the
layer weights are converted once before the timed steps) unless --bf16 or
--precise names another operand mode.

    python bench.py [--gpus N --steps K --warmup W] [--workload NAME] [--impl reference]

Our arm times K steps with CUDA events on the launching stream (inputs
resident in HBM; the cache is restored and 256 MiB written to flush L2
between steps, outside the timed events), runs K more steps with CUDA
events around every library launch for the per-kernel table (gpu_launches
counts those K steps' launches), then K end-to-end steps through
the public API with host inputs (pinned host -> device copies of the step's
inputs and device -> host read of the keep-set inside the timed region).
The reference arm (--impl reference) times the CPU oracle on a bounded row
sample of the same workload.  Under torchrun each rank runs an independent
replica (no collective on the data path) and rank 0 prints one JSON line.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

PEAKS_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
L2_FLUSH_BYTES = 256 << 20


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return PEAKS_FALLBACK, "fallback"


# ---------------------------------------------------------------------------
# distributed plumbing (one process per GPU, independent replicas)
# ---------------------------------------------------------------------------

class Dist:
    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch.distributed as dist
            backend = "nccl" if torch.cuda.is_available() else "gloo"
            if backend == "nccl":
                torch.cuda.set_device(self.local)
            dist.init_process_group(backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            if torch.cuda.is_available():
                self.pg.barrier(device_ids=[self.local])
            else:
                self.pg.barrier()

    def max(self, x: float) -> float:
        if not self.pg:
            return x
        dev = f"cuda:{self.local}" if torch.cuda.is_available() else "cpu"
        t = torch.tensor([x], dtype=torch.float64, device=dev)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


# ---------------------------------------------------------------------------
# clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.samples = []
        self.proc = None
        try:
            bus = torch.cuda.get_device_properties(device_index).pci_bus_id
        except Exception:
            bus = str(device_index)
        self.cmd = ["nvidia-smi", "-i", str(bus), f"--query-gpu={self.FIELDS}",
                    "--format=csv,noheader,nounits", "-lms", "100"]
        self.thread = None

    def start(self):
        try:
            self.proc = subprocess.Popen(self.cmd, stdout=subprocess.PIPE,
                                         stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None
            return
        self.thread = threading.Thread(target=self._read, daemon=True)
        self.thread.start()

    def _read(self):
        for line in self.proc.stdout:
            parts = [x.strip() for x in line.split(",")]
            if len(parts) >= 8:
                self.samples.append(parts)

    def stop(self) -> dict:
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        if self.thread:
            self.thread.join(timeout=5)

        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(s[0]) for s in self.samples if num(s[0]) is not None]
        mx = [num(s[1]) for s in self.samples if num(s[1]) is not None]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for s in self.samples for i in range(4)
                          if s[4 + i].lower() == "active"})
        loaded = [v for v in sm if mx and v > 0.5 * max(mx)] or sm
        return {"sm_mhz": statistics.median(loaded) if loaded else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(self.samples)}


# ---------------------------------------------------------------------------
# workload setup
# ---------------------------------------------------------------------------

def make_inputs(wl, device, kv_fp8=False, paged=0, head_major=False):
    """Weights and cache of the workload on `device` (seeded synthetic)."""
    shape = wl.shape
    fast = wl.mode == "layer"
    layers = [shape.n_layers - 1] if fast else None
    w = synth.model_weights(shape, wl.seed, device=device, layers=layers, with_embed=not fast)
    # the refresh compacts every layer's cache; the fast pass reads only the last layer's
    cache = synth.synthetic_cache(shape, wl.seq_lens, wl.cap, wl.seed, device=device,
                                  with_h_last=fast)
    if kv_fp8:
        to_e4m3_cache(cache)
    if paged:
        to_paged_cache(cache, paged, wl.seed)
    if head_major:   # [B, Hkv, cap, dh] buffers
        for key in ("k", "v"):
            cache[key] = [x.permute(0, 2, 1, 3).contiguous() for x in cache[key]]
        cache["kv_layout"] = 1
    return w, cache


def to_paged_cache(cache, page, seed):
    """The cache's K/V moved into page pools (pages of `page` slots in a
    seeded random order) with a block table; the slot-major buffers freed."""
    b, cap = cache["tokens"].shape
    per = cap // page
    perm = np.random.default_rng(seed).permutation(b * per).reshape(b, per)
    dev = cache["tokens"].device
    idx = torch.from_numpy(perm.reshape(-1)).to(dev).long()
    for key in ("k", "v"):
        for l, x in enumerate(cache[key]):
            pool = torch.empty((b * per, page) + tuple(x.shape[2:]), dtype=x.dtype, device=dev)
            pool[idx] = x.reshape((b * per, page) + tuple(x.shape[2:]))
            cache[key][l] = pool
            del x
    cache["block_table"] = torch.from_numpy(perm.astype(np.int32)).to(dev)
    cache["page_size"] = page
    return cache


def logical_kv(cache, key, l):
    """Slot-major [B, cap, Hkv, dh] view of K or V layer l (gathered from the
    pages of a paged cache)."""
    x = cache[key][l]
    if cache.get("kv_layout", 0) == 1:
        return x.permute(0, 2, 1, 3)
    if cache.get("block_table") is None:
        return x
    t = cache["block_table"].long()
    b, per = t.shape
    return x[t.reshape(-1)].reshape((b, per * cache["page_size"]) + tuple(x.shape[2:]))


def to_e4m3_cache(cache, headroom=2.0):
    """The synthetic cache stored as e4m3 codes: per layer and tensor scale =
    max |x| * headroom / 448, codes cast by torch (float8_e4m3fn); the scales
    go to cache["kv_scale"]."""
    scales = []
    for l in range(len(cache["k"])):
        pair = []
        for key in ("k", "v"):
            x = cache[key][l].float()
            sc = max(float(x.abs().max()), 1e-3) * headroom / 448.0
            cache[key][l] = (x / sc).to(torch.float8_e4m3fn).view(torch.uint8)
            pair.append(sc)
            del x
        scales.append(tuple(pair))
    cache["kv_scale"] = scales
    return cache


def clone_cache(c):
    def cl(x):
        return x.clone() if isinstance(x, torch.Tensor) else x
    return {k: ([cl(x) for x in v] if isinstance(v, list) else cl(v)) for k, v in c.items()}


def restore_cache(dst, src):
    for k, v in src.items():
        if isinstance(v, list):
            for a, b in zip(dst[k], v):
                if isinstance(a, torch.Tensor):
                    a.copy_(b, non_blocking=True)
        elif isinstance(v, torch.Tensor):
            dst[k].copy_(v, non_blocking=True)


def algorithmic_work(wl, kv_bytes=2):
    """Per-launch algorithmic FLOPs / bytes of each kernel kind for one step
    (kv_bytes: bytes per cached K/V element, 1 for the e4m3 cache)."""
    s = wl.shape
    n_rows = sum(wl.seq_lens)
    d, qd, f, hq, dh = s.d_model, s.q_dim, s.d_ff, s.n_q_heads, s.head_dim
    pairs = sum(n * (n - 1) for n in wl.seq_lens)          # 2 x (pairs j > i)
    kv_row = s.kv_dim * kv_bytes
    moved = sum(max(0, min(b, n)) for b, n in zip(wl.budgets, wl.seq_lens))
    n_arrays_kv = 2 * s.n_layers
    h_row = d * 2 if wl.mode == "layer" else 0
    return {
        "gemm_qrope": ("tensor", 2.0 * n_rows * d * qd),
        "attention": ("tensor", 2.0 * dh * hq * pairs),
        "gemm_oproj": ("tensor", 2.0 * n_rows * qd * d),
        "gemm_gateup": ("tensor", 4.0 * n_rows * d * f),
        "gemm_down": ("tensor", 2.0 * n_rows * f * d),
        # combine of the down projection's per-tile (sum h^2, sum h g W_U[x_i]) partials
        # (the gather-dot itself runs in that GEMM's epilogue): partials and token
        # read, score written
        "head_logit": ("hbm", n_rows * (8.0 * -(-d // 256) + 8.0)),
        "gemm_lmhead": ("tensor", 2.0 * n_rows * d * s.vocab),
        # the pre-attention norm (the post-attention one is fused into the O / gate-up
        # GEMMs): input row read (bf16 H^(L-1) in layer mode, fp32 h in the full
        # pass), bf16 row written
        "rmsnorm": ("hbm", n_rows * ((2.0 if wl.mode == "layer" else 4.0) * d + 2.0 * d)),
        # each kept slot: read + write of every layer's K and V row, H row, token, position
        "compact": ("hbm", 2.0 * moved * (n_arrays_kv * kv_row + h_row + 8)),
        # at most 9 passes over the scores (up to 8 radix passes + the emit pass)
        "select": ("hbm", 9.0 * 4.0 * n_rows),
        # a layer's K and V read (e4m3 codes, or bf16 in the fp16 operand mode)
        # and their 2-byte copies written (per launch)
        "kv_dequant": ("hbm", n_rows * 2.0 * s.n_kv_heads * dh * (kv_bytes + 2.0)),
    }


def keyattn_work(wl, scorer, recent):
    """FLOPs of one keyattn launch pair (both sweeps: S = K K^T over the
    causal (query, key) pairs of the proxy queries, 2 dh per pair and head,
    for the last layer (importance) or every layer (H2O))."""
    s = wl.shape
    pairs = 0
    for n in wl.seq_lens:
        q_lo = 0 if scorer == "importance" else max(0, n - recent)
        pairs += sum(i + 1 for i in range(q_lo, n))
    layers = 1 if scorer == "importance" else s.n_layers   # H2O: every layer in one launch
    return ("tensor", 2 * 2.0 * s.head_dim * s.n_kv_heads * pairs * layers)


def step_flops(wl):
    s = wl.shape
    w = algorithmic_work(wl)
    lay = 1 if wl.mode == "layer" else s.n_layers
    per_layer = sum(w[k][1] for k in ("gemm_qrope", "attention", "gemm_oproj", "gemm_gateup",
                                      "gemm_down"))
    return lay * per_layer + 2.0 * sum(wl.seq_lens) * s.d_model


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------

def causal_pass_cache(wl, w, dev, chunk=4096):
    """The workload's cache as the inference cycle leaves it (Algorithm
    CacheManagedInference in pre-fill): a causal pass of the random model over
    seeded uniform token ids, appended chunk by chunk with cc_append_chunk
    (every layer's post-RoPE K/V, tokens, positions 0..n-1 and, for the fast
    pass, H^(L-1)).  Slots past a sequence's end stay zero.  Untimed set-up."""
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    shape, b, cap = wl.shape, wl.batch, wl.cap
    kv = (b, cap, shape.n_kv_heads, shape.head_dim)
    cache = {"k": [torch.zeros(kv, dtype=torch.bfloat16, device=dev) for _ in range(shape.n_layers)],
             "v": [torch.zeros(kv, dtype=torch.bfloat16, device=dev) for _ in range(shape.n_layers)],
             "tokens": torch.zeros(b, cap, dtype=torch.int32, device=dev),
             "pos": torch.zeros(b, cap, dtype=torch.int32, device=dev),
             "seq_len": torch.zeros(b, dtype=torch.int32, device=dev),
             "h_last": (torch.zeros(b, cap, shape.d_model, dtype=torch.bfloat16, device=dev)
                        if wl.mode == "layer" else None)}
    toks = synth.tokens((b, cap), shape.vocab, wl.seed, "bench.cache.tokens", dev)
    weights, kc = pkg.Weights(w), pkg.Cache(cache)
    ws = cc.alloc_workspace(cc.cc_append_workspace_size(shape, b, cap), dev)
    for s0 in range(0, max(wl.seq_lens), chunk):
        cnt = torch.tensor([max(0, min(chunk, n - s0)) for n in wl.seq_lens], dtype=torch.int32,
                           device=dev)
        tin = torch.zeros(b, chunk, dtype=torch.int32, device=dev)
        width = min(chunk, cap - s0)
        tin[:, :width] = toks[:, s0:s0 + width]
        cc.cc_append_chunk(shape, weights, kc, tin, None, cnt, chunk, ws)
    torch.cuda.synchronize(dev)
    status = cc.cc_get_status()
    if status != cc.CC_OK or cache["seq_len"].cpu().tolist() != list(wl.seq_lens):
        raise SystemExit(f"causal pass did not fill the cache: {cc.cc_status_str(status)}")
    del ws
    return cache


def bench_inputs(args, wl, dev):
    """Weights and pristine cache of a workload: the cache from the causal pass
    (default) or drawn directly (--synthetic-cache), then the requested layout
    variants."""
    fast = wl.mode == "layer"
    if args.synthetic_cache or args.kv_fp8 or args.paged or args.head_major:
        return make_inputs(wl, dev, args.kv_fp8, args.paged, args.head_major), "synthetic draws"
    w = synth.model_weights(wl.shape, wl.seed, device=dev, with_kv_proj=True, with_embed=True)
    cache = causal_pass_cache(wl, w, dev)
    if wl.cycles > 1:   # the refresh cycles append through every layer
        return (w, cache), "causal pass of the random model over seeded uniform token ids (cc_append_chunk)"
    if fast:   # the fast pass reads only the last layer's weights
        w["layers"] = [None] * (wl.shape.n_layers - 1) + [w["layers"][-1]]
        w["embed"] = None
    for lw in w["layers"]:
        if lw is not None:
            for key in ("wk", "wv", "bk", "bv"):
                lw.pop(key, None)
    torch.cuda.empty_cache()
    return (w, cache), "causal pass of the random model over seeded uniform token ids (cc_append_chunk)"


def refresh_record(args, dist, wl, w, pristine, mode, steps, with_e2e=True, with_cpu=True):
    """Times one refresh of `wl` (score + select + compaction of every layer)
    over `steps` steps: device-resident inputs with CUDA events on the
    launching stream; the same steps again with events around every library
    launch (per-kernel table, roofline); with_e2e, the same step through the
    public API with its inputs from pinned host memory; with_cpu, the oracle
    on the host cores."""
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    dev = torch.device(f"cuda:{dist.local}")
    shape = wl.shape
    fast = wl.mode == "layer"
    work = clone_cache(pristine)
    f16 = bool(mode & cc.SCORE_F16)
    # fp16 operand mode: the layer matrices converted once (model preparation,
    # outside the timed steps)
    weights, cache = pkg.Weights(cc.f16_weights(w) if f16 else w), pkg.Cache(work)
    b, cap = wl.batch, wl.cap
    scores = torch.empty(b, cap, dtype=torch.float32, device=dev)
    keep_idx = torch.empty(b, cap, dtype=torch.int32, device=dev)
    keep_count = torch.empty(b, dtype=torch.int32, device=dev)
    budget = torch.tensor(wl.budgets, dtype=torch.int32, device=dev)
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode), dev)
    cws = cc.alloc_workspace(cc.cc_compact_workspace_size(shape, cache), dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    score_fn = cc.cc_score_layer if fast else cc.cc_score_full
    stream = torch.cuda.current_stream(dev)
    scorer, recent = args.scorer, args.recent
    row_shard = None
    if args.shard == "rows" and scorer == "counter-causal":
        # this rank's rows of one refresh, then the MAX all-reduce of the scores
        from paper_2607_27600_gb300 import shard as shard_mod
        row_shard = shard_mod.RowShard(shape, not fast, wl.seq_lens, dist.rank, dist.world,
                                       device=dev)
    if scorer in ("importance", "h2o"):
        kws = cc.alloc_workspace(cc.cc_keyattn_workspace_size(shape, b, cap), dev)
    if scorer == "h2o":   # running totals, compacted with the cache
        work["h2o_acc"] = torch.zeros(b, cap, dtype=torch.float32, device=dev)
        cache = pkg.Cache(work)
        cws = cc.alloc_workspace(cc.cc_compact_workspace_size(shape, cache), dev)

    def score():
        if row_shard is not None:
            row_shard.score(shape, weights, cache, mode, scores, ws)
            shard_mod.merge_scores(scores)
        elif scorer == "counter-causal":
            score_fn(shape, weights, cache, mode, scores, ws)
        elif scorer == "recency":
            cc.cc_score_recency(cache, scores)
        elif scorer == "importance":
            cc.cc_score_importance(shape, cache, scores, kws)
        else:
            cc.cc_h2o_accumulate(shape, cache, recent, kws)
            cc.cc_score_h2o(cache, recent, scores)

    def select_compact():
        cc.cc_select_keep(scores, cache.d["seq_len"], b, cap, budget, wl.n_sink, keep_idx,
                          keep_count)
        cc.cc_compact_kv(shape, cache, keep_idx, keep_count, cws)

    def step():
        score()
        select_compact()

    def prepare():
        restore_cache(work, pristine)
        flush.fill_(1)

    for _ in range(args.warmup):
        prepare()
        step()
    torch.cuda.synchronize(dev)
    status = cc.cc_get_status()
    if status != cc.CC_OK:
        raise SystemExit(f"{wl.name}: device status after warm-up: {cc.cc_status_str(status)}")

    clocks = ClockSampler(dist.local)
    clocks.start()
    time.sleep(0.3)
    # (a third event between the scoring and select: the scoring pass's own time)
    ev = [tuple(torch.cuda.Event(enable_timing=True) for _ in range(3)) for _ in range(steps)]
    dist.barrier()
    torch.cuda.synchronize(dev)
    for i in range(steps):
        prepare()
        ev[i][0].record(stream)
        score()
        ev[i][2].record(stream)
        select_compact()
        ev[i][1].record(stream)
    torch.cuda.synchronize(dev)
    dist.barrier()
    step_ms = [a.elapsed_time(bb) for a, bb, _ in ev]
    score_ms = dist.max(sum(a.elapsed_time(c) for a, _, c in ev) / steps)
    ref_idx, ref_cnt = keep_idx.cpu(), keep_count.cpu()   # the last timed step's keep-set
    # per-kernel table: the same steps again with CUDA events around every
    # library launch (kept out of the timed steps above, whose launches they
    # would slow down)
    cc.cc_timing_enable(True)
    for i in range(steps):
        prepare()
        step()
    torch.cuda.synchronize(dev)
    kernels = cc.cc_timing_collect()
    cc.cc_timing_enable(False)
    ms = dist.max(sum(step_ms) / steps)
    status = cc.cc_get_status()
    if status != cc.CC_OK:
        raise SystemExit(f"{wl.name}: device status after timing: {cc.cc_status_str(status)}")
    positions = sum(wl.seq_lens)

    e2e = None
    if with_e2e:
        blocks = None
        # the fast pass's rows scored block by block as their inputs land: one
        # block per ~16k rows, at most 8 (ragged 32k batch, 81920 rows: 2.03 M
        # positions/s end to end in one block, 2.34 M in 4, 2.31 M in 8, 2.14 M
        # in 16; the 8k sequence: 2.75 M in one block, 2.29 M in 8)
        nb = (args.e2e_blocks if args.e2e_blocks > 0 else
              max(1, min(8, sum(wl.seq_lens) // 16384)))
        if fast and scorer == "counter-causal" and row_shard is None and nb > 1:
            blocks = {"n": nb, "select_compact": select_compact,
                      "score": lambda lo, hi: cc.cc_score_rows(
                          shape, weights, cache, mode | cc.SCORE_RANGE_ONLY, False, lo, hi,
                          scores, ws)}
        e2e = e2e_leg(args, dist, wl, work, pristine, cache, step, keep_idx, keep_count, flush,
                      stream, steps, blocks)
        if not (torch.equal(e2e.pop("keep_idx"), ref_idx) and
                torch.equal(e2e.pop("keep_count"), ref_cnt)):
            raise SystemExit(f"{wl.name}: the end-to-end keep-set differs from the "
                             "device-resident step's")
    clk = clocks.stop()

    peaks, peak_src = load_peaks()
    work_tbl = algorithmic_work(wl, 1 if args.kv_fp8 else 2)
    if scorer in ("importance", "h2o"):
        work_tbl["keyattn"] = keyattn_work(wl, scorer, recent)
    timed_s = ms * steps * 1e-3
    table = kernel_table(kernels, steps, work_tbl, peaks, timed_s)
    dom = max(kernels.items(), key=lambda kv: kv[1][1])[0]
    precise = bool(mode & cc.SCORE_PRECISE)
    traffic = None if precise else read_traffic(dom, wl.name, "f16" if f16 else "bf16")
    roof = roofline_of(table, dom, peaks, peak_src, timed_s, traffic)
    # replicas: every rank refreshes its own copy (weak scaling); row shards:
    # the ranks share one refresh (strong scaling)
    value = positions * (1 if row_shard is not None else dist.world) / (ms * 1e-3)
    rec = {
        "workload": wl.name, "value": round(value, 1), "unit": "positions/s",
        "ms_per_step": round(ms, 4), "steps": steps,
        # the metric's other form: positions per second of the scoring pass alone
        "score_only": {"value": round(positions * (1 if row_shard is not None else dist.world) /
                                      (score_ms * 1e-3), 1),
                       "unit": "positions/s", "ms": round(score_ms, 4)},
        "mode": ("precise: [hi | lo] bf16 pairs for activations, queries and P" if precise else
                 "fp16 operands (layer weights converted once; K/V copied per layer), fp32 "
                 "accumulation" if f16 else "bf16 operands, fp32 accumulation"),
        "pass": ("fast single-layer" if fast else f"full {shape.n_layers}-layer")
        if scorer == "counter-causal" else
        {"recency": "position", "importance": "last-layer key attention",
         "h2o": f"all-layer key attention, {recent} recent proxy queries"}[scorer],
        "tflops_per_step_achieved": (round(step_flops(wl) / (ms * 1e-3) / 1e12, 1)
                                     if scorer == "counter-causal" else None),
        "step_tflop": round(step_flops(wl) / 1e12, 3) if scorer == "counter-causal" else None,
        "gpu_launches": int(sum(c for c, _ in kernels.values())),
        "dtype": "f16" if f16 else "bf16",
        "roofline": roof, "kernels": table, "clocks": clk,
    }
    if row_shard is not None:
        rec["shard"] = {"rows_this_rank": row_shard.rows(), "ranks": dist.world,
                        "plan": "cc_partition_rows: contiguous blocks of equal estimated cost"}
    if precise:
        rec["roofline"]["note"] = ("algorithmic FLOPs of the pass; the precise mode issues each "
                                   "product once per operand half (about twice these FLOPs)")
    if f16 and rec["roofline"].get("bound") == "tensor":
        rec["roofline"]["peak_source"] += ("; fp16 operands: the nominal dense fp16 rate equals "
                                           "the bf16 one, so the measured bf16 peak applies")
    if e2e is not None:
        rec["e2e"] = {"value": round(positions * (1 if row_shard is not None else dist.world) /
                                     (e2e["ms"] * 1e-3), 1),
                      "unit": "positions/s", "h2d_bytes_per_step": e2e["h2d"],
                      "d2h_bytes_per_step": e2e["d2h"], "ms_per_step": round(e2e["ms"], 4)}
        if e2e["blocks"] > 1:
            rec["e2e"]["pipeline"] = (f"{e2e['blocks']} row blocks per sequence, uploaded from the "
                                      "sequence ends backwards, each scored once it has landed")
    if (with_cpu and dist.world == 1 and not args.no_cpu_baseline and
            scorer == "counter-causal"):
        rec["cpu_baseline"] = OracleLeg(wl, w, pristine, args.score).cpu_baseline(
            scores.cpu().numpy())
    return rec


def roofline_of(table, dom, peaks, peak_src, timed_s, traffic):
    d = table[dom]
    if d.get("bound") == "tensor":
        peak, which = tensor_peak(peaks, timed_s)
    else:
        peak, which = peaks["hbm_gbs"], "HBM copy"
    return {"kernel": dom, "bound": d.get("bound"), "achieved": d.get("achieved"), "peak": peak,
            "unit": d.get("unit"), "frac": d.get("frac"), "frac_of_burst": d.get("frac_of_burst"),
            "traffic": traffic,
            "peak_source": f"{peak_src} ({which}; the sustained figure when the timed region "
                           f"lasts {SUSTAINED_AFTER_S:.0f} s or more, here {timed_s:.1f} s)"}


def block_bounds(seq_lens, n_blocks, align=128):
    """Starts of `n_blocks` row blocks of every sequence, [n_blocks + 1][batch]:
    block k of sequence b is slots [bounds[k][b], bounds[k + 1][b]), about
    n / n_blocks rows each; every interior start a multiple of `align` (128:
    no key tile of a block's attention reaches below the block, so a block
    scored before the earlier slots have landed never reads them)."""
    out = []
    for k in range(n_blocks + 1):
        out.append([n if k == n_blocks else min(n, -(-(n * k // n_blocks) // align) * align)
                    for n in seq_lens])
    return out


def e2e_leg(args, dist, wl, work, pristine, cache, step, keep_idx, keep_count, flush, stream,
            steps, blocks=None):
    """The refresh through the public API with the step's inputs in pinned
    host memory: token ids, positions and lengths on the compute stream; the
    scored rows' inputs (H^(L-1) in the fast pass, every scored layer's K/V)
    on a copy stream, only each sequence's slots [0, n); the keep-set read
    back.  Copies and reads are inside the timed region.
    Full pass: the library waits per layer for that layer's K/V
    (cc_kv_cache.kv_ready), so the uploads overlap the layers ahead of it.
    Fast pass with `blocks` (n, score(lo, hi), select_compact): the rows are
    uploaded in blocks from the sequence ends backwards and each block is
    scored (cc_score_rows, CC_SCORE_RANGE_ONLY) once it has landed -- a row
    attends only later slots, which arrived before it -- so the uploads
    overlap the scoring; select and compaction follow.
    Before every step the uploaded device tensors are overwritten with NaN
    (outside the timed region): a block scored before its inputs landed
    would change the keep-set, which the caller compares with the
    device-resident step's."""
    dev = torch.device(f"cuda:{dist.local}")
    fast = wl.mode == "layer"
    b, cap = wl.batch, wl.cap
    seq = list(wl.seq_lens)
    n_l = len(work["k"])
    kv_layers = [n_l - 1] if fast else list(range(n_l))
    host = {"h_last": pristine["h_last"].cpu().pin_memory() if fast else None,
            "tokens": pristine["tokens"].cpu().pin_memory(),
            "pos": pristine["pos"].cpu().pin_memory(),
            "seq_len": pristine["seq_len"].cpu().pin_memory(),
            "k": {l: pristine["k"][l].cpu().pin_memory() for l in kv_layers},
            "v": {l: pristine["v"][l].cpu().pin_memory() for l in kv_layers}}
    for t in ([host["h_last"]] if fast else []) + list(host["k"].values()):
        assert t.dim() >= 3 and t.shape[:2] == (b, cap), t.shape   # [batch, cap, ...]
    nb = blocks["n"] if blocks else 1
    bounds = block_bounds(seq, nb)
    lo_host = torch.tensor(bounds[:-1], dtype=torch.int32).pin_memory()   # [nb][batch]
    hi_host = torch.tensor(bounds[1:], dtype=torch.int32).pin_memory()
    lo_dev = torch.empty_like(lo_host, device=dev)
    hi_dev = torch.empty_like(hi_host, device=dev)
    out_idx = torch.empty(b, cap, dtype=torch.int32).pin_memory()
    out_cnt = torch.empty(b, dtype=torch.int32).pin_memory()

    def row_bytes(t):   # bytes of one slot of a [batch, cap, ...] tensor
        return t[0, 0].numel() * t.element_size()

    n_valid = sum(seq)
    h2d = sum(host[key].numel() * host[key].element_size() for key in ("tokens", "pos", "seq_len"))
    if fast:
        h2d += n_valid * row_bytes(host["h_last"])
    h2d += sum(n_valid * row_bytes(t) for key in ("k", "v") for t in host[key].values())
    if blocks:
        h2d += 2 * lo_host.numel() * 4
    d2h = out_idx.numel() * 4 + out_cnt.numel() * 4
    up = torch.cuda.Stream(dev)
    ready = [torch.cuda.Event() if l in kv_layers else None for l in range(n_l)]
    for e in ready:
        if e is not None:
            e.record(up)
    landed = [torch.cuda.Event() for _ in range(nb)]

    def upload_rows(k):
        """Block k's rows of the uploaded tensors (on the copy stream)."""
        for bi, n in enumerate(seq):
            lo, hi = bounds[k][bi], bounds[k + 1][bi]
            if hi <= lo:
                continue
            if fast:
                work["h_last"][bi, lo:hi].copy_(host["h_last"][bi, lo:hi], non_blocking=True)
            for l in kv_layers:
                work["k"][l][bi, lo:hi].copy_(host["k"][l][bi, lo:hi], non_blocking=True)
                work["v"][l][bi, lo:hi].copy_(host["v"][l][bi, lo:hi], non_blocking=True)

    def e2e_step():
        work["seq_len"].copy_(host["seq_len"], non_blocking=True)
        work["tokens"].copy_(host["tokens"], non_blocking=True)
        work["pos"].copy_(host["pos"], non_blocking=True)
        up.wait_stream(stream)
        if blocks:
            lo_dev.copy_(lo_host, non_blocking=True)
            hi_dev.copy_(hi_host, non_blocking=True)
            with torch.cuda.stream(up):
                for k in reversed(range(nb)):   # the sequence ends first
                    upload_rows(k)
                    landed[k].record(up)
            for k in reversed(range(nb)):
                stream.wait_event(landed[k])
                blocks["score"](lo_dev[k], hi_dev[k])
            blocks["select_compact"]()
        else:
            with torch.cuda.stream(up):
                if fast:
                    upload_rows(0)
                for l in kv_layers:
                    if not fast:
                        for bi, n in enumerate(seq):
                            work["k"][l][bi, :n].copy_(host["k"][l][bi, :n], non_blocking=True)
                            work["v"][l][bi, :n].copy_(host["v"][l][bi, :n], non_blocking=True)
                    ready[l].record(up)
            if fast:
                stream.wait_stream(up)
            step()
        out_idx.copy_(keep_idx, non_blocking=True)
        out_cnt.copy_(keep_count, non_blocking=True)

    def poison(t):   # NaN in bf16 / fp32 tensors, the e4m3 NaN code in byte tensors
        if t.dtype.is_floating_point:
            t.fill_(float("nan"))
        else:
            t.fill_(0x7F)

    cache.set_kv_ready(None if (fast or blocks) else ready)
    e2e_ms = []
    try:
        for _ in range(steps):
            restore_cache(work, pristine)   # the rest of the device-resident cache
            if fast:
                poison(work["h_last"])
            for l in kv_layers:
                poison(work["k"][l])
                poison(work["v"][l])
            flush.fill_(1)
            torch.cuda.synchronize(dev)
            t0 = torch.cuda.Event(enable_timing=True)
            t1 = torch.cuda.Event(enable_timing=True)
            t0.record(stream)
            e2e_step()
            t1.record(stream)
            torch.cuda.synchronize(dev)
            e2e_ms.append(t0.elapsed_time(t1))
    finally:
        cache.set_kv_ready(None)
    from paper_2607_27600_gb300 import cc
    status = cc.cc_get_status()
    if status != cc.CC_OK:
        raise SystemExit(f"{wl.name}: device status after e2e: {cc.cc_status_str(status)}")
    return {"ms": dist.max(sum(e2e_ms) / len(e2e_ms)), "h2d": int(h2d), "d2h": int(d2h),
            "blocks": nb, "keep_idx": out_idx.clone(), "keep_count": out_cnt.clone()}


def cycles_record(args, dist, wl, w, pristine, steps):
    """The workload's refresh cycles as configured (Algorithm
    CacheManagedInference, chunked): one step = the refresh of the whole
    cache, then for each later cycle the inference cycle's append of
    `wl.append` new tokens through every layer (cc_append_chunk, seeded token
    ids, positions continuing) and the next refresh.  Appends and refreshes
    are timed separately with CUDA events; positions/s per refresh cycle."""
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    dev = torch.device(f"cuda:{dist.local}")
    shape = wl.shape
    full_w = w
    work = clone_cache(pristine)
    weights, cache = pkg.Weights(full_w), pkg.Cache(work)
    b, cap = wl.batch, wl.cap
    mode = cc.SCORE_LOGIT
    scores = torch.empty(b, cap, dtype=torch.float32, device=dev)
    keep_idx = torch.empty(b, cap, dtype=torch.int32, device=dev)
    keep_count = torch.empty(b, dtype=torch.int32, device=dev)
    budget = torch.tensor(wl.budgets, dtype=torch.int32, device=dev)
    ws = cc.alloc_workspace(cc.cc_score_workspace_size(shape, b, cap, mode), dev)
    cws = cc.alloc_workspace(cc.cc_compact_workspace_size(shape, cache), dev)
    aws = cc.alloc_workspace(cc.cc_append_workspace_size(shape, b, cap), dev)
    chunks = [synth.tokens((b, wl.append), shape.vocab, wl.seed, f"bench.cycle{c}", dev)
              for c in range(1, wl.cycles)]
    count = torch.full((b,), wl.append, dtype=torch.int32, device=dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def refresh():
        cc.cc_score_layer(shape, weights, cache, mode, scores, ws)
        cc.cc_select_keep(scores, cache.d["seq_len"], b, cap, budget, wl.n_sink, keep_idx,
                          keep_count)
        cc.cc_compact_kv(shape, cache, keep_idx, keep_count, cws)

    def one_step(evs=None):
        for c in range(wl.cycles):
            if c > 0:
                if evs is not None:
                    evs[c]["append"][0].record(stream)
                cc.cc_append_chunk(shape, weights, cache, chunks[c - 1], None, count, wl.append,
                                   aws)
                if evs is not None:
                    evs[c]["append"][1].record(stream)
            if evs is not None:
                evs[c]["refresh"][0].record(stream)
            refresh()
            if evs is not None:
                evs[c]["refresh"][1].record(stream)

    def prepare():
        restore_cache(work, pristine)
        flush.fill_(1)

    for _ in range(args.warmup):
        prepare()
        one_step()
    torch.cuda.synchronize(dev)
    status = cc.cc_get_status()
    if status != cc.CC_OK:
        raise SystemExit(f"{wl.name}: device status after warm-up: {cc.cc_status_str(status)}")
    clocks = ClockSampler(dist.local)
    clocks.start()
    time.sleep(0.3)

    def pair():
        return (torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
    per_step = []
    dist.barrier()
    for _ in range(steps):
        prepare()
        torch.cuda.synchronize(dev)
        evs = [{"append": pair(), "refresh": pair()} for _ in range(wl.cycles)]
        one_step(evs)
        torch.cuda.synchronize(dev)
        per_step.append([{k: v[0].elapsed_time(v[1]) for k, v in e.items()
                          if k == "refresh" or c > 0} for c, e in enumerate(evs)])
    dist.barrier()
    # per-kernel table of the first (full-cache) refresh: separate steps with
    # CUDA events around every library launch
    cc.cc_timing_enable(True)
    for _ in range(steps):
        prepare()
        refresh()
    torch.cuda.synchronize(dev)
    kernels = cc.cc_timing_collect()
    cc.cc_timing_enable(False)
    clk = clocks.stop()
    status = cc.cc_get_status()
    if status != cc.CC_OK:
        raise SystemExit(f"{wl.name}: device status after timing: {cc.cc_status_str(status)}")
    peaks, peak_src = load_peaks()
    timed_s = sum(sum(c.values()) for st in per_step for c in st) * 1e-3
    table = kernel_table(kernels, steps, algorithmic_work(wl), peaks, timed_s)
    dom = max(kernels.items(), key=lambda kv: kv[1][1])[0]
    roof = roofline_of(table, dom, peaks, peak_src, timed_s, None)
    roof["scope"] = "the first refresh (full cache)"
    cycles = []
    n = wl.seq_lens[0]
    for c in range(wl.cycles):
        if c > 0:
            n = wl.budgets[0] + wl.append
        r_ms = dist.max(sum(s[c]["refresh"] for s in per_step) / steps)
        e = {"cycle": c + 1, "scored_positions": n * b, "refresh_ms": round(r_ms, 4),
             "positions_per_s": round(n * b * dist.world / (r_ms * 1e-3), 1)}
        if c > 0:
            a_ms = dist.max(sum(s[c]["append"] for s in per_step) / steps)
            e.update({"append_tokens": wl.append * b, "append_ms": round(a_ms, 4),
                      "append_tokens_per_s": round(wl.append * b * dist.world / (a_ms * 1e-3), 1)})
        cycles.append(e)
    total_pos = sum(e["scored_positions"] for e in cycles)
    total_ms = sum(e["refresh_ms"] for e in cycles)
    return {"workload": wl.name, "value": round(total_pos * dist.world / (total_ms * 1e-3), 1),
            "unit": "positions/s",
            "value_basis": "all cycles' scored positions / the cycles' refresh time "
                           "(appends timed separately)",
            "steps": steps, "pass": "fast single-layer", "cycles": cycles, "clocks": clk,
            "roofline": roof, "kernels_first_refresh": table}


def run_suite(args, dist):
    """The default bench line: the headline workload (the full-model pass over
    all 32 layers of the Llama-3-8B shape, the largest single-GPU workload
    with a full pass, fp16 operands unless --bf16 or --precise) plus, in the
    same line, the same pass in the other two operand modes, the ragged
    32k single-layer batch and the long-context refresh cycles."""
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    pkg.load_library()
    dev = torch.device(f"cuda:{dist.local}")
    torch.cuda.set_device(dev)
    wl = synth.WORKLOADS[args.workload]
    if args.layers:   # profiling: the same per-layer launches on a shallower model
        import dataclasses
        wl = dataclasses.replace(wl, name=f"{wl.name}[{args.layers} layers]",
                                 shape=dataclasses.replace(wl.shape, n_layers=args.layers))
        args.no_records = True
    mode = cc.SCORE_LOGPROB if args.score == "logprob" else cc.SCORE_LOGIT
    if args.precise and args.bf16:
        raise SystemExit("--precise and --bf16 are two modes: pick one")
    # the refresh's operand mode: fp16 (the fastest mode that holds the full
    # pass to the stated tolerance) unless --bf16 or --precise asks otherwise
    if args.precise:
        mode |= cc.SCORE_PRECISE
    elif not args.bf16 and args.scorer == "counter-causal":
        mode |= cc.SCORE_F16
    if wl.cycles > 1 and args.scorer == "counter-causal" and not args.single_cycle:
        (w, pristine), cache_src = bench_inputs(args, wl, dev)
        rec = cycles_record(args, dist, wl, w, pristine, args.steps)
        return suite_line(args, dist, wl, rec, cache_src, records={})
    (w, pristine), cache_src = bench_inputs(args, wl, dev)
    head = refresh_record(args, dist, wl, w, pristine, mode, args.steps)
    records = {}
    if not args.no_records and args.scorer == "counter-causal" and dist.world >= 1:
        sub = min(args.steps, 10)
        # the pass in the other two operand modes
        base = mode & ~(cc.SCORE_PRECISE | cc.SCORE_F16)
        for tag, m in (("bf16", base), ("f16", base | cc.SCORE_F16),
                       ("precise", base | cc.SCORE_PRECISE)):
            if m != mode:
                records[f"{wl.name}/{tag}"] = refresh_record(
                    args, dist, wl, w, pristine, m, sub, with_e2e=False, with_cpu=False)
        if args.workload == synth.HEADLINE:
            del w, pristine
            torch.cuda.empty_cache()
            for name in synth.RECORDS:
                rwl = synth.WORKLOADS[name]
                (rw, rp), _ = bench_inputs(args, rwl, dev)
                if rwl.cycles > 1:
                    records[name] = cycles_record(args, dist, rwl, rw, rp, sub)
                else:
                    records[name] = refresh_record(args, dist, rwl, rw, rp, mode, args.steps)
                del rw, rp
                torch.cuda.empty_cache()
    return suite_line(args, dist, wl, head, cache_src, records)


def suite_line(args, dist, wl, head, cache_src, records):
    shape = wl.shape
    # the paper's own figure for this workload (Table 1, another GPU): context only
    vs_baseline = (round(head["value"] / wl.paper_positions_per_s, 2)
                   if wl.paper_positions_per_s and args.scorer == "counter-causal" else None)
    line = {
        "metric": "scored KV positions/sec per refresh",
        "value": head["value"], "unit": "positions/s", "n_gpus": dist.world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": head.get("ms_per_step"),
        "higher_is_better": True, "scaling": "strong" if args.shard == "rows" else "weak",
        "vs_baseline": vs_baseline, "dtype": head.get("dtype", "bf16"),
        "data": f"synthetic (seeded random-init weights N(0,0.02); cache: {cache_src})",
        "config": {"workload": wl.name, "scorer": args.scorer,
                   "kv_cache": ("e4m3 (per-layer scales)" if args.kv_fp8 else "bf16") +
                               (f", paged ({args.paged}-slot pages)" if args.paged else "") +
                               (", head-major" if args.head_major else ""),
                   "pass": head.get("pass"), "mode": head.get("mode"),
                   "score": args.score, "batch": wl.batch, "seq_lens": wl.seq_lens,
                   "budgets": wl.budgets, "cap": wl.cap, "d_model": shape.d_model,
                   "heads": f"{shape.n_q_heads}/{shape.n_kv_heads}x{shape.head_dim}",
                   "d_ff": shape.d_ff, "vocab": shape.vocab,
                   "layers_compacted": shape.n_layers, "step_tflop": head.get("step_tflop"),
                   "l2": "cache restored + 256 MiB written between steps (outside the timed events)",
                   "parallelism": (f"row shards x{dist.world} (one refresh split by query "
                                   f"rows, MAX all-reduce of the scores)" if args.shard == "rows"
                                   else f"replicas x{dist.world}")},
    }
    for key in ("score_only", "shard", "e2e", "gpu_launches", "roofline", "kernels",
                "tflops_per_step_achieved", "clocks", "cpu_baseline", "cycles", "value_basis"):
        if key in head:
            line[key] = head[key]
    if wl.paper_positions_per_s and args.scorer == "counter-causal":
        line["paper"] = {"value": round(wl.paper_positions_per_s, 1), "unit": "positions/s",
                         "source": "Table 1: n / refresh latency, Qwen2.5-7B, RTX 4090, fp16"}
    if records:
        line["records"] = records
    return line


def read_traffic(kernel, workload, operands="bf16"):
    """DRAM bytes per launch from a committed ncu summary, when it was taken
    in the same operand mode (an entry without "operands" is bf16) on the
    current sources of that kernel; else None."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.json")
    if not os.path.exists(p):
        return None
    try:
        with open(p) as f:
            tbl = json.load(f)
        e = tbl.get(workload, {}).get(kernel)
        if not e or e.get("sources_sha") != kernel_digest(kernel):
            return None
        if e.get("operands", "bf16") != operands:
            return None
        return e.get("bytes_per_launch")
    except Exception:
        return None


# the CUDA sources each kernel kind is built from (its own file, its header,
# the shared PTX wrappers)
KERNEL_SOURCES = {
    "gemm": ["gemm.cu", "gemm.cuh", "cc_common.cuh", "api.cu"],   # api.cu: the tile order
    "attention": ["attn.cu", "attn.cuh", "cc_common.cuh"],
    "compact": ["compact.cu", "compact.cuh", "cc_common.cuh"],
    "select": ["select.cu", "select.cuh", "cc_common.cuh"],
    "rowops": ["rowops.cu", "rowops.cuh", "cc_common.cuh"],
}


def code_tokens(text):
    """C/CUDA source without its comments and with runs of whitespace
    collapsed: what a change must touch to change the compiled code."""
    import re
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_digest(kernel, read=None):
    """Hash of the code (comments and layout ignored) of the sources of one
    kernel kind (e.g. gemm_gateup -> gemm.cu, ...); `read(name)` returns a
    source's text (default: the file under csrc/)."""
    import hashlib
    fam = ("gemm" if kernel.startswith("gemm") else "attention" if kernel.startswith("attention")
           else kernel if kernel in KERNEL_SOURCES else "rowops")
    csrc = os.path.join(ROOT, "paper_2607_27600_gb300", "csrc")
    if read is None:
        def read(name):
            with open(os.path.join(csrc, name), encoding="utf-8") as fh:
                return fh.read()
    h = hashlib.sha256()
    for f in KERNEL_SOURCES[fam]:
        h.update((f + "\n" + code_tokens(read(f))).encode())
    return h.hexdigest()[:16]


# ---------------------------------------------------------------------------
# the oracle on the host cores (CPU baseline / reference arm)
# ---------------------------------------------------------------------------

def host_inputs(wl, w, cache, layers):
    """numpy copies for the oracle (bf16 widened to fp32) of the weights and
    K/V of `layers` (a list of layer indices), and raw 16-bit (or e4m3 byte)
    K/V rows of those layers for the compaction."""
    def f32(t):
        return None if t is None else t.float().cpu().numpy()
    nl = wl.shape.n_layers
    lw = [None] * nl
    for l in layers:
        x = w["layers"][l]
        lw[l] = {k: f32(v) for k, v in x.items() if k not in ("wk", "wv", "bk", "bv")}
    wn = {"embed": f32(w["embed"]), "final_norm": f32(w["final_norm"]),
          "lm_head": f32(w["lm_head"]), "layers": lw}
    sc = cache.get("kv_scale")
    if sc is not None:   # e4m3 cache: the oracle gets the codes' values
        import oracle

        def kvf(key, l):
            return (oracle.e4m3_decode(logical_kv(cache, key, l).cpu().numpy()) *
                    sc[l][0 if key == "k" else 1])
    else:
        def kvf(key, l):
            return f32(logical_kv(cache, key, l))
    kf = [kvf("k", l) if l in layers else None for l in range(nl)]
    vf = [kvf("v", l) if l in layers else None for l in range(nl)]
    cn = {"k": kf, "v": vf, "tokens": cache["tokens"].cpu().numpy(), "pos": cache["pos"].cpu().numpy(),
          "seq_len": cache["seq_len"].cpu().numpy(), "h_last": f32(cache["h_last"])}
    kv_raw = torch.uint8 if sc is not None else torch.int16
    raw = {"k": [logical_kv(cache, "k", l).view(kv_raw).cpu().numpy() for l in layers],
           "v": [logical_kv(cache, "v", l).view(kv_raw).cpu().numpy() for l in layers],
           "h": None if cache["h_last"] is None else cache["h_last"].view(torch.int16).cpu().numpy()}
    return wn, cn, raw


def cores_used():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


class OracleLeg:
    """The oracle, as it stands, timed on the host cores on a bounded sample of
    one refresh of a workload; both the cpu_baseline of our arm and the
    reference arm use it with the same sample sizes.

    A refresh is scoring, select and compaction.  Scoring rows are independent
    given the cache and every layer of a pass repeats the same work, so the
    sample scores `rows` rows drawn uniformly over all positions through
    `layers` layers (all of the fast pass's one layer; the first two of a full
    pass, a truncated model), and the time extrapolates linearly: per-call
    fixed cost (widening each sampled layer's weights) from two sample sizes,
    times L / layers, plus the per-row cost times N.  Select runs in full; the
    compaction moves tokens, positions and H^(L-1) in full and the K/V of the
    sampled layers, extrapolated to all L layers.  Every extrapolated figure is
    labelled as such."""

    def __init__(self, wl, w, cache, score_mode):
        import dataclasses
        self.wl, self.mode = wl, score_mode
        nl = wl.shape.n_layers
        self.fast = wl.mode == "layer"
        self.layers = [nl - 1] if self.fast else list(range(min(2, nl)))
        self.shape = wl.shape if self.fast else dataclasses.replace(wl.shape,
                                                                     n_layers=len(self.layers))
        self.kv_layers = [nl - 1] if self.fast else self.layers
        self.wn, self.cn, self.raw = host_inputs(wl, w, cache, sorted(set(self.layers)))
        # sample sizes large enough that the per-row cost stands out of the
        # per-call fixed cost in the fit
        self.rows_small, self.rows_large = (64, 128) if self.fast else (16, 32)
        self.positions = sum(wl.seq_lens)
        self.fixed = None

    def sample(self, count, seed):
        """`count` rows drawn uniformly over all of the workload's positions."""
        r = np.random.default_rng(seed)
        flat = np.sort(r.choice(self.positions, size=min(count, self.positions), replace=False))
        starts = np.cumsum([0] + list(self.wl.seq_lens))
        return [(flat[(flat >= starts[b]) & (flat < starts[b + 1])] - starts[b]).tolist()
                for b in range(self.wl.batch)]

    def _score(self, rows):
        import oracle
        fn = oracle.score_layer if self.fast else oracle.score_full
        t0 = time.perf_counter()
        fn(self.shape, self.wn, self.cn, mode=self.mode, rows=rows)
        return time.perf_counter() - t0, sum(len(r) for r in rows)

    def fit(self):
        """Per-call fixed cost of the sampled scoring, from two sample sizes
        (after one untimed call that pays the one-time set-up)."""
        self._score(self.sample(self.rows_small, seed=10))
        t1, n1 = self._score(self.sample(self.rows_small, seed=11))
        t2, n2 = self._score(self.sample(self.rows_large, seed=12))
        per_row = max(0.0, (t2 - t1) / max(1, n2 - n1))
        self.fixed = max(0.0, t1 - n1 * per_row)
        return self.fixed

    def step(self, scores_np, seed):
        """One sampled refresh; returns (measured seconds, extrapolated seconds
        of the whole refresh, details)."""
        import oracle
        if self.fixed is None:
            self.fit()
        w0 = time.perf_counter()
        t_rows, n_rows = self._score(self.sample(self.rows_large, seed))
        t1 = time.perf_counter()
        idx, cnt = oracle.select_keep(scores_np, self.cn["seq_len"], self.wl.budgets,
                                      self.wl.n_sink)
        t_sel = time.perf_counter() - t1
        t2 = time.perf_counter()
        for arrs in (self.raw["k"], self.raw["v"]):
            for a in arrs:
                oracle.compact(a, idx, cnt)
        t_kv = time.perf_counter() - t2
        t3 = time.perf_counter()
        if self.raw["h"] is not None:
            oracle.compact(self.raw["h"], idx, cnt)
        oracle.compact(self.cn["tokens"], idx, cnt)
        oracle.compact(self.cn["pos"], idx, cnt)
        t_small = time.perf_counter() - t3
        measured = time.perf_counter() - w0
        nl = self.wl.shape.n_layers
        lf = nl / len(self.layers) if not self.fast else 1.0
        per_row = max(0.0, t_rows - self.fixed) / n_rows
        t_score = lf * (self.fixed + per_row * self.positions)
        t_compact = t_small + t_kv * nl / len(self.kv_layers)
        total = t_score + t_sel + t_compact
        return measured, total, {"rows": n_rows, "t_rows": t_rows, "t_sel": t_sel,
                                 "t_compact": t_compact}

    def describe(self, d):
        lay = ("its one layer" if self.fast else
               f"{len(self.layers)} of {self.wl.shape.n_layers} layers (a truncated model), "
               f"x{self.wl.shape.n_layers // len(self.layers)}")
        return (f"{d['rows']} rows drawn uniformly over {self.positions} positions scored through "
                f"{lay} ({d['t_rows']:.2f} s, per-call fixed cost {self.fixed:.2f} s fitted from "
                f"{self.rows_small} and {self.rows_large} rows), extrapolated linearly to every "
                f"row; full select ({d['t_sel']:.3f} s); compaction of tokens, positions and "
                f"H^(L-1) in full and of {len(self.kv_layers)} layers' K/V, extrapolated to "
                f"{self.wl.shape.n_layers} layers ({d['t_compact']:.2f} s); numpy fp64, BLAS "
                f"threads = cores")

    def cpu_baseline(self, scores_np):
        measured, total, d = self.step(scores_np, seed=0)
        return {"value": round(self.positions / total, 3), "unit": "positions/s",
                "cores": cores_used(), "kind": "oracle", "extrapolated": True,
                "sample_s": round(measured, 2), "sample": self.describe(d)}


def run_reference(args, dist):
    """The reference arm: the oracle (CPU) timed on a bounded sample of the
    same workload per step (OracleLeg), rank 0 only."""
    if dist.rank != 0:
        return None
    wl = synth.WORKLOADS[args.workload]
    dev = torch.device("cuda:0") if torch.cuda.is_available() else torch.device("cpu")
    if dev.type == "cuda":
        torch.cuda.set_device(dev)
    # the oracle's inputs come from the seeded generators alone (the cache drawn
    # directly: the oracle's time does not depend on the values); only the
    # layers the sample runs are drawn
    nl = wl.shape.n_layers
    sampled = [nl - 1] if wl.mode == "layer" else list(range(min(2, nl)))
    w = synth.model_weights(wl.shape, wl.seed, device=dev, layers=sampled,
                            with_embed=wl.mode == "full")
    cache = synth.synthetic_cache(wl.shape, wl.seq_lens, wl.cap, wl.seed, device=dev,
                                  layers=sampled, with_h_last=wl.mode == "layer")
    leg = OracleLeg(wl, w, cache, args.score)
    del w, cache
    r = np.random.default_rng(1)
    scores_np = r.standard_normal(size=leg.cn["tokens"].shape).astype(np.float32)
    for b, n in enumerate(wl.seq_lens):
        scores_np[b, n - 1] = np.inf
    leg.fit()
    measured, extrap = [], []
    d = None
    for i in range(args.warmup + args.steps):
        m, total, d = leg.step(scores_np, seed=100 + i)
        if i >= args.warmup:
            measured.append(m)
            extrap.append(total)
    ms = 1e3 * sum(measured) / len(measured)
    ex_ms = 1e3 * sum(extrap) / len(extrap)
    positions = leg.positions
    value = positions / (ex_ms * 1e-3)
    return {"impl": "reference", "metric": "scored KV positions/sec per refresh",
            "value": round(value, 3), "unit": "positions/s", "n_gpus": dist.world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 2),
            "ms_per_step_is": "measured wall time of one sampled step",
            "extrapolated_ms_per_refresh": round(ex_ms, 1),
            "value_basis": "positions / the extrapolated time of one whole refresh",
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": wl.name, "score": args.score},
            "cpu_baseline": {"value": round(value, 3), "unit": "positions/s", "cores": cores_used(),
                             "kind": "oracle", "extrapolated": True,
                             "sample_s": round(ms / 1e3, 2), "sample": leg.describe(d)},
            "e2e": {"value": round(value, 3), "unit": "positions/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}


# ---------------------------------------------------------------------------
# the inference cycle (pre-fill chunk append), --append
# ---------------------------------------------------------------------------

def append_work(shape, j, h):
    """Per-launch algorithmic FLOPs / bytes of the append of h tokens after j memory slots."""
    d, qd, kvd, f, hq, dh = (shape.d_model, shape.q_dim, shape.kv_dim, shape.d_ff,
                             shape.n_q_heads, shape.head_dim)
    keys = h * j + h * (h + 1) // 2            # sum over chunk rows of the keys they attend
    return {"gemm_qrope": ("tensor", 2.0 * h * d * qd),
            "gemm_kv": ("tensor", 2.0 * h * d * kvd),
            "gemm_qkv": ("tensor", 2.0 * h * d * (qd + 2 * kvd)),
            "attention_causal": ("tensor", 4.0 * dh * hq * keys),
            "gemm_oproj": ("tensor", 2.0 * h * qd * d),
            "gemm_gateup": ("tensor", 4.0 * h * d * f),
            "gemm_down": ("tensor", 2.0 * h * f * d),
            "rmsnorm": ("hbm", h * (4.0 * d * 2 + 2.0 * d))}


# A step timed for longer than this runs under the power cap like the
# measured sustained GEMM loop: its tensor fractions take the sustained peak.
SUSTAINED_AFTER_S = 1.0


def tensor_peak(peaks, timed_s):
    """(peak TFLOP/s, which) for a kernel timed inside a region of timed_s seconds."""
    if timed_s >= SUSTAINED_AFTER_S and "bf16_tflops_sustained" in peaks:
        return peaks["bf16_tflops_sustained"], "bf16 dense sustained"
    return peaks["bf16_tflops"], "bf16 dense burst"


def kernel_table(kernels, steps, work_tbl, peaks, timed_s=0.0):
    table = {}
    total = max(1e-9, sum(t for _, t in kernels.values()))
    tpk, _ = tensor_peak(peaks, timed_s)
    for name, (cnt, tot) in kernels.items():
        per = tot / cnt
        entry = {"launches_per_step": cnt / steps, "ms_per_launch": round(per, 4),
                 "share": round(tot / total, 4)}
        if name in work_tbl:
            bound, amount = work_tbl[name]
            if bound == "tensor":
                ach = amount / (per * 1e-3) / 1e12
                entry.update({"bound": "tensor", "achieved": round(ach, 2), "unit": "TFLOP/s",
                              "frac": round(ach / tpk, 4),
                              "frac_of_burst": round(ach / peaks["bf16_tflops"], 4)})
            else:
                ach = amount / (per * 1e-3) / 1e9
                entry.update({"bound": "hbm", "achieved": round(ach, 1), "unit": "GB/s",
                              "frac": round(ach / peaks["hbm_gbs"], 4)})
        table[name] = entry
    return table


def run_append(args, dist):
    """Times cc_append_chunk: the workload's `append` tokens after a memory of
    `budgets[0]` slots (the cache a refresh leaves), through every layer."""
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    pkg.load_library()
    dev = torch.device(f"cuda:{dist.local}")
    torch.cuda.set_device(dev)
    wl = synth.WORKLOADS[args.workload]
    shape = wl.shape
    j, h = wl.budgets[0], wl.append
    if h <= 0:
        raise SystemExit(f"{wl.name} has no append chunk")
    cap = j + h
    w = synth.model_weights(shape, wl.seed, device=dev, with_kv_proj=True)
    cache = synth.synthetic_cache(shape, [j], cap, wl.seed, device=dev)
    if args.kv_fp8:
        to_e4m3_cache(cache)
    chunk = synth.tokens((1, h), shape.vocab, wl.seed, "bench.chunk", dev)
    count = torch.tensor([h], dtype=torch.int32, device=dev)
    weights, kc = pkg.Weights(w), pkg.Cache(cache)
    ws = cc.alloc_workspace(cc.cc_append_workspace_size(shape, 1, cap), dev)
    flush = torch.empty(L2_FLUSH_BYTES, dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream(dev)

    def prepare():
        cache["seq_len"].fill_(j)
        flush.fill_(1)

    for _ in range(args.warmup):
        prepare()
        cc.cc_append_chunk(shape, weights, kc, chunk, None, count, h, ws)
    torch.cuda.synchronize(dev)
    if cc.cc_get_status() != cc.CC_OK:
        raise SystemExit("device status after warm-up")
    clocks = ClockSampler(dist.local)
    clocks.start()
    time.sleep(0.3)
    dist.barrier()
    torch.cuda.synchronize(dev)
    ms_steps = []
    for _ in range(args.steps):
        prepare()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        cc.cc_append_chunk(shape, weights, kc, chunk, None, count, h, ws)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        ms_steps.append(e0.elapsed_time(e1))
    dist.barrier()
    cc.cc_timing_enable(True)   # per-kernel table from separate steps
    for _ in range(args.steps):
        prepare()
        cc.cc_append_chunk(shape, weights, kc, chunk, None, count, h, ws)
    torch.cuda.synchronize(dev)
    kernels = cc.cc_timing_collect()
    cc.cc_timing_enable(False)
    ms = dist.max(sum(ms_steps) / len(ms_steps))
    # end to end: the chunk's token ids and count from pinned host memory, the
    # new length read back
    host_tok = chunk.cpu().pin_memory()
    host_cnt = count.cpu().pin_memory()
    out_len = torch.empty(1, dtype=torch.int32).pin_memory()
    e2e = []
    for _ in range(args.steps):
        prepare()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        tok_d = host_tok.to(dev, non_blocking=True)
        cnt_d = host_cnt.to(dev, non_blocking=True)
        cc.cc_append_chunk(shape, weights, kc, tok_d, None, cnt_d, h, ws)
        out_len.copy_(cache["seq_len"], non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        e2e.append(e0.elapsed_time(e1))
    clk = clocks.stop()
    if cc.cc_get_status() != cc.CC_OK or int(out_len[0]) != j + h:
        raise SystemExit("append did not complete")
    e2e_ms = dist.max(sum(e2e) / len(e2e))
    peaks, peak_src = load_peaks()
    work = append_work(shape, j, h)
    table = kernel_table(kernels, args.steps, work, peaks)
    dom = max(kernels.items(), key=lambda kv: kv[1][1])[0]
    d = table[dom]
    flops = sum(work[k][1] * table[k]["launches_per_step"] for k in work
                if work[k][0] == "tensor" and k in table)
    line = {
        "metric": "appended tokens/sec per inference cycle (pre-fill chunk, all layers)",
        "value": round(h * dist.world / (ms * 1e-3), 1), "unit": "tokens/s",
        "n_gpus": dist.world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(ms, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded random-init weights N(0,0.02); synthetic memory K/V)",
        "config": {"workload": wl.name + "/append", "memory_slots": j, "chunk": h,
                   "kv_cache": "e4m3 (per-layer scales)" if args.kv_fp8 else "bf16",
                   "layers": shape.n_layers, "d_model": shape.d_model,
                   "heads": f"{shape.n_q_heads}/{shape.n_kv_heads}x{shape.head_dim}",
                   "d_ff": shape.d_ff, "step_tflop": round(flops / 1e12, 3),
                   "l2": "256 MiB written between steps (outside the timed events)",
                   "parallelism": f"replicas x{dist.world}"},
        "e2e": {"value": round(h * dist.world / (e2e_ms * 1e-3), 1), "unit": "tokens/s",
                "h2d_bytes_per_step": int(host_tok.numel() * 4 + 4), "d2h_bytes_per_step": 4,
                "ms_per_step": round(e2e_ms, 4)},
        "gpu_launches": int(sum(c for c, _ in kernels.values())),
        "dtype": "f16" if f16 else "bf16",
        "roofline": {"kernel": dom, "bound": d.get("bound"), "achieved": d.get("achieved"),
                     "peak": peaks["bf16_tflops"] if d.get("bound") == "tensor" else peaks["hbm_gbs"],
                     "unit": d.get("unit"), "frac": d.get("frac"), "traffic": None,
                     "peak_source": f"{peak_src} (bf16 dense burst)"},
        "kernels": table,
        "tflops_per_step_achieved": round(flops / (ms * 1e-3) / 1e12, 1),
        "clocks": clk,
    }
    if dist.world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = append_cpu_baseline(shape, w, cache, chunk, j, h)
    return line


def run_decode(args, dist):
    """Times greedy decode steps (cc_decode_step) of one sequence after a
    memory of `budgets[0]` slots: each step appends the current token through
    every layer and picks the next one from the LM head.  The steps are
    replayed from captured graphs (cc_graph_*: one launch per step, the
    launch-bound path a serving loop uses); eager calls are timed beside."""
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    pkg.load_library()
    dev = torch.device(f"cuda:{dist.local}")
    torch.cuda.set_device(dev)
    wl = synth.WORKLOADS[args.workload]
    shape = wl.shape
    j = wl.budgets[0]
    # warm-up, graph-timed, eager-timed, kernel-table and end-to-end steps
    cap = j + args.warmup + 4 * args.steps + 16
    w = synth.model_weights(shape, wl.seed, device=dev, with_kv_proj=True)
    B = args.batch   # sequences decoded together (each with its own memory of j slots)
    cache = synth.synthetic_cache(shape, [j] * B, cap, wl.seed, device=dev)
    if args.kv_fp8:
        to_e4m3_cache(cache)
    weights, kc = pkg.Weights(w), pkg.Cache(cache)
    ws = cc.alloc_workspace(cc.cc_decode_workspace_size(shape, B, cap), dev)
    tok = [torch.ones(B, dtype=torch.int32, device=dev),
           torch.empty(B, dtype=torch.int32, device=dev)]
    stream = torch.cuda.Stream(dev)   # captured work needs a stream other than the legacy default
    graphs = []
    with torch.cuda.stream(stream):
        for i in range(args.warmup):
            cc.cc_decode_step(shape, weights, kc, tok[i % 2], tok[1 - i % 2], None, ws)
        if args.warmup % 2:
            tok[0].copy_(tok[1])
        torch.cuda.synchronize(dev)
        if cc.cc_get_status() != cc.CC_OK:
            raise SystemExit("device status after warm-up")
        for a in (0, 1):   # step a: tokens tok[a] -> next tokens tok[1 - a]
            cc.cc_graph_begin()
            cc.cc_decode_step(shape, weights, kc, tok[a], tok[1 - a], None, ws)
            graphs.append(cc.cc_graph_end())
        clocks = ClockSampler(dist.local)
        clocks.start()
        time.sleep(0.3)
        dist.barrier()
        torch.cuda.synchronize(dev)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(args.steps):
            cc.cc_graph_launch(graphs[i % 2])
        e1.record(stream)
        torch.cuda.synchronize(dev)
        dist.barrier()
        ms = dist.max(e0.elapsed_time(e1) / args.steps)
        if args.steps % 2:
            tok[0].copy_(tok[1])
        e0.record(stream)
        for i in range(args.steps):
            cc.cc_decode_step(shape, weights, kc, tok[i % 2], tok[1 - i % 2], None, ws)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        eager_ms = dist.max(e0.elapsed_time(e1) / args.steps)
        if args.steps % 2:
            tok[0].copy_(tok[1])
        cc.cc_timing_enable(True)   # per-kernel table from separate (eager) steps
        for i in range(args.steps):
            cc.cc_decode_step(shape, weights, kc, tok[i % 2], tok[1 - i % 2], None, ws)
        torch.cuda.synchronize(dev)
        kernels = cc.cc_timing_collect()
        cc.cc_timing_enable(False)
        # end to end: the current token from pinned host memory, the next one
        # read back, the step replayed from its graph
        host_tok = torch.ones(B, dtype=torch.int32).pin_memory()
        host_out = torch.empty(B, dtype=torch.int32).pin_memory()
        e0.record(stream)
        for _ in range(args.steps // 2):
            tok[0].copy_(host_tok, non_blocking=True)
            cc.cc_graph_launch(graphs[0])
            host_out.copy_(tok[1], non_blocking=True)
        e1.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms = dist.max(e0.elapsed_time(e1) / max(1, args.steps // 2))
        clk = clocks.stop()
        for g in graphs:
            cc.cc_graph_destroy(g)
        if cc.cc_get_status() != cc.CC_OK or int(host_out.min()) < 0:
            raise SystemExit("decode did not complete")
    peaks, peak_src = load_peaks()
    d, qd, kvd, f = shape.d_model, shape.q_dim, shape.kv_dim, shape.d_ff
    n_mid = j + args.warmup + 2 * args.steps + args.steps // 2   # slots at a kernel-table step
    work = {"gemm_qkv": ("hbm", 2.0 * d * (qd + 2 * kvd)), "gemm_oproj": ("hbm", 2.0 * qd * d),
            "gemm_gateup": ("hbm", 4.0 * d * f), "gemm_down": ("hbm", 2.0 * f * d),
            "gemm_lmhead": ("hbm", 2.0 * shape.vocab * d),
            "attention_causal": ("hbm", 2.0 * (1 if args.kv_fp8 else 2) * kvd * n_mid * B)}
    table = kernel_table(kernels, args.steps, work, peaks)
    dom = max(kernels.items(), key=lambda kv: kv[1][1])[0]
    dd = table[dom]
    return {
        "metric": ("decoded tokens/sec per sequence (greedy, all layers + LM head)" if B == 1 else
                   f"decoded tokens/sec, {B} sequences per step (greedy, all layers + LM head)"),
        "value": round(dist.world * B / (ms * 1e-3), 1), "unit": "tokens/s", "n_gpus": dist.world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded random-init weights N(0,0.02); synthetic memory K/V)",
        "config": {"workload": wl.name + "/decode", "memory_slots": j, "batch": B,
                   "kv_cache": "e4m3 (per-layer scales)" if args.kv_fp8 else "bf16",
                   "layers": shape.n_layers, "d_model": shape.d_model, "vocab": shape.vocab,
                   "l2": "weights (15 GB) far exceed L2: every step streams them from HBM",
                   "launch": "one captured graph per step (cc_graph_launch)",
                   "eager_ms_per_step": round(eager_ms, 4),
                   "parallelism": f"replicas x{dist.world}"},
        "e2e": {"value": round(dist.world * B / (e2e_ms * 1e-3), 1), "unit": "tokens/s",
                "h2d_bytes_per_step": 4 * B, "d2h_bytes_per_step": 4 * B,
                "ms_per_step": round(e2e_ms, 4)},
        "gpu_launches": int(sum(c for c, _ in kernels.values())),
        "dtype": "f16" if f16 else "bf16",
        "roofline": {"kernel": dom, "bound": dd.get("bound"), "achieved": dd.get("achieved"),
                     "peak": peaks["hbm_gbs"], "unit": dd.get("unit"), "frac": dd.get("frac"),
                     "traffic": None, "peak_source": f"{peak_src} (HBM copy)"},
        "kernels": table,
        "clocks": clk,
    }


def append_cpu_baseline(shape, w, cache, chunk, j, h, sample=8):
    """The oracle's append timed on the host cores for `sample` chunk tokens
    through one layer, extrapolated linearly to the chunk and every layer (a
    row's GEMM work and its attention over ~j memory keys dominate)."""
    import oracle
    one = shape.__class__(**{**shape.__dict__, "n_layers": 1})
    lw = {k: v.float().cpu().numpy() for k, v in w["layers"][0].items()}
    wn = {"embed": w["embed"].float().cpu().numpy(), "layers": [lw]}
    cn = {"k": [cache["k"][0].float().cpu().numpy().astype(np.float64)],
          "v": [cache["v"][0].float().cpu().numpy().astype(np.float64)],
          "tokens": cache["tokens"].cpu().numpy(), "pos": cache["pos"].cpu().numpy(),
          "seq_len": np.array([j]), "h_last": None}
    toks = chunk.cpu().numpy()[0, :sample]
    t0 = time.perf_counter()
    oracle.append_chunk(one, wn, cn, 0, toks)
    dt = time.perf_counter() - t0
    per_token_layer = dt / sample
    total = per_token_layer * h * shape.n_layers
    return {"value": round(h / total, 2), "unit": "tokens/s", "cores": os.cpu_count(),
            "kind": "oracle",
            "sample": f"{sample} chunk tokens through 1 layer ({dt:.1f} s), extrapolated linearly "
                      f"to {h} tokens x {shape.n_layers} layers; numpy fp64"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default=synth.HEADLINE, choices=sorted(synth.WORKLOADS))
    ap.add_argument("--score", choices=["logit", "logprob"], default="logit")
    ap.add_argument("--single-cycle", action="store_true",
                    help="time only the first refresh of a multi-cycle workload")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--precise", action="store_true",
                    help="time the precise mode (CC_SCORE_PRECISE) as the headline")
    ap.add_argument("--bf16", action="store_true",
                    help="time the bf16 operand mode (the library's default) as the headline "
                         "instead of the fp16 one (CC_SCORE_F16)")
    ap.add_argument("--e2e-blocks", type=int, default=0,
                    help="fast pass end to end: row blocks uploaded and scored in turn (1: the "
                         "whole input first; 0: one block per 16k rows, at most 8)")
    ap.add_argument("--no-records", action="store_true",
                    help="only the named workload (no precise-mode and other-workload records)")
    ap.add_argument("--synthetic-cache", action="store_true",
                    help="draw the cache directly instead of building it by a causal pass")
    ap.add_argument("--shard", choices=["replicas", "rows"], default="replicas",
                    help="N > 1: every rank refreshes its own replica (default), or the ranks "
                         "split one refresh by query rows (cc_score_rows + a MAX all-reduce)")
    ap.add_argument("--layers", type=int, default=0,
                    help="profiling only: truncate the model to this many layers (every "
                         "launch keeps its full-size shape; the line is not a headline)")
    ap.add_argument("--kv-fp8", action="store_true",
                    help="store the cache's K/V as e4m3 codes with per-layer scales")
    ap.add_argument("--batch", type=int, default=1,
                    help="--decode: sequences decoded together (1-4 take the GEMV path)")
    ap.add_argument("--head-major", action="store_true",
                    help="keep the refresh bench's K/V head-major ([B, Hkv, cap, dh])")
    ap.add_argument("--paged", type=int, default=0, metavar="SLOTS",
                    help="keep the refresh bench's K/V in page pools of SLOTS-slot pages "
                         "(a multiple of 128) in a shuffled order, with a block table")
    ap.add_argument("--scorer", choices=["counter-causal", "recency", "importance", "h2o"],
                    default="counter-causal",
                    help="refresh scorer: the paper's (default) or one of its comparison "
                         "scorers (Sec. 4) on the same select/compact path")
    ap.add_argument("--recent", type=int, default=256,
                    help="h2o: proxy-query slots (the most recent) per refresh")
    ap.add_argument("--decode", action="store_true",
                    help="time greedy decode steps of one sequence over the workload's "
                         "budget-sized memory (cc_decode_step)")
    ap.add_argument("--append", action="store_true",
                    help="time the inference cycle: the workload's append chunk over its "
                         "budget-sized memory (cc_append_chunk, every layer)")
    args = ap.parse_args()
    if args.warmup < 3:
        raise SystemExit("--warmup must be >= 3")
    dist = Dist()
    try:
        if args.impl == "reference":
            line = run_reference(args, dist)
        elif args.append:
            line = run_append(args, dist)
        elif args.decode:
            line = run_decode(args, dist)
        else:
            line = run_suite(args, dist)
        if dist.rank == 0 and line is not None:
            print(json.dumps(line), flush=True)
    finally:
        dist.close()


if __name__ == "__main__":
    main()
