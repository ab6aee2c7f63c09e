"""Benchmark of one counter-causal memory refresh (arXiv 2607.27600,
Sec. 3.1 and Algorithm DoMemRefresh) on GB300.

A step = one refresh of one synthetic cache: counter-causal scores of every
cached position (fast single-layer approximation, or the full L-layer pass),
keep-set selection at the budget, in-place compaction of every layer's K/V,
H^(L-1), tokens and positions.  Metric: scored KV positions per second.

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

def run_ours(args, dist):
    import paper_2607_27600_gb300 as pkg
    from paper_2607_27600_gb300 import cc
    pkg.load_library()
    dev = torch.device(f"cuda:{dist.local}")
    torch.cuda.set_device(dev)
    wl = synth.WORKLOADS[args.workload]
    shape = wl.shape
    mode = cc.SCORE_LOGPROB if args.score == "logprob" else cc.SCORE_LOGIT
    fast = wl.mode == "layer"
    if wl.cycles > 1 and not args.single_cycle:
        raise SystemExit("multi-cycle workloads: use --single-cycle (the first refresh is timed)")

    w, pristine = make_inputs(wl, dev, args.kv_fp8, args.paged, args.head_major)
    work = clone_cache(pristine)
    weights, cache = pkg.Weights(w), pkg.Cache(work)
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
    if scorer in ("importance", "h2o"):
        kws = cc.alloc_workspace(cc.cc_keyattn_workspace_size(shape, b, cap), dev)
    if scorer == "h2o":   # running totals, compacted with the cache
        work["h2o_acc"] = torch.zeros(b, cap, dtype=torch.float32, device=dev)
        cache = pkg.Cache(work)
        cws = cc.alloc_workspace(cc.cc_compact_workspace_size(shape, cache), dev)

    def score():
        if scorer == "counter-causal":
            score_fn(shape, weights, cache, mode, scores, ws)
        elif scorer == "recency":
            cc.cc_score_recency(cache, scores)
        elif scorer == "importance":
            cc.cc_score_importance(shape, cache, scores, kws)
        else:
            cc.cc_h2o_accumulate(shape, cache, recent, kws)
            cc.cc_score_h2o(cache, recent, scores)

    def step():
        score()
        cc.cc_select_keep(scores, cache.d["seq_len"], b, cap, budget, wl.n_sink, keep_idx,
                          keep_count)
        cc.cc_compact_kv(shape, cache, keep_idx, keep_count, cws)

    def prepare():
        restore_cache(work, pristine)
        flush.fill_(1)

    for _ in range(args.warmup):
        prepare()
        step()
    torch.cuda.synchronize(dev)
    status = cc.cc_get_status()
    if status != cc.CC_OK:
        raise SystemExit(f"device status after warm-up: {cc.cc_status_str(status)}")

    clocks = ClockSampler(dist.local)
    clocks.start()
    time.sleep(0.3)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(args.steps)]
    dist.barrier()
    torch.cuda.synchronize(dev)
    for i in range(args.steps):
        prepare()
        ev[i][0].record(stream)
        step()
        ev[i][1].record(stream)
    torch.cuda.synchronize(dev)
    dist.barrier()
    step_ms = [a.elapsed_time(bb) for a, bb in ev]
    # per-kernel table: the same steps again with CUDA events around every
    # library launch (kept out of the timed steps above, whose launches they
    # would slow down)
    cc.cc_timing_enable(True)
    for i in range(args.steps):
        prepare()
        step()
    torch.cuda.synchronize(dev)
    kernels = cc.cc_timing_collect()
    cc.cc_timing_enable(False)
    ms_local = sum(step_ms) / args.steps
    ms = dist.max(ms_local)
    status = cc.cc_get_status()
    if status != cc.CC_OK:
        raise SystemExit(f"device status after timing: {cc.cc_status_str(status)}")

    # ---- end to end through the public API with host inputs
    host = {"h_last": pristine["h_last"].cpu().pin_memory() if fast else None,
            "k": pristine["k"][-1].cpu().pin_memory(), "v": pristine["v"][-1].cpu().pin_memory(),
            "tokens": pristine["tokens"].cpu().pin_memory(),
            "pos": pristine["pos"].cpu().pin_memory(),
            "seq_len": pristine["seq_len"].cpu().pin_memory()}
    if not fast:   # the full pass reads every layer's K/V
        host["k_all"] = [x.cpu().pin_memory() for x in pristine["k"]]
        host["v_all"] = [x.cpu().pin_memory() for x in pristine["v"]]
    out_idx = torch.empty(b, cap, dtype=torch.int32).pin_memory()
    out_cnt = torch.empty(b, dtype=torch.int32).pin_memory()
    h2d = sum(t.numel() * t.element_size() for k, t in host.items()
              if isinstance(t, torch.Tensor))
    if not fast:
        h2d += sum(t.numel() * t.element_size() for t in host["k_all"] + host["v_all"])
        h2d -= host["k"].numel() * host["k"].element_size() * 2
    d2h = out_idx.numel() * 4 + out_cnt.numel() * 4

    # K/V uploads run on a copy stream and the library waits for each layer's
    # event right before the layer's first K/V reader (cc_kv_cache.kv_ready),
    # so they overlap the kernels ahead of it; the host link is one queue, so
    # they start once the inputs of the first kernels have landed
    up = torch.cuda.Stream(dev)
    n_l = len(work["k"])
    kv_layers = [n_l - 1] if fast else list(range(n_l))
    ready = [torch.cuda.Event() if l in kv_layers else None for l in range(n_l)]
    for e in ready:
        if e is not None:
            e.record(up)

    def e2e_step():
        work["seq_len"].copy_(host["seq_len"], non_blocking=True)
        work["tokens"].copy_(host["tokens"], non_blocking=True)
        work["pos"].copy_(host["pos"], non_blocking=True)
        if fast:
            work["h_last"].copy_(host["h_last"], non_blocking=True)
        up.wait_stream(stream)
        with torch.cuda.stream(up):
            for l in kv_layers:
                work["k"][l].copy_(host["k"] if fast else host["k_all"][l], non_blocking=True)
                work["v"][l].copy_(host["v"] if fast else host["v_all"][l], non_blocking=True)
                ready[l].record(up)
        step()
        out_idx.copy_(keep_idx, non_blocking=True)
        out_cnt.copy_(keep_count, non_blocking=True)

    cache.set_kv_ready(ready)

    e2e_ms = []
    for i in range(args.steps):
        restore_cache(work, pristine)   # the rest of the device-resident cache
        flush.fill_(1)
        torch.cuda.synchronize(dev)
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(stream)
        e2e_step()
        t1.record(stream)
        torch.cuda.synchronize(dev)
        e2e_ms.append(t0.elapsed_time(t1))
    cache.set_kv_ready(None)
    clk = clocks.stop()
    e2e_ms_max = dist.max(sum(e2e_ms) / len(e2e_ms))
    status = cc.cc_get_status()
    if status != cc.CC_OK:
        raise SystemExit(f"device status after e2e: {cc.cc_status_str(status)}")
    # sanity: the e2e keep-set equals the device-resident one of the last timed step
    positions = sum(wl.seq_lens)

    # ---- roofline of the dominant kernel (and a per-kernel table)
    peaks, peak_src = load_peaks()
    work_tbl = algorithmic_work(wl, 1 if args.kv_fp8 else 2)
    if scorer in ("importance", "h2o"):
        work_tbl["keyattn"] = keyattn_work(wl, scorer, recent)
    table = {}
    for name, (cnt, tot) in kernels.items():
        per = tot / cnt
        entry = {"launches_per_step": cnt / args.steps, "ms_per_launch": round(per, 4),
                 "share": round(tot / max(1e-9, sum(t for _, t in kernels.values())), 4)}
        if name in work_tbl:
            bound, amount = work_tbl[name]
            if bound == "tensor":
                ach = amount / (per * 1e-3) / 1e12
                entry.update({"bound": "tensor", "achieved": round(ach, 2), "unit": "TFLOP/s",
                              "frac": round(ach / peaks["bf16_tflops"], 4)})
            else:
                ach = amount / (per * 1e-3) / 1e9
                entry.update({"bound": "hbm", "achieved": round(ach, 1), "unit": "GB/s",
                              "frac": round(ach / peaks["hbm_gbs"], 4)})
        table[name] = entry
    dom = max(kernels.items(), key=lambda kv: kv[1][1])[0]
    traffic = read_traffic(dom, wl.name)
    d = table[dom]
    roof = {"kernel": dom, "bound": d.get("bound"), "achieved": d.get("achieved"),
            "peak": peaks["bf16_tflops"] if d.get("bound") == "tensor" else peaks["hbm_gbs"],
            "unit": d.get("unit"), "frac": d.get("frac"), "traffic": traffic,
            "peak_source": f"{peak_src} ({'bf16 dense burst' if d.get('bound') == 'tensor' else 'HBM copy'})"}

    launches = sum(c for c, _ in kernels.values())
    value = positions * dist.world / (ms * 1e-3)
    # the paper's own figure for this workload (Table 1, another GPU): context only
    vs_baseline = (round(value / wl.paper_positions_per_s, 2)
                   if wl.paper_positions_per_s and scorer == "counter-causal" else None)
    line = {
        "metric": "scored KV positions/sec per refresh",
        "value": round(value, 1), "unit": "positions/s", "n_gpus": dist.world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 4),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": vs_baseline, "dtype": "bf16",
        "data": "synthetic (seeded random-init weights N(0,0.02); synthetic KV cache)",
        "config": {"workload": wl.name, "scorer": scorer,
                   "kv_cache": ("e4m3 (per-layer scales)" if args.kv_fp8 else "bf16") +
                               (f", paged ({args.paged}-slot pages)" if args.paged else "") +
                               (", head-major" if args.head_major else ""),
                   "pass": ("fast single-layer" if fast else f"full {shape.n_layers}-layer")
                   if scorer == "counter-causal" else
                   {"recency": "position", "importance": "last-layer key attention",
                    "h2o": f"all-layer key attention, {recent} recent proxy queries"}[scorer],
                   "score": args.score, "batch": wl.batch, "seq_lens": wl.seq_lens,
                   "budgets": wl.budgets, "cap": wl.cap, "d_model": shape.d_model,
                   "heads": f"{shape.n_q_heads}/{shape.n_kv_heads}x{shape.head_dim}",
                   "d_ff": shape.d_ff, "vocab": shape.vocab,
                   "layers_compacted": shape.n_layers,
                   "step_tflop": (round(step_flops(wl) / 1e12, 3) if scorer == "counter-causal"
                                  else None),
                   "l2": "cache restored + 256 MiB written between steps (outside the timed events)",
                   "parallelism": f"replicas x{dist.world}"},
        "e2e": {"value": round(positions * dist.world / (e2e_ms_max * 1e-3), 1),
                "unit": "positions/s", "h2d_bytes_per_step": int(h2d),
                "d2h_bytes_per_step": int(d2h), "ms_per_step": round(e2e_ms_max, 4)},
        "gpu_launches": int(launches),
        "roofline": roof,
        "kernels": table,
        # the counter-causal pass's algorithmic FLOPs (the comparison scorers' are
        # in their keyattn entry)
        "tflops_per_step_achieved": (round(step_flops(wl) / (ms * 1e-3) / 1e12, 1)
                                     if scorer == "counter-causal" else None),
        "clocks": clk,
    }
    if wl.paper_positions_per_s and scorer == "counter-causal":
        line["paper"] = {"value": round(wl.paper_positions_per_s, 1), "unit": "positions/s",
                         "source": "Table 1: n / refresh latency, Qwen2.5-7B, RTX 4090, fp16"}
    if dist.world == 1 and not args.no_cpu_baseline and scorer == "counter-causal":
        line["cpu_baseline"] = cpu_baseline(wl, w, pristine, scores, args.cpu_rows, args.score)
    return line


def read_traffic(kernel, workload):
    """DRAM bytes per launch from a committed ncu summary, when it matches the
    current kernel sources; else None."""
    p = os.path.join(ROOT, "profiles", "dram_traffic.json")
    if not os.path.exists(p):
        return None
    try:
        with open(p) as f:
            tbl = json.load(f)
        e = tbl.get(workload, {}).get(kernel)
        if not e or e.get("csrc_sha") != csrc_digest():
            return None
        return e.get("bytes_per_launch")
    except Exception:
        return None


def csrc_digest():
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2607_27600_gb300", "csrc")
    for f in sorted(os.listdir(csrc)):
        with open(os.path.join(csrc, f), "rb") as fh:
            h.update(f.encode() + fh.read())
    return h.hexdigest()[:16]


# ---------------------------------------------------------------------------
# the oracle on the host cores (CPU baseline / reference arm)
# ---------------------------------------------------------------------------

def host_inputs(wl, w, cache):
    """numpy copies (bf16 widened to fp32; K/V of the compacted layers kept as raw 16-bit)."""
    def f32(t):
        return None if t is None else t.float().cpu().numpy()
    last = wl.shape.n_layers - 1
    fast = wl.mode == "layer"
    lw = [None] * wl.shape.n_layers
    for l, x in enumerate(w["layers"]):
        if x is not None:
            lw[l] = {k: f32(v) for k, v in x.items()}
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
    kf = [kvf("k", l) if (not fast or l == last) else None for l in range(wl.shape.n_layers)]
    vf = [kvf("v", l) if (not fast or l == last) else None for l in range(wl.shape.n_layers)]
    cn = {"k": kf, "v": vf, "tokens": cache["tokens"].cpu().numpy(), "pos": cache["pos"].cpu().numpy(),
          "seq_len": cache["seq_len"].cpu().numpy(), "h_last": f32(cache["h_last"])}
    kv_raw = torch.uint8 if sc is not None else torch.int16
    raw = {"k": [logical_kv(cache, "k", l).view(kv_raw).cpu().numpy()
                 for l in range(len(cache["k"]))],
           "v": [logical_kv(cache, "v", l).view(kv_raw).cpu().numpy()
                 for l in range(len(cache["v"]))],
           "h": None if cache["h_last"] is None else cache["h_last"].view(torch.int16).cpu().numpy()}
    return wn, cn, raw


def sample_rows(wl, count, seed=0):
    r = np.random.default_rng(seed)
    rows = []
    per = max(2, count // wl.batch)
    for n in wl.seq_lens:
        pick = {0, n - 2, n - 1} | set(r.choice(n, size=min(n, per), replace=False).tolist())
        rows.append(sorted(x for x in pick if 0 <= x < n)[:max(per, 3)])
    return rows


def _oracle_score_time(wl, wn, cn, rows, score_mode):
    import oracle
    fn = oracle.score_layer if wl.mode == "layer" else oracle.score_full
    t0 = time.perf_counter()
    fn(wl.shape, wn, cn, mode=score_mode, rows=rows)
    return time.perf_counter() - t0, sum(len(r) for r in rows)


def oracle_fixed_cost(wl, wn, cn, score_mode, small, large):
    """Per-call cost of the oracle's scoring that does not grow with the rows
    (widening the weights to fp64), from two sample sizes."""
    t1, n1 = _oracle_score_time(wl, wn, cn, sample_rows(wl, small, seed=11), score_mode)
    t2, n2 = _oracle_score_time(wl, wn, cn, sample_rows(wl, large, seed=12), score_mode)
    per_row = max(0.0, (t2 - t1) / max(1, n2 - n1))
    return max(0.0, t1 - n1 * per_row)


def oracle_refresh_time(wl, wn, cn, raw, scores_np, rows, score_mode, fixed):
    """Seconds the oracle takes for one refresh of the whole workload: its
    scoring timed on the sampled rows and extrapolated linearly in the row
    count (rows are independent given the cache; the per-call fixed cost is
    counted once), plus its select and compaction run in full."""
    import oracle
    t_rows, n_sampled = _oracle_score_time(wl, wn, cn, rows, score_mode)
    per_row = max(0.0, t_rows - fixed) / n_sampled
    t1 = time.perf_counter()
    idx, cnt = oracle.select_keep(scores_np, cn["seq_len"], wl.budgets, wl.n_sink)
    t_sel = time.perf_counter() - t1
    t2 = time.perf_counter()
    for arrs in (raw["k"], raw["v"]):
        for a in arrs:
            oracle.compact(a, idx, cnt)
    if raw["h"] is not None:
        oracle.compact(raw["h"], idx, cnt)
    oracle.compact(cn["tokens"], idx, cnt)
    oracle.compact(cn["pos"], idx, cnt)
    t_cmp = time.perf_counter() - t2
    positions = sum(wl.seq_lens)
    total = fixed + per_row * positions + t_sel + t_cmp
    return total, n_sampled, t_rows, t_sel, t_cmp


def cores_used():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


def cpu_baseline(wl, w, cache, scores_dev, n_rows, score_mode):
    wn, cn, raw = host_inputs(wl, w, cache)
    scores_np = scores_dev.cpu().numpy()
    fixed = oracle_fixed_cost(wl, wn, cn, score_mode, n_rows // 4, n_rows // 2)
    rows = sample_rows(wl, n_rows)
    total, ns, t_rows, t_sel, t_cmp = oracle_refresh_time(wl, wn, cn, raw, scores_np, rows,
                                                          score_mode, fixed)
    return {"value": round(sum(wl.seq_lens) / total, 3), "unit": "positions/s",
            "cores": cores_used(), "kind": "oracle",
            "sample": (f"{ns} sampled rows scored ({t_rows:.1f} s incl. {fixed:.1f} s per-call "
                       f"fixed cost), extrapolated linearly to {sum(wl.seq_lens)} rows, + full "
                       f"select ({t_sel:.2f} s) + full compaction ({t_cmp:.2f} s); numpy fp64, "
                       f"BLAS threads = cores")}


def run_reference(args, dist):
    if dist.rank != 0:
        return None
    wl = synth.WORKLOADS[args.workload]
    dev = torch.device("cuda:0") if torch.cuda.is_available() else torch.device("cpu")
    w, cache = make_inputs(wl, dev)
    wn, cn, raw = host_inputs(wl, w, cache)
    r = np.random.default_rng(1)
    scores_np = r.standard_normal(size=cn["tokens"].shape).astype(np.float32)
    for b, n in enumerate(wl.seq_lens):
        scores_np[b, n - 1] = np.inf
    times = []
    ns = 0
    fixed = oracle_fixed_cost(wl, wn, cn, args.score, max(2, args.ref_rows // 2),
                              args.ref_rows * 3 // 2)
    for i in range(args.warmup + args.steps):
        rows = sample_rows(wl, args.ref_rows, seed=i)
        total, ns, *_ = oracle_refresh_time(wl, wn, cn, raw, scores_np, rows, args.score, fixed)
        if i >= args.warmup:
            times.append(total)
    ms = 1e3 * sum(times) / len(times)
    positions = sum(wl.seq_lens)
    value = positions / (ms * 1e-3)
    sample = (f"per step {ns} sampled rows scored by the oracle, extrapolated linearly to "
              f"{positions} rows (per-call fixed cost {fixed:.1f} s counted once), + full "
              f"select and compaction")
    return {"impl": "reference", "metric": "scored KV positions/sec per refresh",
            "value": round(value, 3), "unit": "positions/s", "n_gpus": dist.world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms, 2),
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": {"workload": wl.name, "score": args.score},
            "cpu_baseline": {"value": round(value, 3), "unit": "positions/s", "cores": cores_used(),
                             "kind": "oracle", "sample": sample},
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


def kernel_table(kernels, steps, work_tbl, peaks):
    table = {}
    total = max(1e-9, sum(t for _, t in kernels.values()))
    for name, (cnt, tot) in kernels.items():
        per = tot / cnt
        entry = {"launches_per_step": cnt / steps, "ms_per_launch": round(per, 4),
                 "share": round(tot / total, 4)}
        if name in work_tbl:
            bound, amount = work_tbl[name]
            if bound == "tensor":
                ach = amount / (per * 1e-3) / 1e12
                entry.update({"bound": "tensor", "achieved": round(ach, 2), "unit": "TFLOP/s",
                              "frac": round(ach / peaks["bf16_tflops"], 4)})
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
    ap.add_argument("--cpu-rows", type=int, default=256)
    ap.add_argument("--ref-rows", type=int, default=32)
    ap.add_argument("--no-cpu-baseline", action="store_true")
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
            line = run_ours(args, dist)
        if dist.rank == 0 and line is not None:
            print(json.dumps(line), flush=True)
    finally:
        dist.close()


if __name__ == "__main__":
    main()
