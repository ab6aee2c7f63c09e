"""Python binding of the counter-causal refresh C ABI (include/cc.h,
include/cc_kernels.h).

Argument marshalling only: every function here passes device pointers of
torch CUDA tensors and the current CUDA stream to the library, whose CUDA
kernels do all the work.  A non-OK status raises CCError.  There is no
fallback: if libcc.so is missing, every call raises.
"""
import ctypes
import os

import torch

from . import build as _build

CC_OK = 0
CC_ERR_INVALID_ARG = 1
CC_ERR_CUDA = 2
CC_ERR_BUDGET = 3
CC_ERR_WORKSPACE = 4
CC_ERR_TIMEOUT = 5
CC_ERR_UNSUPPORTED = 6
CC_ERR_DEVICE_ARG = 7
CC_ERR_RANGE = 8
STATUS_NAMES = {0: "CC_OK", 1: "CC_ERR_INVALID_ARG", 2: "CC_ERR_CUDA", 3: "CC_ERR_BUDGET",
                4: "CC_ERR_WORKSPACE", 5: "CC_ERR_TIMEOUT", 6: "CC_ERR_UNSUPPORTED",
                7: "CC_ERR_DEVICE_ARG", 8: "CC_ERR_RANGE"}
SCORE_LOGIT = 0
SCORE_LOGPROB = 1
SCORE_PRECISE = 0x100   # flag: hi + lo bf16 GEMM activations, queries and P (either pass)
SCORE_RANGE_ONLY = 0x200   # flag (cc_score_rows): entries outside the row range keep their values
SCORE_F16 = 0x400   # flag: fp16 tensor-core operands (the layer weights passed as fp16)


class CCError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = code
        extra = f" [{cc_last_error()}]" if code == CC_ERR_CUDA else ""
        super().__init__(f"{where}: {STATUS_NAMES.get(code, code)} ({cc_status_str(code)}){extra}")


class cc_model_cfg(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("d_model", ctypes.c_int32),
                ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
                ("head_dim", ctypes.c_int32), ("d_ff", ctypes.c_int32), ("vocab", ctypes.c_int32),
                ("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float),
                ("rope_scaling_factor", ctypes.c_float), ("rope_low_freq_factor", ctypes.c_float),
                ("rope_high_freq_factor", ctypes.c_float), ("rope_original_max_pos", ctypes.c_int32)]


class cc_layer_weights(ctypes.Structure):
    _fields_ = [(n, ctypes.c_void_p) for n in
                ("attn_norm", "wq", "wo", "mlp_norm", "w_gate", "w_up", "w_down", "bq",
                 "wk", "wv", "bk", "bv")]


class cc_model_weights(ctypes.Structure):
    _fields_ = [("embed", ctypes.c_void_p), ("final_norm", ctypes.c_void_p),
                ("lm_head", ctypes.c_void_p), ("layers", ctypes.POINTER(cc_layer_weights))]


class cc_kv_cache(ctypes.Structure):
    _fields_ = [("batch", ctypes.c_int32), ("cap", ctypes.c_int32),
                ("seq_len", ctypes.c_void_p), ("k", ctypes.POINTER(ctypes.c_void_p)),
                ("v", ctypes.POINTER(ctypes.c_void_p)), ("tokens", ctypes.c_void_p),
                ("pos", ctypes.c_void_p), ("h_last", ctypes.c_void_p),
                ("h2o_acc", ctypes.c_void_p), ("kv_format", ctypes.c_int32),
                ("kv_scale", ctypes.POINTER(ctypes.c_float)),
                ("block_table", ctypes.c_void_p), ("page_size", ctypes.c_int32),
                ("n_pages", ctypes.c_int32), ("kv_layout", ctypes.c_int32),
                ("kv_ready", ctypes.POINTER(ctypes.c_void_p))]

KV_BF16, KV_E4M3 = 0, 1
KV_SLOT_MAJOR, KV_HEAD_MAJOR = 0, 1


_LIB = None
_SIGS = {
    "cc_score_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(cc_model_cfg), ctypes.c_int32,
                                                  ctypes.c_int32, ctypes.c_int]),
    "cc_score_layer": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.POINTER(cc_model_weights),
                                      ctypes.POINTER(cc_kv_cache), ctypes.c_int, ctypes.c_void_p,
                                      ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]),
    "cc_score_full": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.POINTER(cc_model_weights),
                                     ctypes.POINTER(cc_kv_cache), ctypes.c_int, ctypes.c_void_p,
                                     ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]),
    "cc_score_rows": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.POINTER(cc_model_weights),
                                     ctypes.POINTER(cc_kv_cache), ctypes.c_int, ctypes.c_int32,
                                     ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                     ctypes.c_void_p, ctypes.c_size_t, ctypes.c_void_p]),
    "cc_partition_rows": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.c_int32,
                                         ctypes.POINTER(ctypes.c_int32), ctypes.c_int32,
                                         ctypes.c_int32, ctypes.c_int32,
                                         ctypes.POINTER(ctypes.c_int32),
                                         ctypes.POINTER(ctypes.c_int32)]),
    "cc_append_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(cc_model_cfg), ctypes.c_int32,
                                                   ctypes.c_int32]),
    "cc_append_chunk": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.POINTER(cc_model_weights),
                                       ctypes.POINTER(cc_kv_cache), ctypes.c_void_p, ctypes.c_void_p,
                                       ctypes.c_void_p, ctypes.c_int32, ctypes.c_void_p,
                                       ctypes.c_size_t, ctypes.c_void_p]),
    "cc_score_recency": (ctypes.c_int, [ctypes.POINTER(cc_kv_cache), ctypes.c_void_p,
                                        ctypes.c_void_p]),
    "cc_keyattn_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(cc_model_cfg), ctypes.c_int32,
                                                    ctypes.c_int32]),
    "cc_score_importance": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.POINTER(cc_kv_cache),
                                           ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t,
                                           ctypes.c_void_p]),
    "cc_h2o_accumulate": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.POINTER(cc_kv_cache),
                                         ctypes.c_int32, ctypes.c_void_p, ctypes.c_size_t,
                                         ctypes.c_void_p]),
    "cc_score_h2o": (ctypes.c_int, [ctypes.POINTER(cc_kv_cache), ctypes.c_int32, ctypes.c_void_p,
                                    ctypes.c_void_p]),
    "cc_decode_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(cc_model_cfg), ctypes.c_int32,
                                                   ctypes.c_int32]),
    "cc_decode_step": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.POINTER(cc_model_weights),
                                      ctypes.POINTER(cc_kv_cache), ctypes.c_void_p, ctypes.c_void_p,
                                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t,
                                      ctypes.c_void_p]),
    "cc_select_workspace_size": (ctypes.c_size_t, [ctypes.c_int32, ctypes.c_int32]),
    "cc_select_keep": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_int32,
                                      ctypes.c_int32, ctypes.c_void_p, ctypes.c_int32,
                                      ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                      ctypes.c_size_t, ctypes.c_void_p]),
    "cc_compact_workspace_size": (ctypes.c_size_t, [ctypes.POINTER(cc_model_cfg),
                                                    ctypes.POINTER(cc_kv_cache)]),
    "cc_compact_kv": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg), ctypes.POINTER(cc_kv_cache),
                                     ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                     ctypes.c_size_t, ctypes.c_void_p]),
    "cc_compact_kv_static": (ctypes.c_int, [ctypes.POINTER(cc_model_cfg),
                                            ctypes.POINTER(cc_kv_cache), ctypes.c_void_p,
                                            ctypes.c_void_p, ctypes.c_void_p]),
    "cc_graph_begin": (ctypes.c_int, [ctypes.c_void_p]),
    "cc_graph_end": (ctypes.c_int, [ctypes.c_void_p, ctypes.POINTER(ctypes.c_void_p)]),
    "cc_graph_launch": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p]),
    "cc_graph_destroy": (ctypes.c_int, [ctypes.c_void_p]),
    "cc_bf16_to_f16": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_size_t,
                                      ctypes.c_void_p]),
    "cc_get_status": (ctypes.c_int, [ctypes.c_void_p]),
    "cc_status_str": (ctypes.c_char_p, [ctypes.c_int]),
    "cc_last_error": (ctypes.c_char_p, []),
    "cc_linear_f32": (ctypes.c_int, [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                     ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                                     ctypes.c_void_p]),
    "cc_counter_causal_attention": (ctypes.c_int, [ctypes.c_void_p] * 5 + [ctypes.c_int32] * 5
                                    + [ctypes.c_void_p]),
    "cc_counter_causal_attention_split": (ctypes.c_int, [ctypes.c_void_p] * 5
                                          + [ctypes.c_int32] * 5 + [ctypes.c_void_p]),
    "cc_timing_enable": (ctypes.c_int, [ctypes.c_int32]),
    "cc_timing_collect": (ctypes.c_int, [ctypes.POINTER(ctypes.c_int32),
                                         ctypes.POINTER(ctypes.c_double)]),
    "cc_kernel_name": (ctypes.c_char_p, [ctypes.c_int32]),
    "cc_debug_withhold_compact_unit": (ctypes.c_int, [ctypes.c_int32]),
}
KERNEL_COUNT = 19


def library_path() -> str:
    return _build.LIB


def load_library(path: str = None) -> ctypes.CDLL:
    """Loads libcc.so (built by paper_2607_27600_gb300.build); raises if absent."""
    global _LIB
    if _LIB is None:
        path = path or library_path()
        if not os.path.exists(path):
            raise ImportError(f"{path} not found: build it first "
                              "(python -m paper_2607_27600_gb300.build)")
        lib = ctypes.CDLL(path)
        for name, (res, args) in _SIGS.items():
            fn = getattr(lib, name)
            fn.restype, fn.argtypes = res, args
        _LIB = lib
    return _LIB


def exported_symbols():
    return sorted(_SIGS)


# ---------------------------------------------------------------------------
# marshalling helpers
# ---------------------------------------------------------------------------

def _dev_ptr(t, name):
    if t is None:
        return None
    if not isinstance(t, torch.Tensor) or not t.is_cuda:
        raise TypeError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _stream(stream):
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _check(code, where):
    if code != CC_OK:
        raise CCError(code, where)


def model_cfg(shape) -> cc_model_cfg:
    """cc_model_cfg from any object with the ModelShape fields (rope_scaling,
    if present and not None: (factor, low_freq_factor, high_freq_factor,
    original_max_position))."""
    sc = getattr(shape, "rope_scaling", None) or (0.0, 0.0, 0.0, 0)
    return cc_model_cfg(shape.n_layers, shape.d_model, shape.n_q_heads, shape.n_kv_heads,
                        shape.head_dim, shape.d_ff, shape.vocab, float(shape.rope_theta),
                        float(shape.rms_eps), float(sc[0]), float(sc[1]), float(sc[2]),
                        int(sc[3]))


class Weights:
    """cc_model_weights over a dict of CUDA bf16 tensors (embed, final_norm,
    lm_head, layers[l] = {attn_norm, wq, wo, mlp_norm, w_gate, w_up, w_down,
    optional bq, and wk, wv, bk, bv for the append}); keeps the tensors alive."""

    def __init__(self, w: dict):
        self.w = w
        layers = w["layers"]
        self._layers = (cc_layer_weights * len(layers))()
        for l, lw in enumerate(layers):
            if lw is None:
                continue
            for f in ("attn_norm", "wq", "wo", "mlp_norm", "w_gate", "w_up", "w_down"):
                setattr(self._layers[l], f, _dev_ptr(lw[f], f"layers[{l}].{f}"))
            for f in ("bq", "wk", "wv", "bk", "bv"):   # optional (wk, wv: append only)
                if lw.get(f) is not None:
                    setattr(self._layers[l], f, _dev_ptr(lw[f], f"layers[{l}].{f}"))
        self.c = cc_model_weights(_dev_ptr(w.get("embed"), "embed"),
                                  _dev_ptr(w["final_norm"], "final_norm"),
                                  _dev_ptr(w["lm_head"], "lm_head"), self._layers)


F16_MATRICES = ("wq", "wo", "w_gate", "w_up", "w_down")   # what SCORE_F16 reads as fp16


def f16_weights(w: dict, stream=None) -> dict:
    """The weights dict of Weights with the layer matrices that SCORE_F16
    reads (F16_MATRICES) converted to fp16 by cc_bf16_to_f16; every other
    entry is shared with `w`."""
    out = dict(w)
    out["layers"] = []
    for lw in w["layers"]:
        if lw is None:
            out["layers"].append(None)
            continue
        nl = dict(lw)
        for f in F16_MATRICES:
            nl[f] = torch.empty(lw[f].shape, dtype=torch.float16, device=lw[f].device)
            cc_bf16_to_f16(lw[f], nl[f], stream)
        out["layers"].append(nl)
    return out


class Cache:
    """cc_kv_cache over a dict of CUDA tensors (k[l], v[l] bf16 [B, cap, Hkv, dh],
    or e4m3 codes (uint8) when the dict holds "kv_scale": per layer the (K, V)
    scales; tokens, pos int32 [B, cap]; seq_len int32 [B]; h_last bf16
    [B, cap, d] or None); with "block_table" (int32 [B, cap // page_size]),
    "page_size" and k[l], v[l] page pools [n_pages, page_size, Hkv, dh] the
    K/V are paged; with "kv_layout": KV_HEAD_MAJOR, k[l], v[l] are
    [B, Hkv, cap, dh].  Keeps the tensors alive.  set_kv_ready() attaches the
    per-layer events of K/V uploads still in flight on another stream."""

    def __init__(self, c: dict):
        self.d = c
        b, cap = c["tokens"].shape
        ks, vs = c["k"], c["v"]
        self._k = (ctypes.c_void_p * len(ks))(*[_dev_ptr(x, "k") for x in ks])
        self._v = (ctypes.c_void_p * len(vs))(*[_dev_ptr(x, "v") for x in vs])
        sc = c.get("kv_scale")
        fmt, self._scale = KV_BF16, None
        if sc is not None:
            flat = [float(x) for pair in sc for x in pair]
            if len(flat) != 2 * len(ks):
                raise ValueError("kv_scale needs one (K, V) pair per layer")
            self._scale = (ctypes.c_float * len(flat))(*flat)
            fmt = KV_E4M3
        table, page, n_pages = c.get("block_table"), 0, 0
        if table is not None:
            page = int(c["page_size"])
            n_pages = int(next(x for x in ks if x is not None).shape[0])
        self.c = cc_kv_cache(b, cap, _dev_ptr(c["seq_len"], "seq_len"), self._k, self._v,
                             _dev_ptr(c["tokens"], "tokens"), _dev_ptr(c["pos"], "pos"),
                             _dev_ptr(c.get("h_last"), "h_last"),
                             _dev_ptr(c.get("h2o_acc"), "h2o_acc"), fmt, self._scale,
                             _dev_ptr(table, "block_table"), page, n_pages,
                             int(c.get("kv_layout", KV_SLOT_MAJOR)), None)
        self._ready = None

    def set_kv_ready(self, events):
        """events: one torch.cuda.Event (already recorded once) or None per
        layer, or None for no waits (cc_kv_cache.kv_ready)."""
        if events is None:
            self._ready = None
            self.c.kv_ready = None
            return
        if len(events) != len(self._k):
            raise ValueError("kv_ready needs one entry per layer")
        handles = []
        for e in events:
            h = 0 if e is None else int(e.cuda_event)
            if e is not None and h == 0:
                raise ValueError("record a kv_ready event once before attaching it")
            handles.append(h or None)
        self._ready = (ctypes.c_void_p * len(handles))(*handles)
        self.c.kv_ready = self._ready


def _cfg(cfg):
    return cfg if isinstance(cfg, cc_model_cfg) else model_cfg(cfg)


# ---------------------------------------------------------------------------
# the C ABI, one Python function per entry point
# ---------------------------------------------------------------------------

def cc_status_str(code: int) -> str:
    return load_library().cc_status_str(int(code)).decode()


def cc_last_error() -> str:
    return load_library().cc_last_error().decode()


def cc_score_workspace_size(cfg, batch: int, cap: int, mode: int = SCORE_LOGIT) -> int:
    return int(load_library().cc_score_workspace_size(ctypes.byref(_cfg(cfg)), batch, cap, mode))


def _check_operand_type(weights, mode):
    """The layer matrices must be fp16 exactly when the mode has SCORE_F16
    (the library reads the same pointers as bf16 otherwise)."""
    want = torch.float16 if int(mode) & SCORE_F16 else torch.bfloat16
    for l, lw in enumerate(weights.w["layers"]):
        if lw is None:
            continue
        for f in F16_MATRICES:
            if lw[f].dtype != want:
                raise ValueError(f"layers[{l}].{f} is {lw[f].dtype}; this mode reads {want} "
                                 "(f16_weights converts the matrices for SCORE_F16)")


def _score(fn, cfg, weights: Weights, cache: Cache, mode, scores, ws, stream):
    _check_operand_type(weights, mode)
    c = _cfg(cfg)
    code = getattr(load_library(), fn)(ctypes.byref(c), ctypes.byref(weights.c),
                                       ctypes.byref(cache.c), int(mode),
                                       _dev_ptr(scores, "scores"), _dev_ptr(ws, "ws"),
                                       ws.numel() * ws.element_size(), _stream(stream))
    _check(code, fn)


def cc_score_layer(cfg, weights, cache, mode, scores, ws, stream=None):
    _score("cc_score_layer", cfg, weights, cache, mode, scores, ws, stream)


def cc_score_full(cfg, weights, cache, mode, scores, ws, stream=None):
    _score("cc_score_full", cfg, weights, cache, mode, scores, ws, stream)


def cc_bf16_to_f16(src, dst, stream=None):
    """dst (fp16) = src (bf16), element by element (same number of elements,
    a multiple of 8): the layer weights of SCORE_F16."""
    if src.dtype != torch.bfloat16 or dst.dtype != torch.float16 or src.numel() != dst.numel():
        raise ValueError("cc_bf16_to_f16: src bf16 and dst fp16 of one size")
    code = load_library().cc_bf16_to_f16(_dev_ptr(src, "src"), _dev_ptr(dst, "dst"), src.numel(),
                                         _stream(stream))
    _check(code, "cc_bf16_to_f16")


def cc_score_rows(cfg, weights, cache, mode, full: bool, row_lo, row_hi, scores, ws, stream=None):
    """Scores only rows [row_lo[b], row_hi[b]) of each sequence (device int32
    [batch] each, or both None for every row); every other entry of `scores`
    gets -inf, or keeps its value with SCORE_RANGE_ONLY in `mode`."""
    _check_operand_type(weights, mode)
    code = load_library().cc_score_rows(
        ctypes.byref(_cfg(cfg)), ctypes.byref(weights.c), ctypes.byref(cache.c), int(mode),
        1 if full else 0, _dev_ptr(row_lo, "row_lo"), _dev_ptr(row_hi, "row_hi"),
        _dev_ptr(scores, "scores"), _dev_ptr(ws, "ws"), ws.numel() * ws.element_size(),
        _stream(stream))
    _check(code, "cc_score_rows")


def cc_partition_rows(cfg, full: bool, seq_lens, world: int, align: int = 128):
    """Host-side plan of a refresh split over `world` ranks: returns
    (row_lo, row_hi), int32 numpy [world][batch]; rank r scores rows
    [row_lo[r][b], row_hi[r][b]) of sequence b.  Needs no GPU."""
    import numpy as np
    sl = np.ascontiguousarray(np.asarray(seq_lens, dtype=np.int32))
    lo = np.zeros((world, sl.size), np.int32)
    hi = np.zeros((world, sl.size), np.int32)
    p32 = ctypes.POINTER(ctypes.c_int32)
    code = load_library().cc_partition_rows(
        ctypes.byref(_cfg(cfg)), 1 if full else 0, sl.ctypes.data_as(p32), int(sl.size),
        int(world), int(align), lo.ctypes.data_as(p32), hi.ctypes.data_as(p32))
    _check(code, "cc_partition_rows")
    return lo, hi


def cc_append_workspace_size(cfg, batch: int, cap: int) -> int:
    return int(load_library().cc_append_workspace_size(ctypes.byref(_cfg(cfg)), batch, cap))


def cc_append_chunk(cfg, weights, cache, tokens_in, pos_in, count, max_count: int, ws,
                    stream=None):
    """Inference cycle in pre-fill: append count[b] tokens (tokens_in [B, max_count]
    int32, positions pos_in or None) to every sequence of `cache`, all layers."""
    c = _cfg(cfg)
    code = load_library().cc_append_chunk(
        ctypes.byref(c), ctypes.byref(weights.c), ctypes.byref(cache.c),
        _dev_ptr(tokens_in, "tokens_in"), _dev_ptr(pos_in, "pos_in"), _dev_ptr(count, "count"),
        int(max_count), _dev_ptr(ws, "ws"), ws.numel() * ws.element_size(), _stream(stream))
    _check(code, "cc_append_chunk")


# ---- the paper's comparison scorers (Sec. 4) ---------------------------------

def cc_score_recency(cache, scores, stream=None):
    _check(load_library().cc_score_recency(ctypes.byref(cache.c), _dev_ptr(scores, "scores"),
                                           _stream(stream)), "cc_score_recency")


def cc_keyattn_workspace_size(cfg, batch: int, cap: int) -> int:
    return int(load_library().cc_keyattn_workspace_size(ctypes.byref(_cfg(cfg)), batch, cap))


def cc_score_importance(cfg, cache, scores, ws, stream=None):
    _check(load_library().cc_score_importance(
        ctypes.byref(_cfg(cfg)), ctypes.byref(cache.c), _dev_ptr(scores, "scores"),
        _dev_ptr(ws, "ws"), ws.numel() * ws.element_size(), _stream(stream)),
        "cc_score_importance")


def cc_h2o_accumulate(cfg, cache, recent: int, ws, stream=None):
    _check(load_library().cc_h2o_accumulate(
        ctypes.byref(_cfg(cfg)), ctypes.byref(cache.c), int(recent), _dev_ptr(ws, "ws"),
        ws.numel() * ws.element_size(), _stream(stream)), "cc_h2o_accumulate")


def cc_score_h2o(cache, recent: int, scores, stream=None):
    _check(load_library().cc_score_h2o(ctypes.byref(cache.c), int(recent),
                                       _dev_ptr(scores, "scores"), _stream(stream)),
           "cc_score_h2o")


def cc_decode_workspace_size(cfg, batch: int, cap: int) -> int:
    return int(load_library().cc_decode_workspace_size(ctypes.byref(_cfg(cfg)), batch, cap))


def cc_decode_step(cfg, weights, cache, tokens_in, next_tokens, next_logit, ws, stream=None):
    """Decode step: append tokens_in [B] (one each), greedy next tokens [B]."""
    _check(load_library().cc_decode_step(
        ctypes.byref(_cfg(cfg)), ctypes.byref(weights.c), ctypes.byref(cache.c),
        _dev_ptr(tokens_in, "tokens_in"), _dev_ptr(next_tokens, "next_tokens"),
        _dev_ptr(next_logit, "next_logit"), _dev_ptr(ws, "ws"), ws.numel() * ws.element_size(),
        _stream(stream)), "cc_decode_step")


def cc_select_workspace_size(batch: int, cap: int) -> int:
    return int(load_library().cc_select_workspace_size(batch, cap))


def cc_select_keep(scores, seq_len, batch, cap, budget, n_sink, keep_idx, keep_count, ws=None,
                   stream=None):
    nbytes = 0 if ws is None else ws.numel() * ws.element_size()
    code = load_library().cc_select_keep(
        _dev_ptr(scores, "scores"), _dev_ptr(seq_len, "seq_len"), batch, cap,
        _dev_ptr(budget, "budget"), n_sink, _dev_ptr(keep_idx, "keep_idx"),
        _dev_ptr(keep_count, "keep_count"), _dev_ptr(ws, "ws"), nbytes, _stream(stream))
    _check(code, "cc_select_keep")


def cc_compact_workspace_size(cfg, cache: Cache) -> int:
    return int(load_library().cc_compact_workspace_size(ctypes.byref(_cfg(cfg)),
                                                        ctypes.byref(cache.c)))


def cc_compact_kv(cfg, cache: Cache, keep_idx, keep_count, ws, stream=None):
    code = load_library().cc_compact_kv(ctypes.byref(_cfg(cfg)), ctypes.byref(cache.c),
                                        _dev_ptr(keep_idx, "keep_idx"),
                                        _dev_ptr(keep_count, "keep_count"), _dev_ptr(ws, "ws"),
                                        ws.numel() * ws.element_size(), _stream(stream))
    _check(code, "cc_compact_kv")


def cc_compact_kv_static(cfg, cache: Cache, keep_idx, keep_count, stream=None):
    """cc_compact_kv without a workspace: the library's fixed 1 MiB device
    scratch array is used instead (shared by every call on the device)."""
    code = load_library().cc_compact_kv_static(ctypes.byref(_cfg(cfg)), ctypes.byref(cache.c),
                                               _dev_ptr(keep_idx, "keep_idx"),
                                               _dev_ptr(keep_count, "keep_count"), _stream(stream))
    _check(code, "cc_compact_kv_static")


def cc_graph_begin(stream=None):
    """Starts recording the cc_* calls made on `stream` (not the legacy
    default stream) by this thread.  Replays reuse every pointer recorded:
    keep the tensors (and the Weights/Cache objects) alive meanwhile."""
    _check(load_library().cc_graph_begin(_stream(stream)), "cc_graph_begin")


def cc_graph_end(stream=None) -> int:
    """Stops the recording; returns the executable graph's handle."""
    h = ctypes.c_void_p()
    _check(load_library().cc_graph_end(_stream(stream), ctypes.byref(h)), "cc_graph_end")
    return h.value


def cc_graph_launch(graph: int, stream=None):
    _check(load_library().cc_graph_launch(graph, _stream(stream)), "cc_graph_launch")


def cc_graph_destroy(graph: int):
    _check(load_library().cc_graph_destroy(graph), "cc_graph_destroy")


def cc_get_status(stream=None) -> int:
    return int(load_library().cc_get_status(_stream(stream)))


def cc_linear_f32(x, w, y, stream=None):
    code = load_library().cc_linear_f32(_dev_ptr(x, "x"), _dev_ptr(w, "w"), _dev_ptr(y, "y"),
                                        x.shape[0], w.shape[0], x.shape[1], _stream(stream))
    _check(code, "cc_linear_f32")


def cc_counter_causal_attention(q, k, v, seq_len, out, batch, cap, n_q_heads, n_kv_heads,
                                head_dim, stream=None):
    code = load_library().cc_counter_causal_attention(
        _dev_ptr(q, "q"), _dev_ptr(k, "k"), _dev_ptr(v, "v"), _dev_ptr(seq_len, "seq_len"),
        _dev_ptr(out, "out"), batch, cap, n_q_heads, n_kv_heads, head_dim, _stream(stream))
    _check(code, "cc_counter_causal_attention")


def cc_counter_causal_attention_split(q, k, v, seq_len, out, batch, cap, n_q_heads, n_kv_heads,
                                      head_dim, stream=None):
    code = load_library().cc_counter_causal_attention_split(
        _dev_ptr(q, "q"), _dev_ptr(k, "k"), _dev_ptr(v, "v"), _dev_ptr(seq_len, "seq_len"),
        _dev_ptr(out, "out"), batch, cap, n_q_heads, n_kv_heads, head_dim, _stream(stream))
    _check(code, "cc_counter_causal_attention_split")


def cc_timing_enable(on: bool):
    _check(load_library().cc_timing_enable(1 if on else 0), "cc_timing_enable")


def cc_timing_collect() -> dict:
    """{kernel name: (launches, total ms)} of the launches recorded since enabling."""
    counts = (ctypes.c_int32 * KERNEL_COUNT)()
    total = (ctypes.c_double * KERNEL_COUNT)()
    lib = load_library()
    _check(lib.cc_timing_collect(counts, total), "cc_timing_collect")
    return {lib.cc_kernel_name(k).decode(): (int(counts[k]), float(total[k]))
            for k in range(KERNEL_COUNT) if counts[k]}


def cc_debug_withhold_compact_unit(unit: int):
    """Test hook: the next cc_compact_kv runs with `unit` never publishing its flag."""
    _check(load_library().cc_debug_withhold_compact_unit(int(unit)),
           "cc_debug_withhold_compact_unit")


def alloc_workspace(nbytes: int, device="cuda") -> torch.Tensor:
    """A caller-owned device workspace of at least nbytes (256-byte aligned by torch)."""
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)
