"""The C ABI library builds, loads without a GPU and exports every entry
point the public headers declare; host-side argument checks answer without
touching the device (no GPU)."""
import ctypes
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    names = set()
    for h in os.listdir(os.path.join(ROOT, "include")):
        if h.endswith(".h"):
            src = open(os.path.join(ROOT, "include", h)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"\b(cc_[a-z0-9_]+)\s*\(", src))
    return names


@pytest.fixture(scope="module")
def lib():
    from paper_2607_27600_gb300 import build, cc
    build.build_library()
    return cc.load_library()


def test_every_declared_symbol_is_exported(lib):
    names = declared_functions()
    assert {"cc_score_layer", "cc_score_full", "cc_select_keep", "cc_compact_kv"} <= names
    for n in sorted(names):
        assert hasattr(lib, n), n


def test_binding_covers_every_declared_symbol(lib):
    from paper_2607_27600_gb300 import cc
    assert declared_functions() == set(cc.exported_symbols())


def test_status_strings(lib):
    from paper_2607_27600_gb300 import cc
    assert cc.cc_status_str(cc.CC_OK) == "ok"
    assert "workspace" in cc.cc_status_str(cc.CC_ERR_WORKSPACE)


def test_host_side_validation_without_device(lib):
    from paper_2607_27600_gb300 import cc
    # null arguments are rejected before anything reaches the device
    assert lib.cc_select_keep(None, None, 1, 1, None, 0, None, None, None, 0, None) == \
        cc.CC_ERR_INVALID_ARG
    assert lib.cc_score_layer(None, None, None, 0, None, None, 0, None) == cc.CC_ERR_INVALID_ARG
    assert lib.cc_append_chunk(None, None, None, None, None, None, 1, None, 0, None) == \
        cc.CC_ERR_INVALID_ARG
    bad = cc.cc_model_cfg(1, 100, 8, 3, 128, 256, 10, 1e4, 1e-5)   # Hq % Hkv != 0
    assert lib.cc_score_workspace_size(ctypes.byref(bad), 1, 16, 0) == 0
    odd = cc.cc_model_cfg(1, 256, 8, 2, 96, 256, 10, 1e4, 1e-5)    # head_dim 96
    assert lib.cc_score_workspace_size(ctypes.byref(odd), 1, 16, 0) == 0
    # RoPE scaling: off when zero, else factor >= 1 and 0 < low < high, orig > 0
    ok = cc.cc_model_cfg(1, 256, 8, 2, 64, 256, 10, 5e5, 1e-5, 8.0, 1.0, 4.0, 8192)
    assert lib.cc_score_workspace_size(ctypes.byref(ok), 1, 16, 0) > 0
    for sc in [(0.5, 1.0, 4.0, 8192), (8.0, 4.0, 1.0, 8192), (8.0, 0.0, 4.0, 8192),
               (8.0, 1.0, 4.0, 0)]:
        bad_sc = cc.cc_model_cfg(1, 256, 8, 2, 64, 256, 10, 5e5, 1e-5, *sc)
        assert lib.cc_score_workspace_size(ctypes.byref(bad_sc), 1, 16, 0) == 0, sc


def test_workspace_size_formula(lib):
    from paper_2607_27600_gb300 import cc
    from synth.configs import LLAMA3_8B
    n = cc.cc_score_workspace_size(LLAMA3_8B, 1, 8192, cc.SCORE_LOGIT)
    rows, d, q, f = 8192, 4096, 4096, 14336
    assert n >= rows * (2 * d + 2 * q * 2 + 4 * d + 2 * f)
    assert cc.cc_score_workspace_size(LLAMA3_8B, 1, 8192, cc.SCORE_LOGPROB) > n
    # the append reuses the scoring rows plus two int32 [batch] range arrays
    assert cc.cc_append_workspace_size(LLAMA3_8B, 1, 8192) >= n


def test_compaction_plan_covers_every_array(lib):
    """The compaction workspace grows with every array the cache holds (a plan
    that registered no arrays would compact nothing); computed on the host."""
    import ctypes
    from paper_2607_27600_gb300 import cc
    cfg = cc.cc_model_cfg(2, 256, 8, 2, 64, 384, 1000, 1e4, 1e-5)
    fake = [ctypes.c_void_p(4096 * (i + 1)) for i in range(8)]   # never dereferenced
    ks = (ctypes.c_void_p * 2)(fake[0], fake[1])
    vs = (ctypes.c_void_p * 2)(fake[2], fake[3])
    none = (ctypes.c_void_p * 2)(None, None)
    full = cc.cc_kv_cache(1, 4096, fake[4], ks, vs, fake[5], fake[6], fake[7])
    only_x = cc.cc_kv_cache(1, 4096, fake[4], none, none, fake[5], fake[6], None)
    n_full = lib.cc_compact_workspace_size(ctypes.byref(cfg), ctypes.byref(full))
    n_x = lib.cc_compact_workspace_size(ctypes.byref(cfg), ctypes.byref(only_x))
    assert n_x > 256 and n_full > n_x


def _header_struct_fields(name):
    src = open(os.path.join(ROOT, "include", "cc.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    m = re.search(r"typedef struct\s*\{([^}]*)\}\s*" + name + r"\s*;", src)
    assert m, name
    fields = []
    for decl in m.group(1).split(";"):
        decl = decl.strip()
        if decl:
            fields += [re.findall(r"(\w+)\s*$", part.strip())[0] for part in decl.split(",")]
    return fields


@pytest.mark.parametrize("name", ["cc_model_cfg", "cc_layer_weights", "cc_model_weights",
                                  "cc_kv_cache"])
def test_binding_structs_match_the_header(name):
    """The ctypes mirrors of the public structs list the header's fields in
    the header's order (a missing or reordered field would shift every later
    member the library reads)."""
    from paper_2607_27600_gb300 import cc
    assert [f[0] for f in getattr(cc, name)._fields_] == _header_struct_fields(name)


def header_enums():
    """name -> value of every enumerator the public headers define."""
    vals = {}
    for h in os.listdir(os.path.join(ROOT, "include")):
        if not h.endswith(".h"):
            continue
        src = re.sub(r"/\*.*?\*/", "", open(os.path.join(ROOT, "include", h)).read(), flags=re.S)
        for body in re.findall(r"typedef\s+enum\s*\{(.*?)\}", src, flags=re.S):
            nxt = 0
            for item in body.split(","):
                item = item.strip()
                if not item:
                    continue
                name, _, val = item.partition("=")
                nxt = int(val.strip(), 0) if val.strip() else nxt
                vals[name.strip()] = nxt
                nxt += 1
    return vals


def test_binding_constants_match_the_headers(lib):
    from paper_2607_27600_gb300 import cc
    e = header_enums()
    pairs = {"CC_OK": cc.CC_OK, "CC_ERR_INVALID_ARG": cc.CC_ERR_INVALID_ARG,
             "CC_ERR_CUDA": cc.CC_ERR_CUDA, "CC_ERR_BUDGET": cc.CC_ERR_BUDGET,
             "CC_ERR_WORKSPACE": cc.CC_ERR_WORKSPACE, "CC_ERR_TIMEOUT": cc.CC_ERR_TIMEOUT,
             "CC_ERR_UNSUPPORTED": cc.CC_ERR_UNSUPPORTED, "CC_ERR_DEVICE_ARG": cc.CC_ERR_DEVICE_ARG,
             "CC_SCORE_LOGIT": cc.SCORE_LOGIT, "CC_SCORE_LOGPROB": cc.SCORE_LOGPROB,
             "CC_SCORE_PRECISE": cc.SCORE_PRECISE, "CC_SCORE_RANGE_ONLY": cc.SCORE_RANGE_ONLY,
             "CC_KV_BF16": cc.KV_BF16, "CC_KV_E4M3": cc.KV_E4M3,
             "CC_KV_SLOT_MAJOR": cc.KV_SLOT_MAJOR, "CC_KV_HEAD_MAJOR": cc.KV_HEAD_MAJOR,
             "CC_KERNEL_COUNT": cc.KERNEL_COUNT}
    for name, val in pairs.items():
        assert e[name] == val, (name, e[name], val)
    # every profiled kernel kind has its own name in the library
    names = [lib.cc_kernel_name(k).decode() for k in range(cc.KERNEL_COUNT)]
    assert len(set(names)) == cc.KERNEL_COUNT and "unknown" not in names
    assert lib.cc_kernel_name(cc.KERNEL_COUNT).decode() == "unknown"


def test_bf16_to_f16_argument_checks_without_device(lib):
    """cc_bf16_to_f16 refuses null, misaligned, overlapping and non-multiple-
    of-8 arguments on the host (nothing reaches a device); n = 0 is a no-op."""
    from paper_2607_27600_gb300 import cc
    assert lib.cc_bf16_to_f16(None, None, 0, None) == cc.CC_OK
    assert lib.cc_bf16_to_f16(None, None, 8, None) == cc.CC_ERR_INVALID_ARG
    base = 1 << 20   # addresses only: none is dereferenced on these paths
    assert lib.cc_bf16_to_f16(base, base + 4096, 12, None) == cc.CC_ERR_INVALID_ARG   # n % 8
    assert lib.cc_bf16_to_f16(base + 2, base + 4096, 8, None) == cc.CC_ERR_INVALID_ARG  # align
    assert lib.cc_bf16_to_f16(base, base + 16, 16, None) == cc.CC_ERR_INVALID_ARG     # overlap


def test_binding_operand_type_check_without_device():
    """The binding's dtype check of the layer matrices against the operand
    mode (host logic: the CUDA tensors only carry the dtype)."""
    import types

    import torch
    from paper_2607_27600_gb300 import cc
    layer = {f: torch.zeros(8, 8, dtype=torch.bfloat16) for f in cc.F16_MATRICES}
    w = types.SimpleNamespace(w={"layers": [None, layer]})
    cc._check_operand_type(w, cc.SCORE_LOGIT)
    cc._check_operand_type(w, cc.SCORE_LOGPROB | cc.SCORE_PRECISE)
    with pytest.raises(ValueError):
        cc._check_operand_type(w, cc.SCORE_LOGIT | cc.SCORE_F16)
    w16 = types.SimpleNamespace(w={"layers": [{f: t.half() for f, t in layer.items()}]})
    cc._check_operand_type(w16, cc.SCORE_LOGIT | cc.SCORE_F16)
    with pytest.raises(ValueError):
        cc._check_operand_type(w16, cc.SCORE_LOGIT)
