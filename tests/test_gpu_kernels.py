"""GPU unit tests of single kernels through the C ABI: the tcgen05 GEMM and
the counter-causal attention (Sec. 3.1), against the CPU oracle / fp64
reference on seeded inputs."""
import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def cc():
    from paper_2607_27600_gb300 import cc as mod
    mod.load_library()
    return mod


@pytest.mark.parametrize("rows,n,k", [(128, 256, 64), (300, 96, 200), (1000, 512, 4096),
                                      (129, 32, 8), (2048, 4096, 1408)])
def test_linear_matches_fp64(cc, rows, n, k):
    x = synth.normal((rows, k), 1.0, 1, f"x{rows}.{n}.{k}")
    w = synth.normal((n, k), 0.05, 1, f"w{rows}.{n}.{k}")
    y = torch.empty(rows, n, dtype=torch.float32, device="cuda")
    cc.cc_linear_f32(x.cuda(), w.cuda(), y)
    torch.cuda.synchronize()
    want = x.double() @ w.double().T
    err = (y.cpu().double() - want).abs().max().item()
    scale = want.abs().max().item()
    assert err <= 1e-4 * scale + 1e-5, (err, scale)


def _attn_case(cc, batch, cap, seq, hq, hkv, dh, seed, kscale=1.0, rows=None):
    q = synth.normal((batch * cap, hq, dh), 1.0, seed, "q")
    k = synth.normal((batch, cap, hkv, dh), kscale, seed, "k")
    v = synth.normal((batch, cap, hkv, dh), 1.0, seed, "v")
    sl = torch.tensor(seq, dtype=torch.int32)
    out = torch.full((batch * cap, hq, dh), float("nan"), dtype=torch.bfloat16, device="cuda")
    cc.cc_counter_causal_attention(q.cuda(), k.cuda(), v.cuda(), sl.cuda(), out, batch, cap, hq,
                                   hkv, dh)
    assert cc.cc_get_status() == cc.CC_OK
    got = out.float().cpu().numpy().reshape(batch, cap, hq, dh)
    qn = q.float().numpy().reshape(batch, cap, hq, dh)
    kn, vn = k.float().numpy(), v.float().numpy()
    for b, n in enumerate(seq):
        r = np.arange(n) if rows is None else np.unique(np.clip(rows(n), 0, n - 1))
        want = oracle.counter_causal_attention(qn[b, r], kn[b], vn[b], r, n)
        g = got[b, r]
        assert np.all(np.isfinite(g))
        err = np.abs(g - want).max() if n else 0.0
        # bf16 output rounding (2^-9 relative) plus bf16 P in the PV product
        assert err <= 2e-2 * max(1.0, np.abs(want).max()), (b, n, err)
        if n and r[-1] == n - 1:
            np.testing.assert_array_equal(g[-1], 0.0)   # last row: nothing to attend


# group sizes 3, 5, 6, 7 leave 1-4 of a unit's 256 query rows unused
@pytest.mark.parametrize("hq,hkv,dh", [(8, 2, 64), (32, 8, 128), (28, 4, 128), (4, 4, 128),
                                       (8, 1, 64), (6, 2, 128), (10, 2, 64), (12, 2, 128)])
def test_attention_shapes(cc, hq, hkv, dh):
    _attn_case(cc, 2, 384, [384, 301], hq, hkv, dh, seed=hq * 7 + dh)


@pytest.mark.parametrize("seq", [[1], [2], [3], [129], [127, 128], [256, 1, 5, 200]])
def test_attention_edge_lengths(cc, seq):
    _attn_case(cc, len(seq), 256, seq, 8, 2, 128, seed=sum(seq))


def test_attention_ragged_large_ragged_tail(cc):
    _attn_case(cc, 2, 1200, [1200, 777], 32, 8, 128, seed=5, kscale=2.0)


@pytest.mark.parametrize("batch,seq", [(1, [40960]), (2, [40960, 30001])])
def test_attention_grouped_unit_order(cc, batch, seq):
    """Caches long enough that units run in groups of a few (sequence, KV
    head) streams, the last group smaller: sampled rows of every stream."""
    def rows(n):
        return np.array([0, 1, 63, 64, 65, 5000, n // 2, n - 130, n - 129, n - 2, n - 1])
    _attn_case(cc, batch, 40960, seq, 32, 8, 128, seed=41 + batch, rows=rows)


@pytest.mark.parametrize("hq,hkv", [(8, 2), (28, 4)])
def test_attention_ignores_non_finite_stale_slots(cc, hq, hkv):
    """Slots past seq_len may hold any bits (NaN here); outputs must not see them."""
    batch, cap, dh = 1, 256, 128
    seq = [150]
    q = synth.normal((cap, hq, dh), 1.0, 9, "q").cuda()
    k = synth.normal((batch, cap, hkv, dh), 1.0, 9, "k").cuda()
    v = synth.normal((batch, cap, hkv, dh), 1.0, 9, "v").cuda()
    k2, v2 = k.clone(), v.clone()
    k2[:, 150:] = float("nan")
    v2[:, 150:] = float("inf")
    sl = torch.tensor(seq, dtype=torch.int32, device="cuda")
    o1 = torch.zeros(cap, hq, dh, dtype=torch.bfloat16, device="cuda")
    o2 = torch.zeros_like(o1)
    cc.cc_counter_causal_attention(q, k, v, sl, o1, batch, cap, hq, hkv, dh)
    cc.cc_counter_causal_attention(q, k2, v2, sl, o2, batch, cap, hq, hkv, dh)
    torch.cuda.synchronize()
    assert torch.equal(o1[:150], o2[:150])


def test_attention_past_slots_do_not_leak(cc):
    """Row i is bitwise unchanged when K/V at slots <= i change (masked p = 0)."""
    batch, cap, hq, hkv, dh = 1, 512, 8, 2, 128
    q = synth.normal((cap, hq, dh), 1.0, 10, "q").cuda()
    k = synth.normal((batch, cap, hkv, dh), 1.0, 10, "k").cuda()
    v = synth.normal((batch, cap, hkv, dh), 1.0, 10, "v").cuda()
    sl = torch.tensor([512], dtype=torch.int32, device="cuda")
    o1 = torch.zeros(cap, hq, dh, dtype=torch.bfloat16, device="cuda")
    o2 = torch.zeros_like(o1)
    cc.cc_counter_causal_attention(q, k, v, sl, o1, batch, cap, hq, hkv, dh)
    k2, v2 = k.clone(), v.clone()
    k2[:, :301] += 3.0
    v2[:, :301] -= 5.0
    cc.cc_counter_causal_attention(q, k2, v2, sl, o2, batch, cap, hq, hkv, dh)
    torch.cuda.synchronize()
    assert torch.equal(o1[300:], o2[300:])
    assert not torch.equal(o1[:299], o2[:299])


def _split_pair(x):
    """fp64 -> bf16 pair (hi, lo) with hi = bf16(x), lo = bf16(x - hi)."""
    hi = torch.from_numpy(np.asarray(x, np.float32)).to(torch.bfloat16)
    lo = (torch.from_numpy(np.asarray(x, np.float64)) - hi.double()).float().to(torch.bfloat16)
    return hi, lo


@pytest.mark.parametrize("hq,hkv,dh,seq", [(32, 8, 128, [384, 301]), (8, 2, 64, [384, 1]),
                                           (28, 4, 128, [129, 255]), (12, 2, 128, [2, 384]),
                                           (10, 2, 64, [3, 200])])
def test_attention_split_operands_match_oracle_tightly(cc, hq, hkv, dh, seq):
    """The precise pass's attention: queries in as hi + lo, probabilities into
    P V as hi + lo, output out as hi + lo.  With K and V exact bf16 inputs the
    only roundings left are about 2^-17 relative (the pairs) and fp32
    arithmetic, so the output matches the oracle's fp64 attention of the same
    queries within 1e-4 of its scale (a single bf16 operand would miss by
    about 2^-9)."""
    batch, cap = len(seq), 384
    q = synth.normal((batch * cap, hq, dh), 1.0, 50 + dh, "q").double().numpy()
    q = q * (1 + 1e-3 * synth.normal(q.shape, 1.0, 51, "qj").double().numpy())   # not bf16 values
    k = synth.normal((batch, cap, hkv, dh), 1.5, 50 + dh, "k")
    v = synth.normal((batch, cap, hkv, dh), 1.0, 50 + dh, "v")
    qh, ql = _split_pair(q)
    qpair = torch.cat([qh, ql], dim=1).cuda()                 # [rows][2 hq][dh]
    out = torch.full((batch * cap, 2 * hq, dh), float("nan"), dtype=torch.bfloat16, device="cuda")
    sl = torch.tensor(seq, dtype=torch.int32, device="cuda")
    cc.cc_counter_causal_attention_split(qpair, k.cuda(), v.cuda(), sl, out, batch, cap, hq, hkv,
                                         dh)
    assert cc.cc_get_status() == cc.CC_OK
    o = out.double().cpu()
    got = (o[:, :hq] + o[:, hq:]).numpy().reshape(batch, cap, hq, dh)
    qx = (qh.double() + ql.double()).numpy().reshape(batch, cap, hq, dh)   # the value the pair holds
    kn, vn = k.float().numpy(), v.float().numpy()
    for b, n in enumerate(seq):
        r = np.arange(n)
        want = oracle.counter_causal_attention(qx[b, r], kn[b], vn[b], r, n)
        err = np.abs(got[b, r] - want).max()
        assert err <= 1e-4 * max(1.0, np.abs(want).max()), (b, n, err)
        np.testing.assert_array_equal(got[b, n - 1], 0.0)


def test_attention_split_needs_the_lo_halves(cc):
    """Dropping the lo halves of the queries moves the output by the bf16
    rounding of q (far beyond the split bar), so the kernel really reads them."""
    batch, cap, hq, hkv, dh = 1, 256, 8, 2, 128
    q = synth.normal((cap, hq, dh), 1.0, 60, "q").double().numpy() * (1 + 1e-3)
    k = synth.normal((batch, cap, hkv, dh), 2.0, 60, "k").cuda()
    v = synth.normal((batch, cap, hkv, dh), 1.0, 60, "v").cuda()
    qh, ql = _split_pair(q)
    sl = torch.tensor([cap], dtype=torch.int32, device="cuda")
    outs = []
    for lo in (ql, torch.zeros_like(ql)):
        out = torch.zeros(cap, 2 * hq, dh, dtype=torch.bfloat16, device="cuda")
        cc.cc_counter_causal_attention_split(torch.cat([qh, lo], dim=1).cuda(), k, v, sl, out,
                                             batch, cap, hq, hkv, dh)
        torch.cuda.synchronize()
        outs.append((out[:, :hq].double() + out[:, hq:].double()).cpu())
    assert (outs[0] - outs[1]).abs().max().item() > 1e-3
