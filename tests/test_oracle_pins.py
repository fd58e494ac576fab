"""Pins for the CPU oracle: each test checks the oracle against something
other than itself (hand-worked values, closed forms, brute force, a second
independent formulation, printed paper values)."""
import json
import math
import os

import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# rounding helpers
# --------------------------------------------------------------------------
def test_fp16_rn_is_single_rounding():
    # 1 + 2^-11 + 2^-40 lies just above the midpoint between fp16 1 and
    # 1 + 2^-10; a detour through fp32 would round to the midpoint first and
    # then to even (1.0).
    assert O.fp16_rn(1 + 2.0 ** -11 + 2.0 ** -40) == 1 + 2.0 ** -10
    assert O.fp16_rn(1 + 2.0 ** -11) == 1.0            # tie -> even
    assert O.fp16_rn(1 + 3 * 2.0 ** -11) == 1 + 2 * 2.0 ** -10  # tie -> even
    assert O.fp16_rn(2.0 ** -24) == 2.0 ** -24           # smallest subnormal
    assert O.fp16_rn(2.0 ** -26) == 0.0


def test_bf16_rn_examples():
    assert O.bf16_rn(1 + 2.0 ** -8) == 1.0               # tie -> even
    assert O.bf16_rn(1 + 3 * 2.0 ** -8) == 1 + 2.0 ** -6
    assert O.bf16_rn(-3.0) == -3.0
    bits = synth.bf16_bits(np.array([1 + 2.0 ** -8, 1 + 3 * 2.0 ** -8], np.float32))
    assert list(bits) == [0x3F80, 0x3F82]


# --------------------------------------------------------------------------
# P1: bitstream layout and round trips
# --------------------------------------------------------------------------
def _bit_reader(seg_bytes, b, kb):
    """Pure-Python reader: code p = sum_j bit(p*b + j) << j."""
    out = []
    for p in range(kb):
        v = 0
        for j in range(b):
            pos = p * b + j
            v |= ((seg_bytes[pos // 8] >> (pos % 8)) & 1) << j
        out.append(v)
    return out


def test_bitstream_hand_examples():
    with open(os.path.join(GOLDEN, "bitstream_examples.json")) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        codes = np.array([c["codes"]], dtype=np.int64)
        got = O.pack_codes(codes, c["b"], 16)[0]
        assert bytes(got).hex() == c["bytes_hex"], c


@pytest.mark.parametrize("b", [2, 3, 4, 8])
@pytest.mark.parametrize("kb", [1, 5, 63, 64, 65, 127, 128, 129, 200])
def test_pack_unpack_roundtrip(b, kb):
    rng = np.random.default_rng(1000 * b + kb)
    codes = rng.integers(0, 1 << b, size=(3, kb))
    nbytes = O.seg_bytes(b, kb)
    assert nbytes % 16 == 0 and nbytes * 8 >= kb * b and nbytes * 8 - kb * b < 128
    seg = O.pack_codes(codes, b, nbytes)
    assert seg.shape == (3, nbytes)
    for n in range(3):
        assert _bit_reader(list(seg[n]), b, kb) == list(codes[n])
        # padding bits are zero
        tail = int.from_bytes(bytes(seg[n]), "little") >> (kb * b)
        assert tail == 0
    assert np.array_equal(O.unpack_codes_from_bytes(seg, b, kb), codes)


def _forced_layer(N, K, seed, widths=(2, 3, 4, 8, 16)):
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed, widths)
    return W, a, O.pack_layer(W, a, 3.0, bits=bits)


def test_layer_layout_invariants():
    W, a, L = _forced_layer(5, 300, 11)
    assert L["row_stride"] % 16 == 0
    off = 0
    for blk in L["blocks"]:
        assert blk["seg_off"] == off
        off += blk["seg_bytes"]
        cols = L["perm"][blk["pos0"]:blk["pos0"] + blk["n_ch"]]
        assert np.all(L["bits"][cols] == blk["bits"])
        assert np.all(np.diff(cols) > 0)  # ascending original index in a block
    assert off == L["row_stride"]
    assert [blk["bits"] for blk in L["blocks"]] == [2, 3, 4, 8, 16]
    # codes read back with the pure-python reader, block by block
    codes = O.unpack_codes(L)
    for blk in L["blocks"]:
        if blk["bits"] == 16:
            continue
        o, kb, b = blk["seg_off"], blk["n_ch"], blk["bits"]
        for n in range(L["N"]):
            seg = list(L["packed"][n, o:o + blk["seg_bytes"]])
            assert _bit_reader(seg, b, kb) == list(codes[n, blk["pos0"]:blk["pos0"] + kb])


# --------------------------------------------------------------------------
# P2: 16-bit channels are fp16(w) bit for bit
# --------------------------------------------------------------------------
def test_16bit_channels_are_fp16():
    W, a = synth.layer_weights(4, 70, 3)
    bits = np.full(70, 16)
    L = O.pack_layer(W, a, 16.0, bits=bits)
    Wd = O.dequant(L)
    ref = W[:, L["perm"]].astype(np.float16).astype(np.float64)
    assert np.array_equal(Wd, ref)
    assert L["n_groups"] == 0
    assert L["row_stride"] == O.seg_bytes(16, 70) == 144


# --------------------------------------------------------------------------
# P3: quantiser against brute force and closed forms
# --------------------------------------------------------------------------
@pytest.mark.parametrize("b", [2, 3, 4, 8])
def test_quantizer_brute_force(b):
    rng = np.random.default_rng(b)
    qmax = (1 << b) - 1
    for trial in range(60):
        n = int(rng.integers(1, 17))
        w = rng.normal(rng.normal(0, 0.5), rng.uniform(1e-3, 2), size=n)
        s, z, q = O.quantize_group(w, b)
        assert s > 0 and float(np.float16(s)) == s
        assert z == int(z) and 0 <= z <= qmax
        grid = (np.arange(qmax + 1) - z) * s
        for i in range(n):
            err = np.abs(grid - w[i])
            best = np.min(err)
            wq = (q[i] - z) * s
            raw = np.rint(w[i] / s) + z
            if 0 <= raw <= qmax:
                # unclamped: nearest grid point (a tie may pick either side)
                assert abs(abs(wq - w[i]) - best) <= 1e-12 * max(1.0, abs(w[i]))
                assert abs(wq - w[i]) <= s / 2 * (1 + 1e-12)
            else:
                assert q[i] in (0, qmax)
                assert abs(wq - w[i]) == pytest.approx(best, rel=1e-12, abs=1e-300)


def test_quantizer_exact_on_grid_and_constant_groups():
    s = float(np.float16(0.0123))
    w = np.array([-2 * s, -s, 0.0, s])
    s2, z, q = O.quantize_group(w, 2)
    assert s2 == s and z == 2 and list(q) == [0, 1, 2, 3]
    for c in (0.5, -0.5, 0.0, 3.0):
        w = np.full(7, c)
        s, z, q = O.quantize_group(w, 3)
        assert np.all((q - z) * s == c)
    # constant zero group falls back to s = 2^-14
    s, z, q = O.quantize_group(np.zeros(4), 4)
    assert s == 2.0 ** -14 and z == 0 and np.all(q == 0)


def test_quantize_rows_matches_scalar():
    rng = np.random.default_rng(5)
    Wb = rng.normal(0, 0.02, size=(6, 150))
    Wb[2, :64] = 0.25
    for b in (2, 3, 4, 8):
        S, Z, Q = O.quantize_rows(Wb, b)
        for n in range(6):
            for g in range(3):
                cols = slice(64 * g, min(64 * g + 64, 150))
                s, z, q = O.quantize_group(Wb[n, cols], b)
                assert S[n, g] == s and Z[n, g] == z
                assert np.array_equal(Q[n, cols], q)


def test_reject_out_of_range_weights():
    W = np.zeros((2, 8), np.float32)
    W[0, 0] = 70000.0
    with pytest.raises(ValueError):
        O.pack_layer(W, np.ones(8, np.float32), 3.0)
    W[0, 0] = np.nan
    with pytest.raises(ValueError):
        O.pack_layer(W, np.ones(8, np.float32), 3.0)


# --------------------------------------------------------------------------
# saliency closed form
# --------------------------------------------------------------------------
def test_saliency_closed_form():
    N, K = 16, 5
    c = np.array([0.5, -2.0, 0.0, 0.25, 3.0], np.float32)
    W = np.tile(c, (N, 1))
    a = np.array([1.0, 2.0, 3.0, 0.5, 4.0], np.float32)
    sal = O.saliency(W, a)
    ref = a.astype(np.float64) * np.abs(c.astype(np.float64)) * 4.0
    assert np.array_equal(sal, ref)


# --------------------------------------------------------------------------
# P4 / P7: allocation
# --------------------------------------------------------------------------
def test_residual_budget_formula():
    assert O.residual_budget(3.0, 2048, 2) == 2048
    assert O.residual_budget(2.5, 11, 2) == 6      # round(27.5) = 28 (half up)
    assert O.residual_budget(2.5, 10, 2) == 5
    assert O.residual_budget(2.0, 10, 2) == 0
    assert O.residual_budget(1.5, 10, 2) == -5


@pytest.mark.parametrize("K", [10, 11, 64])
def test_allocation_equal_saliency(K):
    sal = np.ones(K)
    assert np.all(O.allocate_bits(sal, 3.0) == 3)
    assert np.all(O.allocate_bits(sal, 4.0) == 4)
    assert np.all(O.allocate_bits(sal, 2.0) == 2)
    b25 = O.allocate_bits(sal, 2.5)
    n3 = O.residual_budget(2.5, K, 2)
    assert list(b25) == [3] * n3 + [2] * (K - n3)   # index tie-break
    assert np.all(O.allocate_bits(sal, 16.0) == 16)


def test_gain_ladder_strictly_decreasing():
    for s in (0.01, 1.0, 123.0):
        g = [O.gain(s, 2, 3), O.gain(s, 3, 4), O.gain(s, 4, 8), O.gain(s, 8, 16)]
        assert all(g[i] > g[i + 1] > 0 for i in range(3))
        # closed forms of the four gains as multiples of sal^2
        c = [1 / 9 - 1 / 49, 1 / 49 - 1 / 225, (1 / 225 - 1 / 65025) / 4, (1 / 65025) / 8]
        for gi, ci in zip(g, c):
            assert gi == pytest.approx(ci * s * s, rel=1e-12)


def _alloc_sorted_scan(sal, B):
    """Second formulation: every (channel, step) candidate sorted by
    (gain desc, channel asc), scanned once."""
    K = len(sal)
    pal = O.PALETTE
    delta = O.residual_budget(B, K, pal[0])
    bits = [pal[0]] * K
    stopped = [False] * K
    cands = []
    for k in range(K):
        for i in range(len(pal) - 1):
            cands.append((-O.gain(sal[k], pal[i], pal[i + 1]), k, pal[i], pal[i + 1]))
    cands.sort()
    for _, k, b0, b1 in cands:
        if delta <= 0:
            break
        if stopped[k] or bits[k] != b0:
            continue
        if b1 - b0 > delta:
            stopped[k] = True
            continue
        bits[k] = b1
        delta -= b1 - b0
    return np.array(bits)


@pytest.mark.parametrize("seed", range(8))
def test_allocation_matches_sorted_scan(seed):
    rng = np.random.default_rng(seed)
    K = int(rng.integers(1, 300))
    sal = rng.lognormal(0, 1.5, size=K)
    if seed % 3 == 0:
        sal[: K // 2] = sal[0]  # ties
    for B in (2.0, 2.3, 3.0, 3.7, 4.5, 6.0, 9.9, 16.0):
        assert np.array_equal(O.allocate_bits(sal, B), _alloc_sorted_scan(sal, B))


@pytest.mark.parametrize("B", [2.1, 3.0, 3.5, 4.0, 4.5, 5.0, 6.0])
def test_budget_invariant(B):
    W, a = synth.layer_weights(32, 2048, 1)
    bits = O.allocate_bits(O.saliency(W, a), B)
    total = int(bits.sum())
    target = int(math.floor(B * 2048 + 0.5))
    if np.any(bits <= 3):
        assert total == target
    else:
        assert 0 <= target - total <= 3
    assert abs(bits.mean() - B) <= 0.5 / 2048 + 1e-12


def test_allocation_respects_saliency_order():
    # a channel never ends below a less salient one
    W, a = synth.layer_weights(16, 512, 2)
    sal = O.saliency(W, a)
    bits = O.allocate_bits(sal, 3.3)
    order = np.argsort(-sal, kind="stable")
    assert np.all(np.diff(bits[order]) <= 0)


def test_saliency_ladder_rule():
    sal = np.array([1.0, 5.0, 3.0, 2.0])
    # Delta = 12 - 8 = 4: channel 1 climbs 2->3->4 (2 bits), then 4->8 does
    # not fit (needs 4 > 2); channel 2 takes 2->3->4 with the last 2.
    bits = O.allocate_bits(sal, 3.0, rule=O.SALIENCY_LADDER)
    assert list(bits) == [2, 4, 4, 2]
    # Delta = 12: channel 1 reaches 8 (8->16 needs 8 > 6 left), channel 2
    # then spends the remaining 6 bits on 2->3->4->8.
    bits = O.allocate_bits(sal, 5.0, rule=O.SALIENCY_LADDER)
    assert list(bits) == [2, 8, 8, 2]


def test_synthetic_allocation_shape():
    # K=2048 at B=3.0: mostly 2/3/4 with a few 8-bit channels (Table 1 shape)
    W, a = synth.layer_weights(2048, 2048, 1001)
    L = O.pack_layer(W, a, 3.0)
    cnt = {b: int(np.sum(L["bits"] == b)) for b in O.PALETTE}
    assert cnt[3] > 0 and cnt[4] > 0 and cnt[2] > 0
    assert cnt[8] < 0.1 * 2048 and cnt[16] < 0.01 * 2048
    assert O.realized_budget(L) == 3.0


# --------------------------------------------------------------------------
# P5 / P6: products
# --------------------------------------------------------------------------
def test_permutation_invariance():
    W, a, L = _forced_layer(9, 333, 21)
    _, x = synth.activations(a, 3, 21)
    y1 = O.linear(L, x)
    y2 = O.linear_natural(L, x)
    assert np.max(np.abs(y1 - y2)) <= 1e-12 * np.max(np.abs(y2))


@pytest.mark.parametrize("seed", range(6))
def test_brute_force_dot_small(seed):
    rng = np.random.default_rng(seed)
    K = int(rng.integers(1, 17))
    N = int(rng.integers(1, 5))
    W = rng.normal(0, 0.3, size=(N, K)).astype(np.float32)
    bits = rng.choice([2, 3, 4, 8, 16], size=K)
    L = O.pack_layer(W, np.ones(K, np.float32), 3.0, bits=bits)
    x = rng.normal(size=K)
    y = O.linear(L, x)[0]
    # direct: quantise each width class of each row straight from W in
    # original channel order (K <= 16 < 64: one group per width)
    for n in range(N):
        acc = 0.0
        for b in set(bits.tolist()):
            ks = [k for k in range(K) if bits[k] == b]
            if b == 16:
                for k in ks:
                    acc += x[k] * float(np.float16(W[n, k]))
                continue
            s, z, q = O.quantize_group(W[n, ks].astype(np.float64), b)
            for qi, k in zip(q, ks):
                acc += x[k] * ((qi - z) * s)
        assert y[n] == pytest.approx(acc, rel=1e-12, abs=1e-15)


def test_all16_matches_torch_fp32():
    torch = pytest.importorskip("torch")
    W, a = synth.layer_weights(8, 96, 4)
    L = O.pack_layer(W, a, 16.0, bits=np.full(96, 16))
    xb, x = synth.activations(a, 2, 4)
    y = O.linear(L, x)
    Wt = torch.from_numpy(W.astype(np.float16).astype(np.float32))
    yt = (torch.from_numpy(x.astype(np.float32)) @ Wt.T).numpy().astype(np.float64)
    assert np.max(np.abs(y - yt)) <= 1e-5 * np.max(np.abs(y)) + 1e-6


# --------------------------------------------------------------------------
# P8: merge
# --------------------------------------------------------------------------
def test_permute_merge_definition():
    rng = np.random.default_rng(0)
    for n in (1, 2, 17):
        beta = rng.permutation(n)
        pc = rng.permutation(n)
        r = O.permute_merge(beta, pc)
        y = rng.normal(size=n)
        emitted = y[beta]
        assert np.array_equal(emitted[r], y[pc])
    with pytest.raises(ValueError):
        O.permute_merge([0, 0, 1], [0, 1, 2])


def test_merged_chain_equals_explicit_gather():
    # producer (N=K_c outputs) -> consumer; merging permutes producer rows
    Wp, ap = synth.layer_weights(200, 96, 31)
    Wc, ac = synth.layer_weights(40, 200, 32)
    P = O.pack_layer(Wp, ap, 3.0)
    C = O.pack_layer(Wc, ac, 3.0)
    _, x = synth.activations(ap, 2, 31)
    y_p = O.linear(P, x)                       # natural basis
    y_c = O.linear(C, y_p)                     # gather = perm
    Pm = O.permute_rows(P, C["perm"])
    r = O.permute_merge(Pm["out_perm"], C["perm"])
    assert np.array_equal(r, np.arange(200))   # merged: identity gather
    y_pm = O.linear(Pm, x)
    assert np.array_equal(y_pm, y_p[:, C["perm"]])
    y_cm = O.linear(C, y_pm, gather=r)
    assert np.array_equal(y_cm, y_c)
    # codes move with their rows, bit for bit
    assert np.array_equal(O.unpack_codes(Pm), O.unpack_codes(P)[C["perm"]])


# --------------------------------------------------------------------------
# P9: reorder-traffic model against the paper's printed totals
# --------------------------------------------------------------------------
def test_reorder_traffic_matches_paper():
    with open(os.path.join(GOLDEN, "paper_values.json")) as f:
        g = json.load(f)
    pv = g["reorder_traffic_no_merge_mib"]
    shapes = g["model_shapes"]
    for model in ("Llama2-13B", "Qwen3-32B"):
        sh = shapes[model]
        lin = [("q", sh["q"], sh["hidden"]), ("k", sh["kv"], sh["hidden"]),
               ("v", sh["kv"], sh["hidden"]), ("o", sh["hidden"], sh["q"]),
               ("gate", sh["ffn"], sh["hidden"]), ("up", sh["ffn"], sh["hidden"]),
               ("down", sh["hidden"], sh["ffn"])]
        mib = O.reorder_traffic_bytes([k for _, _, k in lin], sh["layers"]) / 2 ** 20
        assert round(mib, pv["printed_decimals"]) == pv[model]


def test_w3_overhead_table():
    with open(os.path.join(GOLDEN, "paper_values.json")) as f:
        g = json.load(f)["w3_overhead_percent"]
    for model in ("Falcon-H1-3B", "Llama2-13B", "Qwen3-32B"):
        v = g[model]
        assert round(100 * (3 / v["B_min"] - 1), 1) == v["overhead"]


# --------------------------------------------------------------------------
# decode-step glue and the merged decoder layer (R11)
# --------------------------------------------------------------------------
def test_rmsnorm_closed_forms():
    for c in (3.0, -0.25, 1e3):
        v = O.rmsnorm(np.full(7, c), eps=1e-6)
        assert np.allclose(v, np.sign(c) / np.sqrt(1.0 + 1e-6 / (c * c)), rtol=0, atol=1e-15)
    s = np.random.default_rng(0).standard_normal((3, 50))
    r = O.rmsnorm(s, eps=0.0)
    assert np.allclose(np.mean(r * r, axis=-1), 1.0, atol=1e-13)        # unit mean square
    assert np.allclose(O.rmsnorm(5.5 * s, eps=0.0), r, atol=1e-13)       # scale invariant


def test_silu_identities():
    assert O.silu(0.0) == 0.0
    x = np.linspace(-8, 8, 33)
    assert np.allclose(O.silu(x) - O.silu(-x), x, atol=1e-13)           # x*(s(x)+s(-x)) = x
    assert abs(O.silu(40.0) - 40.0) < 1e-12
    assert abs(O.silu(1.0) - 1.0 / (1.0 + np.exp(-1.0))) < 1e-15


def _small_layer_set(hidden, ffn, seed, bits16=False):
    lin = {}
    for i, (name, N, K) in enumerate(O.llama_layer_linears(hidden, ffn)):
        W, a = synth.layer_weights(N, K, seed + i)
        bits = np.full(K, 16) if bits16 else None
        lin[name] = O.pack_layer(W, a, 3.0, bits=bits)
    return lin


def test_merged_layer_equals_unmerged():
    lin = _small_layer_set(64, 160, 300)
    s = np.random.default_rng(1).standard_normal((2, 64))
    merged = O.merge_decoder_layer(lin)
    plain = {n: (L, L["perm"]) for n, L in lin.items()}
    s_m, mid_m = O.decode_layer(s, merged)
    s_p, mid_p = O.decode_layer(s, plain)
    assert np.allclose(s_m, s_p, rtol=1e-12, atol=1e-12)
    # v and gate/up come out permuted into o's and down's input orders
    assert np.allclose(mid_m["v"], mid_p["v"][:, lin["o"]["perm"]], rtol=1e-12, atol=0)
    assert np.allclose(mid_m["gate"], mid_p["gate"][:, lin["down"]["perm"]], rtol=1e-12, atol=0)


def test_decoder_layer_matches_dense_graph():
    # all-16-bit weights: the layer's weights are fp16(W) in natural order, so
    # the step is the plain dense graph written out with matmuls
    hidden, ffn, seed = 48, 96, 310
    lin = _small_layer_set(hidden, ffn, seed, bits16=True)
    Wd = {}
    for i, (name, N, K) in enumerate(O.llama_layer_linears(hidden, ffn)):
        W, _ = synth.layer_weights(N, K, seed + i)
        Wd[name] = W.astype(np.float16).astype(np.float64)
    s = np.random.default_rng(2).standard_normal((1, hidden)) * 3.0
    out, _ = O.decode_layer(s, O.merge_decoder_layer(lin))

    def bf16(v):
        return O.bf16_rn(v)

    def rms(v):
        return v / np.sqrt(np.mean(v * v, axis=-1, keepdims=True) + 1e-6)

    h = bf16(rms(s))
    v = h @ Wd["v"].T
    s1 = s + bf16(v) @ Wd["o"].T
    h2 = bf16(rms(s1))
    g = h2 @ Wd["gate"].T
    u = h2 @ Wd["up"].T
    ref = s1 + bf16(g / (1 + np.exp(-g)) * u) @ Wd["down"].T
    assert np.allclose(out, ref, rtol=1e-12, atol=1e-12)


def test_row_slice_of_stacked_layer():
    # a stack allocated jointly, split by rows, multiplies like the stack
    W1, a = synth.layer_weights(40, 96, 320)
    W2, _ = synth.layer_weights(24, 96, 321)
    Ls = O.pack_layer(np.vstack([W1, W2]), a, 3.0)
    x = np.random.default_rng(3).standard_normal((2, 96))
    y = O.linear(Ls, x)
    assert np.array_equal(O.linear(O.row_slice(Ls, 0, 40), x), y[:, :40])
    assert np.array_equal(O.linear(O.row_slice(Ls, 40, 64), x), y[:, 40:])


@pytest.mark.parametrize("N,K,seed", [(9, 333, 21), (3, 1, 22), (17, 700, 23)])
def test_dense_layer_equals_the_packed_route(N, K, seed):
    # the direct quantise-dequantise route and the bitstream round trip give
    # the same W' bit for bit (all five widths, ragged blocks)
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed, widths=(2, 3, 4, 8, 16)[: min(5, K)])
    L = O.pack_layer(W, a, 3.0, bits=bits)
    D = O.dense_layer(W, bits)
    assert np.array_equal(D["perm"], L["perm"])
    assert np.array_equal(D["Wd"], O.dequant(L))
    _, x = synth.activations(a, 2, seed)
    assert np.array_equal(O.linear(D, x), O.linear(L, x))
    rp = np.random.default_rng(seed).permutation(N)
    assert np.array_equal(O.permute_rows(D, rp)["Wd"], O.dequant(O.permute_rows(L, rp)))
    assert np.array_equal(O.row_slice(D, 1, N)["Wd"], O.dequant(O.row_slice(L, 1, N)))


@pytest.mark.parametrize("seed", range(3))
def test_dense_layer_brute_force_small(seed):
    # K <= 16: one group per width, quantised straight from W in original
    # channel order, then placed at each channel's clustered position
    rng = np.random.default_rng(100 + seed)
    K = int(rng.integers(2, 17))
    N = int(rng.integers(1, 5))
    W = rng.normal(0, 0.3, size=(N, K)).astype(np.float32)
    bits = rng.choice([2, 3, 4, 8, 16], size=K)
    D = O.dense_layer(W, bits)
    pos = np.empty(K, np.int64)
    pos[D["perm"]] = np.arange(K)
    for n in range(N):
        for b in set(bits.tolist()):
            ks = [k for k in range(K) if bits[k] == b]
            if b == 16:
                want = [float(np.float16(W[n, k])) for k in ks]
            else:
                s, z, q = O.quantize_group(W[n, ks].astype(np.float64), b)
                want = [(qi - z) * s for qi in q]
            assert [D["Wd"][n, pos[k]] for k in ks] == want


def test_decode_layer_on_dense_layers_equals_packed():
    lin = _small_layer_set(64, 160, 330)
    dense = {}
    for i, (name, N, K) in enumerate(O.llama_layer_linears(64, 160)):
        W, _ = synth.layer_weights(N, K, 330 + i)
        dense[name] = O.dense_layer(W, lin[name]["bits"])
    s = np.random.default_rng(4).standard_normal((1, 64))
    s_p, _ = O.decode_layer(s, O.merge_decoder_layer(lin))
    s_d, _ = O.decode_layer(s, O.merge_decoder_layer(dense))
    assert np.array_equal(s_p, s_d)
