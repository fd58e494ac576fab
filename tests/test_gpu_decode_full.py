"""Decode-step parity at the full Llama2-13B width (hidden 5120, FFN 13824,
B = 3.0): two decoder layers run through polyq_linear_gemv_input with the
RMSNorm and SiLU * up glue fused into the pre-pass and the Section 4.3 merges
(v -> o, gate/up -> down), in both merge modes:

* separate: every linear allocated on its own;
* grouped: q/k/v and gate/up each allocated jointly over their stacked rows.

Checks, each against the oracle:
* every linear on sampled output rows, with the oracle fed the GPU's actual
  bf16 input (the relative tolerance of the GEMV tests);
* the fused glue on the full vectors (RMSNorm over 5120 channels, SiLU * up
  over 13824) within one bf16 step of the fp64 value of the GPU's own input;
* (separate mode) the stream after both layers against the oracle's own
  chain from the same start, rel-L2 <= 1e-2: bf16 rounding points may fall on
  the other side between fp32 and fp64, and such flips compound."""
import functools

import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth
from tests.gpu_util import check_tolerance

torch = pytest.importorskip("torch")
pytestmark = [pytest.mark.gpu, pytest.mark.slow]

HIDDEN, FFN, LAYERS, B = 5120, 13824, 2, 3.0
NAMES = [n for n, _, _ in O.llama_layer_linears(HIDDEN, FFN)]


@functools.lru_cache(maxsize=None)
def _weights(layer):
    return {name: synth.layer_weights(N, K, synth.seed_for(5, 10 * layer + i))
            for i, (name, N, K) in enumerate(O.llama_layer_linears(HIDDEN, FFN))}


def _bf16_bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def _bf16_vals(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _ulps(got_bits, want):
    return np.abs(got_bits.astype(np.int64) - synth.bf16_bits(want).astype(np.int64))


def _glue_ok(got_bits, want):
    d = _ulps(got_bits, want)
    assert d.max() <= 1 and (d == 0).mean() > 0.99


class _Linear:
    """One linear as the library runs it: the weights it was packed from, its
    width map, its row permutation (emitted output i = original row
    rows[i]) and its input gather (None: identity)."""

    def __init__(self, W, bits, rows, gather):
        self.W, self.bits, self.rows, self.gather = W, bits, rows, gather

    def check(self, y_gpu, x_in, n_sample=64, seed=0):
        N, K = self.W.shape
        rng = np.random.default_rng(seed)
        idx = np.unique(np.concatenate([[0, N - 1], rng.integers(0, N, n_sample)]))
        D = O.dense_layer(self.W[self.rows[idx]], self.bits)
        g = np.arange(K) if self.gather is None else self.gather
        check_tolerance(y_gpu[:, idx], O.linear(D, x_in, gather=g), x_in, K)


def _build(polyq_lib, layer, mode):
    """Library device layers and the matching oracle descriptions."""
    w = _weights(layer)
    h = {}
    if mode == "separate":
        for n in NAMES:
            h[n] = polyq_lib.HostLayer.pack(*w[n], B)
        p_o = h["o"].export()["perm"]
        p_d = h["down"].export()["perm"]
        h["v"].permute_rows(p_o)
        h["gate"].permute_rows(p_d)
        h["up"].permute_rows(p_d)
        dev = {n: polyq_lib.DeviceLayer(h[n], "cuda", identity_gather=n in ("o", "down"))
               for n in NAMES}
        lin = {}
        for n in NAMES:
            ex = h[n].export()
            bits = O.allocate_bits(O.saliency(*w[n]), B)
            assert np.array_equal(ex["bits"], bits.astype(np.uint8))
            rows = ex["out_perm"].astype(np.int64)
            lin[n] = _Linear(w[n][0], bits, rows, None if n in ("o", "down") else ex["perm"])
        return dev, lin
    # grouped: q/k/v share one allocation and permutation, gate/up another
    Wqkv = np.vstack([w["q"][0], w["k"][0], w["v"][0]])
    Wgu = np.vstack([w["gate"][0], w["up"][0]])
    aq, ag = w["q"][1], w["gate"][1]
    hq = polyq_lib.HostLayer.pack(Wqkv, aq, B)
    hg = polyq_lib.HostLayer.pack(Wgu, ag, B)
    ho = polyq_lib.HostLayer.pack(*w["o"], B)
    hd = polyq_lib.HostLayer.pack(*w["down"], B)
    p_o, p_d = ho.export()["perm"], hd.export()["perm"]
    hq.permute_rows(np.concatenate([np.arange(2 * HIDDEN), 2 * HIDDEN + p_o]))
    hg.permute_rows(np.concatenate([p_d, FFN + p_d]))
    dev = {"qkv": polyq_lib.DeviceLayer(hq, "cuda"), "gu": polyq_lib.DeviceLayer(hg, "cuda"),
           "o": polyq_lib.DeviceLayer(ho, "cuda", identity_gather=True),
           "down": polyq_lib.DeviceLayer(hd, "cuda", identity_gather=True)}
    lin = {}
    for key, Wm, a in (("qkv", Wqkv, aq), ("gu", Wgu, ag), ("o", *w["o"]),
                       ("down", *w["down"])):
        ex = {"qkv": hq, "gu": hg, "o": ho, "down": hd}[key].export()
        bits = O.allocate_bits(O.saliency(Wm, a), B)
        assert np.array_equal(ex["bits"], bits.astype(np.uint8))
        lin[key] = _Linear(Wm, bits, ex["out_perm"].astype(np.int64),
                           None if key in ("o", "down") else ex["perm"])
    return dev, lin


def _run_layer(polyq_lib, dev, mode, s, ws):
    """One decoder layer on the GPU (four calls); returns its intermediates."""
    L = polyq_lib
    out = {"s0": s.clone()}
    h = torch.empty((1, HIDDEN), dtype=torch.bfloat16, device="cuda")
    if mode == "separate":
        q, k, v = L.linear_gemv_input([dev["q"], dev["k"], dev["v"]], L.X_RMSNORM, s, eps=1e-6,
                                      x_out=h, workspace=ws)
        out.update(q=q, k=k, v=v)
    else:
        qkv, = L.linear_gemv_input([dev["qkv"]], L.X_RMSNORM, s, eps=1e-6, x_out=h, workspace=ws)
        out["qkv"] = qkv
        v = qkv[:, 2 * HIDDEN:]
    xo = torch.empty((1, HIDDEN), dtype=torch.bfloat16, device="cuda")
    L.linear_gemv_input([dev["o"]], L.X_F32, v.contiguous(), ys=[s], residuals=[s], x_out=xo,
                        workspace=ws)
    out["s1"] = s.clone()
    h2 = torch.empty((1, HIDDEN), dtype=torch.bfloat16, device="cuda")
    if mode == "separate":
        g, u = L.linear_gemv_input([dev["gate"], dev["up"]], L.X_RMSNORM, s, eps=1e-6,
                                   x_out=h2, workspace=ws)
        out.update(gate=g, up=u)
    else:
        gu, = L.linear_gemv_input([dev["gu"]], L.X_RMSNORM, s, eps=1e-6, x_out=h2, workspace=ws)
        out["gu"] = gu
        g, u = gu[:, :FFN].contiguous(), gu[:, FFN:].contiguous()
    xd = torch.empty((1, FFN), dtype=torch.bfloat16, device="cuda")
    L.linear_gemv_input([dev["down"]], L.X_SILU_MUL, g, b=u, ys=[s], residuals=[s], x_out=xd,
                        workspace=ws)
    torch.cuda.synchronize()
    out.update(h=h, xo=xo, h2=h2, xd=xd, v_=v, g_=g, u_=u, s2=s.clone())
    return {k: v.cpu().numpy() if v.dtype != torch.bfloat16 else _bf16_bits(v)
            for k, v in out.items()}


@pytest.mark.parametrize("mode", ["separate", "grouped"])
def test_decode_step_full_width(polyq_lib, mode):
    s0 = np.random.default_rng(55).standard_normal((1, HIDDEN)).astype(np.float32)
    s = torch.from_numpy(s0).cuda()
    ws = torch.zeros(1 << 22, dtype=torch.uint8, device="cuda")
    for layer in range(LAYERS):
        dev, lin = _build(polyq_lib, layer, mode)
        r = _run_layer(polyq_lib, dev, mode, s, ws)
        del dev
        hx, xox, h2x, xdx = (_bf16_vals(r[k]) for k in ("h", "xo", "h2", "xd"))
        # the fused glue, on the GPU's own inputs, over the full vectors
        _glue_ok(r["h"], O.rmsnorm(r["s0"].astype(np.float64), 1e-6))
        assert np.array_equal(r["xo"], synth.bf16_bits(r["v_"]))  # fp32 -> bf16, same rounding
        _glue_ok(r["h2"], O.rmsnorm(r["s1"].astype(np.float64), 1e-6))
        g64, u64 = r["g_"].astype(np.float64), r["u_"].astype(np.float64)
        _glue_ok(r["xd"], O.silu(g64) * u64)
        # every linear on sampled rows, fed the GPU's actual input
        if mode == "separate":
            for n, x in (("q", hx), ("k", hx), ("v", hx), ("gate", h2x), ("up", h2x)):
                lin[n].check(r[n], x, seed=layer)
        else:
            lin["qkv"].check(r["qkv"], hx, n_sample=96, seed=layer)
            lin["gu"].check(r["gu"], h2x, n_sample=96, seed=layer)
        # o and down add into the stream in place: their outputs are the
        # stream's increments
        lin["o"].check(r["s1"] - r["s0"], xox, seed=layer)
        lin["down"].check(r["s2"] - r["s1"], xdx, seed=layer)
    if mode != "separate":
        return
    # the oracle's own two-layer chain from the same start
    s_ref = s0.astype(np.float64)
    for layer in range(LAYERS):
        w = _weights(layer)
        dense = {n: O.dense_layer(w[n][0], O.allocate_bits(O.saliency(*w[n]), B)) for n in NAMES}
        s_ref, _ = O.decode_layer(s_ref, O.merge_decoder_layer(dense))
        del dense
    got = s.cpu().numpy().astype(np.float64)
    rel = np.linalg.norm(got - s_ref) / np.linalg.norm(s_ref)
    assert rel <= 1e-2, rel
