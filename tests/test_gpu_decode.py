"""GPU parity of the decode-step path: the input transforms fused into the GEMV
pre-pass, and a two-layer Llama-shaped decode step with the §4.3 merges
(v -> o and gate/up -> down), against the oracle.  All calls go through the
C ABI."""
import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth
from tests.gpu_util import check_tolerance

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _bf16_bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def _bf16_vals(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def _ulp_diff(got_bits, want):
    """bf16 ulps between GPU results and fp64 values rounded to bf16."""
    w = synth.bf16_bits(want)
    return np.abs(got_bits.astype(np.int64) - w.astype(np.int64))


@pytest.mark.parametrize("batch", [1, 3])
@pytest.mark.parametrize("kind", ["bf16", "f32", "rmsnorm", "silu_mul"])
def test_input_transforms(polyq_lib, kind, batch):
    N, K, seed = 200, 1100, 61
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    ref = O.pack_layer(W, a, 3.0, bits=bits)
    rng = np.random.default_rng(seed)
    A = (rng.standard_normal((batch, K)) * 2.0).astype(np.float32)
    Bm = rng.standard_normal((batch, K)).astype(np.float32)
    x_out = torch.empty((batch, K), dtype=torch.bfloat16, device="cuda")
    if kind == "bf16":
        xb = synth.bf16_bits(A.astype(np.float64))
        a_dev = torch.from_numpy(xb.view(np.int16)).cuda().view(torch.bfloat16)
        y, = polyq_lib.linear_gemv_input([dev], polyq_lib.X_BF16, a_dev, x_out=x_out)
        want = _bf16_vals(xb)
    else:
        a_dev = torch.from_numpy(A).cuda()
        b_dev = torch.from_numpy(Bm).cuda() if kind == "silu_mul" else None
        k = {"f32": polyq_lib.X_F32, "rmsnorm": polyq_lib.X_RMSNORM,
             "silu_mul": polyq_lib.X_SILU_MUL}[kind]
        y, = polyq_lib.linear_gemv_input([dev], k, a_dev, b=b_dev, eps=1e-6, x_out=x_out)
        A64 = A.astype(np.float64)
        if kind == "f32":
            want = O.bf16_rn(A64)
        elif kind == "rmsnorm":
            want = O.bf16_rn(O.rmsnorm(A64, 1e-6))
        else:
            want = O.bf16_rn(O.silu(A64) * Bm.astype(np.float64))
    torch.cuda.synchronize()
    got = _bf16_bits(x_out)
    d = _ulp_diff(got, want)
    if kind in ("bf16", "f32"):
        assert d.max() == 0  # the same fp32 value rounded the same way
    else:
        # fp32 on the GPU against fp64 here: a result next to a rounding
        # boundary may land one bf16 step away
        assert d.max() <= 1 and (d == 0).mean() > 0.99
    # the GEMV on the activation the pre-pass actually produced
    x_gpu = _bf16_vals(got)
    check_tolerance(y.cpu().numpy(), O.linear(ref, x_gpu), x_gpu, K)


def _pack_pair(polyq_lib, W, a, seed_bits=None):
    host = polyq_lib.HostLayer.pack(W, a, 3.0)
    ref = O.pack_layer(W, a, 3.0)
    assert np.array_equal(host.export()["perm"], ref["perm"].astype(np.int32))
    return host, ref


def test_two_layer_decode_step(polyq_lib):
    hidden, ffn, n_layers = 256, 640, 2
    names = [n for n, _, _ in O.llama_layer_linears(hidden, ffn)]
    dev_layers, ora_layers = [], []
    for layer in range(n_layers):
        hosts, refs = {}, {}
        for i, (name, N, K) in enumerate(O.llama_layer_linears(hidden, ffn)):
            W, a = synth.layer_weights(N, K, synth.seed_for(5, 10 * layer + i))
            hosts[name], refs[name] = _pack_pair(polyq_lib, W, a)
        merged = O.merge_decoder_layer(refs)
        # the same merges on the library side: v emits in o's basis, gate/up
        # in down's; o and down then read their input without a gather
        o_perm = hosts["o"].export()["perm"]
        d_perm = hosts["down"].export()["perm"]
        hosts["v"].permute_rows(o_perm)
        hosts["gate"].permute_rows(d_perm)
        hosts["up"].permute_rows(d_perm)
        dev = {n: polyq_lib.DeviceLayer(hosts[n], "cuda", identity_gather=n in ("o", "down"))
               for n in names}
        dev_layers.append(dev)
        ora_layers.append(merged)

    rng = np.random.default_rng(5)
    s0 = rng.standard_normal((1, hidden)).astype(np.float32)
    s = torch.from_numpy(s0).cuda()
    ws = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
    s_ref = s0.astype(np.float64)
    for dev, merged in zip(dev_layers, ora_layers):
        h = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
        q, k, v = polyq_lib.linear_gemv_input([dev["q"], dev["k"], dev["v"]], polyq_lib.X_RMSNORM,
                                              s, eps=1e-6, x_out=h, workspace=ws)
        s_before = s.clone()
        xo = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
        polyq_lib.linear_gemv_input([dev["o"]], polyq_lib.X_F32, v, ys=[s], residuals=[s],
                                    x_out=xo, workspace=ws)
        s_mid = s.clone()
        h2 = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
        g, u = polyq_lib.linear_gemv_input([dev["gate"], dev["up"]], polyq_lib.X_RMSNORM, s,
                                           eps=1e-6, x_out=h2, workspace=ws)
        xd = torch.empty((1, ffn), dtype=torch.bfloat16, device="cuda")
        polyq_lib.linear_gemv_input([dev["down"]], polyq_lib.X_SILU_MUL, g, b=u, ys=[s],
                                    residuals=[s], x_out=xd, workspace=ws)
        torch.cuda.synchronize()

        # each linear against the oracle fed the GPU's actual input
        hx, xox, h2x, xdx = (_bf16_vals(_bf16_bits(t)) for t in (h, xo, h2, xd))
        for name, y, x in (("q", q, hx), ("k", k, hx), ("v", v, hx), ("gate", g, h2x),
                           ("up", u, h2x)):
            L, gat = merged[name]
            check_tolerance(y.cpu().numpy(), O.linear(L, x, gather=gat), x, x.shape[1])
        o_ref = O.linear(merged["o"][0], xox, gather=np.arange(hidden))
        check_tolerance((s_mid - s_before).cpu().numpy(), o_ref, xox, hidden)
        d_ref = O.linear(merged["down"][0], xdx, gather=np.arange(ffn))
        check_tolerance((s - s_mid).cpu().numpy(), d_ref, xdx, ffn)
        # the glue itself, from the GPU's previous values
        assert _ulp_diff(_bf16_bits(h), O.rmsnorm(s_before.cpu().numpy().astype(np.float64),
                                                  1e-6)).max() <= 1
        s_ref, _ = O.decode_layer(s_ref, merged)

    # the whole chain against the oracle's chain (bf16 rounding points can
    # flip by one step between fp32 and fp64, and the effect compounds)
    got = s.cpu().numpy().astype(np.float64)
    rel = np.linalg.norm(got - s_ref) / np.linalg.norm(s_ref)
    assert rel <= 1e-2, rel


def test_grouped_decode_layer(polyq_lib):
    # q/k/v and gate/up each allocated jointly over their stacked rows (one
    # permutation per group), v rows merged into o's basis, gate/up rows into
    # down's; the library runs four calls, the oracle the same layer split
    hidden, ffn = 256, 640
    W = {}
    for i, (name, N, K) in enumerate(O.llama_layer_linears(hidden, ffn)):
        W[name] = synth.layer_weights(N, K, synth.seed_for(6, i))
    Wqkv = np.vstack([W["q"][0], W["k"][0], W["v"][0]])
    Wgu = np.vstack([W["gate"][0], W["up"][0]])
    aq, ag = W["q"][1], W["gate"][1]
    h_qkv, r_qkv = polyq_lib.HostLayer.pack(Wqkv, aq, 3.0), O.pack_layer(Wqkv, aq, 3.0)
    h_gu, r_gu = polyq_lib.HostLayer.pack(Wgu, ag, 3.0), O.pack_layer(Wgu, ag, 3.0)
    h_o, r_o = polyq_lib.HostLayer.pack(*W["o"], 3.0), O.pack_layer(*W["o"], 3.0)
    h_d, r_d = polyq_lib.HostLayer.pack(*W["down"], 3.0), O.pack_layer(*W["down"], 3.0)
    p_o, p_d = r_o["perm"], r_d["perm"]
    rp_qkv = np.concatenate([np.arange(2 * hidden), 2 * hidden + p_o])
    rp_gu = np.concatenate([p_d, ffn + p_d])
    h_qkv.permute_rows(rp_qkv)
    h_gu.permute_rows(rp_gu)
    r_qkv = O.permute_rows(r_qkv, rp_qkv)
    r_gu = O.permute_rows(r_gu, rp_gu)
    merged = {"q": (O.row_slice(r_qkv, 0, hidden), r_qkv["perm"]),
              "k": (O.row_slice(r_qkv, hidden, 2 * hidden), r_qkv["perm"]),
              "v": (O.row_slice(r_qkv, 2 * hidden, 3 * hidden), r_qkv["perm"]),
              "o": (r_o, None),
              "gate": (O.row_slice(r_gu, 0, ffn), r_gu["perm"]),
              "up": (O.row_slice(r_gu, ffn, 2 * ffn), r_gu["perm"]),
              "down": (r_d, None)}
    d_qkv = polyq_lib.DeviceLayer(h_qkv, "cuda")
    d_gu = polyq_lib.DeviceLayer(h_gu, "cuda")
    d_o = polyq_lib.DeviceLayer(h_o, "cuda", identity_gather=True)
    d_d = polyq_lib.DeviceLayer(h_d, "cuda", identity_gather=True)

    s0 = np.random.default_rng(6).standard_normal((1, hidden)).astype(np.float32)
    s = torch.from_numpy(s0).cuda()
    h = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
    yqkv, = polyq_lib.linear_gemv_input([d_qkv], polyq_lib.X_RMSNORM, s, x_out=h)
    xo = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
    polyq_lib.linear_gemv_input([d_o], polyq_lib.X_F32, yqkv[:, 2 * hidden:], ys=[s],
                                residuals=[s], x_out=xo)
    h2 = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
    ygu, = polyq_lib.linear_gemv_input([d_gu], polyq_lib.X_RMSNORM, s, x_out=h2)
    xd = torch.empty((1, ffn), dtype=torch.bfloat16, device="cuda")
    polyq_lib.linear_gemv_input([d_d], polyq_lib.X_SILU_MUL, ygu[:, :ffn], b=ygu[:, ffn:],
                                ys=[s], residuals=[s], x_out=xd)
    torch.cuda.synchronize()
    hx, h2x = _bf16_vals(_bf16_bits(h)), _bf16_vals(_bf16_bits(h2))
    y = yqkv.cpu().numpy()
    for name, sl in (("q", slice(0, hidden)), ("k", slice(hidden, 2 * hidden)),
                     ("v", slice(2 * hidden, 3 * hidden))):
        L, gat = merged[name]
        check_tolerance(y[:, sl], O.linear(L, hx, gather=gat), hx, hidden)
    g = ygu.cpu().numpy()
    check_tolerance(g[:, :ffn], O.linear(*merged["gate"][:1], h2x, gather=merged["gate"][1]),
                    h2x, hidden)
    s_ref, _ = O.decode_layer(s0.astype(np.float64), merged)
    got = s.cpu().numpy().astype(np.float64)
    assert np.linalg.norm(got - s_ref) / np.linalg.norm(s_ref) <= 1e-2


@pytest.mark.parametrize("kind", ["bf16", "f32", "rmsnorm", "silu_mul"])
@pytest.mark.parametrize("K", [1100, 1101])
def test_in_place_call_with_every_input_kind(polyq_lib, kind, K):
    """Batch 1 with every output accumulated in place (y aliases its
    residual), for each fused input kind, on a row width that is and one that
    is not a multiple of 4.  Three layers of different shapes and widths
    share the input; the results must match the oracle fed the GPU's own
    transformed input (x_out), and a second call must add the product again."""
    rng = np.random.default_rng(K)
    specs = [(200, 3.0, 71, True), (130, 4.5, 72, False), (64, 2.0, 73, False)]
    devs, refs = [], []
    for N, B, seed, forced in specs:
        W, a = synth.layer_weights(N, K, seed)
        bits = synth.random_codes_layer_bits(K, seed) if forced else None
        host = polyq_lib.HostLayer.pack(W, a, B, forced_bits=bits)
        devs.append(polyq_lib.DeviceLayer(host, "cuda"))
        refs.append(O.pack_layer(W, a, B, bits=bits))
    A = (rng.standard_normal((1, K)) * 2.0).astype(np.float32)
    Bm = rng.standard_normal((1, K)).astype(np.float32)
    if kind == "bf16":
        a_dev = torch.from_numpy(synth.bf16_bits(A.astype(np.float64)).view(np.int16)).cuda()
        a_dev = a_dev.view(torch.bfloat16)
    else:
        a_dev = torch.from_numpy(A).cuda()
    b_dev = torch.from_numpy(Bm).cuda() if kind == "silu_mul" else None
    k = {"bf16": polyq_lib.X_BF16, "f32": polyq_lib.X_F32, "rmsnorm": polyq_lib.X_RMSNORM,
         "silu_mul": polyq_lib.X_SILU_MUL}[kind]
    y0 = [torch.randn(1, N, device="cuda") for N, _, _, _ in specs]
    ys = [y.clone() for y in y0]
    x_out = torch.empty((1, K), dtype=torch.bfloat16, device="cuda")
    polyq_lib.linear_gemv_input(devs, k, a_dev, b=b_dev, eps=1e-6, ys=ys, residuals=ys,
                                x_out=x_out)
    torch.cuda.synchronize()
    x = _bf16_vals(_bf16_bits(x_out))
    if kind == "bf16":
        assert np.array_equal(_bf16_bits(x_out), _bf16_bits(a_dev))
    for y, y_init, ref in zip(ys, y0, refs):
        want = O.linear(ref, x) + y_init.cpu().numpy().astype(np.float64)
        check_tolerance(y.cpu().numpy(), want, x, K)
    # the same call again accumulates once more: y = y0 + 2 W x
    polyq_lib.linear_gemv_input(devs, k, a_dev, b=b_dev, eps=1e-6, ys=ys, residuals=ys)
    torch.cuda.synchronize()
    for y, y_init, ref in zip(ys, y0, refs):
        want = 2.0 * O.linear(ref, x) + y_init.cpu().numpy().astype(np.float64)
        check_tolerance(y.cpu().numpy(), want, x, K)


@pytest.mark.parametrize("scale_exp", [-40, -10, 12, 40])
def test_in_place_at_any_activation_scale(polyq_lib, scale_exp):
    W, a = synth.layer_weights(300, 3001, 74)
    bits = synth.random_codes_layer_bits(3001, 74)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    ref = O.pack_layer(W, a, 3.0, bits=bits)
    _, x = synth.activations(a, 1, 74)
    xs = x * 2.0 ** scale_exp
    xb = synth.bf16_bits(xs.astype(np.float32))
    assert np.array_equal(synth.bf16_to_f64(xb), xs)
    y = torch.zeros(1, 300, device="cuda")
    polyq_lib.linear_gemv(dev, torch.from_numpy(xb.view(np.int16)).cuda().view(torch.bfloat16),
                          y=y, residual=y)
    torch.cuda.synchronize()
    check_tolerance(y.cpu().numpy(), O.linear(ref, xs), xs, 3001)
