"""GPU parity of the decode GEMV and the code unpacker against the oracle.
All calls go through the C ABI (ctypes binding)."""
import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth
from tests.gpu_util import check_tolerance, make_case, oracle_layer, oracle_rows

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _dev(polyq_lib, W, a, B, bits=None, gather=None, identity=False):
    host = polyq_lib.HostLayer.pack(W, a, B, forced_bits=bits)
    return host, polyq_lib.DeviceLayer(host, "cuda", gather=gather, identity_gather=identity)


def _x_dev(xb):
    return torch.from_numpy(xb.view(np.int16)).cuda().view(torch.bfloat16)


@pytest.mark.parametrize("N,K,B,seed,forced", [
    (2048, 2048, 3.0, 1001, False),
    (37, 1000, 3.0, 3, True),
    (8, 16, 3.0, 4, True),
    (130, 4099, 4.5, 5, True),
])
def test_unpack_codes_bit_exact(polyq_lib, N, K, B, seed, forced):
    W, a, bits, _, _ = make_case(N, K, B, seed, forced)
    host, dev = _dev(polyq_lib, W, a, B, bits)
    ref = oracle_layer(W, a, B, bits)
    assert np.array_equal(dev.perm, ref["perm"].astype(np.int32))
    got = polyq_lib.unpack_codes(dev)
    assert np.array_equal(got.astype(np.int64), O.unpack_codes(ref))


@pytest.mark.parametrize("batch", [1, 2, 3, 4])
@pytest.mark.parametrize("N,K,B,seed,forced", [
    (2048, 2048, 3.0, 1001, False),   # 2048 x 2048 at B = 3.0
    (300, 5120, 4.5, 2002, False),
    (61, 3001, 3.0, 7, True),         # all five widths, ragged blocks
    (8, 16, 3.0, 8, True),            # tiny
    (5, 1, 16.0, 9, False),           # a single channel
    (257, 700, 2.0, 10, False),       # all 2-bit
    (64, 640, 16.0, 11, False),       # all 16-bit
])
def test_gemv_matches_oracle(polyq_lib, batch, N, K, B, seed, forced):
    W, a, bits, xb, x = make_case(N, K, B, seed, forced, batch)
    host, dev = _dev(polyq_lib, W, a, B, bits)
    ref = oracle_layer(W, a, B, bits)
    y = polyq_lib.linear_gemv(dev, _x_dev(xb))
    torch.cuda.synchronize()
    check_tolerance(y.cpu().numpy(), O.linear(ref, x), x, K)


def test_gemv_residual_and_identity_gather(polyq_lib):
    W, a, bits, xb, x = make_case(500, 1500, 3.0, 12, True, 2)
    ref = oracle_layer(W, a, 3.0, bits)
    # merged edge: x already in the clustered basis, gather = identity
    xs_bits = xb[:, ref["perm"]]
    host, dev = _dev(polyq_lib, W, a, 3.0, bits, identity=True)
    res = torch.randn(2, 500, device="cuda")
    y = polyq_lib.linear_gemv(dev, _x_dev(np.ascontiguousarray(xs_bits)), residual=res)
    torch.cuda.synchronize()
    yref = O.linear(ref, x) + res.cpu().numpy().astype(np.float64)
    check_tolerance(y.cpu().numpy(), yref, x, 1500)
    # in-place residual (y aliases residual); split tiles add their pieces
    # atomically, so agreement is to fp32 rounding
    res2 = res.clone()
    polyq_lib.linear_gemv(dev, _x_dev(np.ascontiguousarray(xs_bits)), y=res2, residual=res2)
    torch.cuda.synchronize()
    assert torch.allclose(res2, y, rtol=1e-5, atol=1e-5 * float(y.abs().max()))


def test_gemv_merged_rows_match_unmerged(polyq_lib):
    """Section 4.3: producer rows permuted by the consumer's perm emit the
    consumer's basis; outputs equal the unmerged outputs gathered.  Rows of a
    tile whose K range is split over CTAs sum their pieces in a different
    association, so equality is to fp32 rounding, not bitwise."""
    Wp, ap, _, xb, x = make_case(900, 640, 3.0, 13, False, 1)
    host = polyq_lib.HostLayer.pack(Wp, ap, 3.0)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    y = polyq_lib.linear_gemv(dev, _x_dev(xb)).cpu().numpy()
    cperm = np.random.default_rng(0).permutation(900)
    host.permute_rows(cperm)
    devm = polyq_lib.DeviceLayer(host, "cuda")
    ym = polyq_lib.linear_gemv(devm, _x_dev(xb)).cpu().numpy()
    ref = y[:, cperm]
    assert np.max(np.abs(ym - ref)) <= 1e-5 * np.max(np.abs(ref))


@pytest.mark.parametrize("name,N,K,B,batch", [
    ("llama-q", 5120, 5120, 3.0, 1),
    ("llama-gate", 13824, 5120, 3.0, 1),
    ("llama-down", 5120, 13824, 4.5, 1),
    ("qwen-q", 8192, 5120, 5.0, 1),
    ("qwen-kv", 1024, 5120, 3.5, 4),
    ("qwen-o", 5120, 8192, 4.0, 1),
    ("qwen-gate", 25600, 5120, 3.0, 4),
    ("qwen-down", 5120, 25600, 6.0, 4),
])
def test_gemv_full_size_sampled_rows(polyq_lib, name, N, K, B, batch):
    """Full-size layers in the benchmark's launch configuration; the oracle
    recomputes a sample of output rows."""
    seed = 7000 + N + K
    W, a = synth.layer_weights(N, K, seed)
    xb, x = synth.activations(a, batch, seed)
    host, dev = _dev(polyq_lib, W, a, B)
    y = polyq_lib.linear_gemv(dev, _x_dev(xb))
    torch.cuda.synchronize()
    rows = np.unique(np.concatenate([[0, N - 1], np.random.default_rng(1).integers(0, N, 60)]))
    ref, bits_full = oracle_rows(W, a, B, rows)
    assert np.array_equal(host.export()["bits"], bits_full.astype(np.uint8))
    check_tolerance(y.cpu().numpy()[:, rows], O.linear(ref, x), x, K)


@pytest.mark.parametrize("batch", [1, 4])
def test_gemv_residual_not_16_byte_aligned(polyq_lib, batch):
    """The outputs are set to the residual by CTAs of the pre-pass with
    16-byte loads and stores where the pointers allow; a residual at a 4-byte
    offset takes the scalar path."""
    N, K = 200, 1024
    W, a = synth.layer_weights(N, K, 37)
    host = polyq_lib.HostLayer.pack(W, a, 3.0)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    ref = O.pack_layer(W, a, 3.0)
    xb, x = synth.activations(a, batch, 37)
    res = torch.randn(batch * N + 1, device="cuda")[1:].view(batch, N)
    assert res.data_ptr() % 16 != 0
    y = polyq_lib.linear_gemv(dev, _x_dev(xb), residual=res)
    torch.cuda.synchronize()
    check_tolerance(y.cpu().numpy(), O.linear(ref, x) + res.cpu().numpy().astype(np.float64), x, K)


@pytest.mark.parametrize("batch", [1, 4])
def test_gemv_group_matches_oracle(polyq_lib, batch):
    """Several layers in one launch (q/k/v-like: shared input, own widths and
    gathers; plus a layer of another shape and forced widths)."""
    K = 1536
    specs = [(640, 3.0, 31, False), (256, 3.5, 32, False), (256, 4.5, 33, True), (130, 3.0, 34, True)]
    layers, refs, xs = [], [], []
    _, a0 = synth.layer_weights(8, K, 30)
    xb, x = synth.activations(a0, batch, 30)
    for N, B, seed, forced in specs:
        W, a = synth.layer_weights(N, K, seed)
        bits = synth.random_codes_layer_bits(K, seed) if forced else None
        host = polyq_lib.HostLayer.pack(W, a, B, forced_bits=bits)
        layers.append(polyq_lib.DeviceLayer(host, "cuda"))
        refs.append(O.pack_layer(W, a, B, bits=bits))
    xt = _x_dev(xb)
    res = [None, torch.randn(batch, 256, device="cuda"), None, None]
    ys = polyq_lib.linear_gemv_group(layers, [xt] * 4, residuals=res)
    torch.cuda.synchronize()
    for i, (y, ref) in enumerate(zip(ys, refs)):
        yref = O.linear(ref, x)
        if res[i] is not None:
            yref = yref + res[i].cpu().numpy().astype(np.float64)
        check_tolerance(y.cpu().numpy(), yref, x, K)
    with pytest.raises(polyq_lib.PolyqError):  # at most POLYQ_MAX_GROUP = 8 layers
        polyq_lib.linear_gemv_group(layers * 2 + layers[:1], [xt] * 9)


@pytest.mark.parametrize("batch", [1, 3])
def test_gemv_group_of_seven_layers_with_own_inputs(polyq_lib, batch):
    """The seven linears of a decoder layer (scaled down) in one launch, each
    reading its own activation."""
    hidden, ffn = 384, 1024
    layers, refs, xs, xts = [], [], [], []
    for i, (name, N, K) in enumerate(O.llama_layer_linears(hidden, ffn)):
        W, a = synth.layer_weights(N, K, 400 + i)
        bits = synth.random_codes_layer_bits(K, 400 + i) if i % 3 == 0 else None
        host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
        layers.append(polyq_lib.DeviceLayer(host, "cuda"))
        refs.append(O.pack_layer(W, a, 3.0, bits=bits))
        xb, x = synth.activations(a, batch, 410 + i)
        xs.append(x)
        xts.append(_x_dev(xb))
    ys = polyq_lib.linear_gemv_group(layers, xts)
    torch.cuda.synchronize()
    for y, ref, x in zip(ys, refs, xs):
        check_tolerance(y.cpu().numpy(), O.linear(ref, x), x, x.shape[1])


def _scaled_bf16(x, f):
    """bf16 bits of x * f for a power of two f (exact for bf16 x in range)."""
    xs = x * f
    bits = synth.bf16_bits(xs.astype(np.float32))
    assert np.array_equal(synth.bf16_to_f64(bits), xs)
    return bits, xs


@pytest.mark.parametrize("batch", [1, 4])
@pytest.mark.parametrize("scale_exp", [-40, -12, -8, 4, 10, 40])
def test_gemv_meets_tolerance_at_any_activation_scale(polyq_lib, batch, scale_exp):
    """The tolerance is relative, so it must hold whatever the activations'
    absolute scale: the record builder scales each chunk by a power of two
    before rounding to fp16.  All five widths, ragged blocks."""
    W, a, bits, xb, x = make_case(200, 3001, 3.0, 17, True, batch)
    xsb, xs = _scaled_bf16(x, 2.0 ** scale_exp)
    host, dev = _dev(polyq_lib, W, a, 3.0, bits)
    ref = oracle_layer(W, a, 3.0, bits)
    y = polyq_lib.linear_gemv(dev, _x_dev(xsb))
    torch.cuda.synchronize()
    check_tolerance(y.cpu().numpy(), O.linear(ref, xs), xs, 3001)


@pytest.mark.parametrize("batch", [1, 3])
def test_gemv_chunks_of_very_different_magnitude(polyq_lib, batch):
    """Channels whose magnitudes differ by 2^24 inside one layer: each
    64-channel chunk (and each 16-bit step) gets its own exponent."""
    W, a, bits, xb, x = make_case(130, 2500, 3.0, 18, True, batch)
    f = np.where(np.arange(2500) % 3 == 0, 2.0 ** 12, 2.0 ** -12)
    xsb, xs = _scaled_bf16(x, f[None, :])
    host, dev = _dev(polyq_lib, W, a, 3.0, bits)
    ref = oracle_layer(W, a, 3.0, bits)
    y = polyq_lib.linear_gemv(dev, _x_dev(xsb))
    torch.cuda.synchronize()
    check_tolerance(y.cpu().numpy(), O.linear(ref, xs), xs, 2500)
