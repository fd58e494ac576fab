"""GPU parity for layers packed with the Section 3.3 quanta matching and the
Section 3.4 activation factors: the GEMV (plain and with a fused input
transform) and the GEMM against the oracle, through the C ABI."""
import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth
from tests.gpu_util import check_tolerance

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _x_dev(xb):
    return torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).cuda().view(torch.bfloat16)


def _x2(a):
    return np.asarray(a, np.float32).astype(np.float64) ** 2


def _scaled_pair(polyq_lib, W, a, B, bits=None):
    """Library layer (quantiser proxy, quanta, scaling) and the oracle's."""
    if bits is None:
        host = polyq_lib.HostLayer.pack(W, a, B, proxy=polyq_lib.PROXY_QUANT, snap_quanta=True,
                                        act_scaling=True)
        E = O.quant_error_table(W, _x2(a))
        bits = O.snap_to_quanta(O.allocate_from_table(E, B), E, B)
    else:
        host = polyq_lib.HostLayer.pack(W, a, B, forced_bits=bits, act_scaling=True)
    _, t = O.choose_alphas(W, bits, a, _x2(a))
    ref = O.pack_layer_scaled(W, bits, t)
    assert np.array_equal(host.xscale(), ref["xscale"].astype(np.float32))
    return host, ref


@pytest.mark.parametrize("batch", [1, 3, 4])
@pytest.mark.parametrize("N,K,B,seed,forced", [
    (2048, 2048, 3.0, 1000, False),   # the 2048 x 2048 layer at B = 3
    (61, 3001, 3.0, 7, True),         # all five widths, ragged blocks
    (130, 1024, 4.5, 8, False),
])
def test_scaled_gemv_matches_oracle(polyq_lib, batch, N, K, B, seed, forced):
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed) if forced else None
    host, ref = _scaled_pair(polyq_lib, W, a, B, bits)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    assert dev.xscale is not None
    xb, x = synth.activations(a, batch, seed)
    y = polyq_lib.linear_gemv(dev, _x_dev(xb))
    torch.cuda.synchronize()
    check_tolerance(y.cpu().numpy(), O.linear_scaled(ref, x), x, K)


def test_snapped_gemv_matches_oracle(polyq_lib):
    W, a = synth.layer_weights(512, 5120, 2001)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, snap_quanta=True)
    sal = O.saliency(W, a)
    bits = O.snap_to_quanta(O.allocate_bits(sal, 3.0), O.saliency_error_table(sal), 3.0)
    ref = O.pack_layer(W, a, 3.0, bits=bits)
    assert host.info()["pad_bytes"] == 0
    dev = polyq_lib.DeviceLayer(host, "cuda")
    xb, x = synth.activations(a, 2, 2001)
    y = polyq_lib.linear_gemv(dev, _x_dev(xb))
    torch.cuda.synchronize()
    check_tolerance(y.cpu().numpy(), O.linear(ref, x), x, 5120)


def test_scaled_gemv_with_fused_rmsnorm(polyq_lib):
    # The transform's bf16 copy is the layer input, unscaled; the factors
    # apply only inside the product.
    K = 1536
    W, a = synth.layer_weights(300, K, 21)
    host, ref = _scaled_pair(polyq_lib, W, a, 3.0)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    s = np.random.default_rng(5).normal(0, 1, (3, K)) * a[None, :]
    s32 = s.astype(np.float32)
    xo = torch.empty(3, K, dtype=torch.bfloat16, device="cuda")
    ys = polyq_lib.linear_gemv_input([dev], polyq_lib.X_RMSNORM, torch.from_numpy(s32).cuda(),
                                     eps=1e-6, x_out=xo)
    torch.cuda.synchronize()
    h = O.bf16_rn(O.rmsnorm(s32.astype(np.float64), 1e-6))
    got_x = xo.float().cpu().numpy().astype(np.float64)
    # fp32 on the GPU against fp64 here: at most one bf16 step apart
    assert np.all(np.abs(got_x - h) <= np.abs(h) * 2.0 ** -7)
    assert np.mean(got_x == h) > 0.99
    check_tolerance(ys[0].cpu().numpy(), O.linear_scaled(ref, got_x), got_x, K)


@pytest.mark.parametrize("M,N,K,seed,forced", [
    (256, 256, 1100, 61, True),
    (512, 640, 2048, 62, False),
    (2000, 320, 2048, 63, True),  # more rows than pre-pass CTAs: the next row loads while one is gathered
])
def test_scaled_gemm_matches_oracle(polyq_lib, M, N, K, seed, forced):
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed) if forced else None
    host, ref = _scaled_pair(polyq_lib, W, a, 3.0, bits)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    Xb, X = synth.activations(a, M, seed)
    Y = polyq_lib.linear_gemm(dev, _x_dev(Xb))
    torch.cuda.synchronize()
    check_tolerance(Y.cpu().numpy(), O.linear_scaled(ref, X), X, K)
