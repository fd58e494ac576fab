"""GPU parity of the tcgen05 prefill GEMM against the oracle (through the C ABI)."""
import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth
from tests.gpu_util import check_tolerance, oracle_rows

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _x_dev(xb):
    return torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).cuda().view(torch.bfloat16)


@pytest.mark.parametrize("M,N,K,B,seed,forced", [
    (256, 256, 1100, 3.0, 51, True),     # all five widths, one work unit
    (300, 300, 1100, 3.0, 52, True),     # ragged M and N, two units per axis
    (1, 100, 700, 3.0, 53, True),        # a single token
    (512, 640, 2048, 3.0, 54, False),    # allocation at B = 3
    (130, 257, 1536, 6.0, 55, False),    # B = 6: many 8-bit channels
    (64, 64, 320, 16.0, 56, False),      # all 16-bit
    (96, 96, 640, 2.0, 57, False),       # all 2-bit
    (300, 520, 2100, 3.0, 60, True),     # stream-K: ~3 K tiles per CTA, cut across tiles
    (64, 2000, 4000, 3.0, 61, False),    # uniform K split into 8 ranges
    (2000, 320, 1600, 3.0, 62, True),    # more rows than pre-pass CTAs (rows held in registers)
])
def test_gemm_matches_oracle(polyq_lib, M, N, K, B, seed, forced):
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed) if forced else None
    Xb, X = synth.activations(a, M, seed)
    host = polyq_lib.HostLayer.pack(W, a, B, forced_bits=bits)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    ref = O.pack_layer(W, a, B, bits=bits)
    ws = torch.zeros(polyq_lib.gemm_workspace_bytes(dev, M), dtype=torch.uint8, device="cuda")
    Y = polyq_lib.linear_gemm(dev, _x_dev(Xb), workspace=ws)
    torch.cuda.synchronize()
    assert polyq_lib.workspace_status(ws[-256:]) == 0  # no bounded wait gave up
    check_tolerance(Y.cpu().numpy(), O.linear(ref, X), X, K)


def test_gemm_identity_gather_and_repeat(polyq_lib):
    W, a = synth.layer_weights(384, 1200, 58)
    bits = synth.random_codes_layer_bits(1200, 58)
    Xb, X = synth.activations(a, 200, 58)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
    ref = O.pack_layer(W, a, 3.0, bits=bits)
    dev = polyq_lib.DeviceLayer(host, "cuda", identity_gather=True)
    Xs = np.ascontiguousarray(Xb[:, ref["perm"]])
    ws = torch.zeros(polyq_lib.gemm_workspace_bytes(dev, 200), dtype=torch.uint8, device="cuda")
    Y1 = polyq_lib.linear_gemm(dev, _x_dev(Xs), workspace=ws)
    Y2 = polyq_lib.linear_gemm(dev, _x_dev(Xs), workspace=ws)
    torch.cuda.synchronize()
    check_tolerance(Y1.cpu().numpy(), O.linear(ref, X), X, 1200)
    # a small problem splits K over CTAs: repeated runs agree to fp32 rounding
    assert torch.allclose(Y1, Y2, rtol=1e-5, atol=1e-5 * float(Y1.abs().max()))


@pytest.mark.parametrize("name,N,K,M", [
    ("llama-gate", 13824, 5120, 512),
    ("llama-down", 5120, 13824, 2048),
])
def test_gemm_full_size_sampled(polyq_lib, name, N, K, M):
    seed = 9000 + N + K
    W, a = synth.layer_weights(N, K, seed)
    Xb, X = synth.activations(a, M, seed)
    host = polyq_lib.HostLayer.pack(W, a, 3.0)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    Y = polyq_lib.linear_gemm(dev, _x_dev(Xb))
    torch.cuda.synchronize()
    rng = np.random.default_rng(2)
    rows = np.unique(np.concatenate([[0, N - 1], rng.integers(0, N, 40)]))
    ms = np.unique(np.concatenate([[0, M - 1], rng.integers(0, M, 6)]))
    ref, _ = oracle_rows(W, a, 3.0, rows)
    yref = O.linear(ref, X[ms])
    check_tolerance(Y.cpu().numpy()[np.ix_(ms, rows)], yref, X[ms], K)


@pytest.mark.parametrize("scale_exp", [-40, -12, -8, 4, 10, 40])
def test_gemm_meets_tolerance_at_any_activation_scale(polyq_lib, scale_exp):
    """Each row of X is scaled by a power of two before its fp16 conversion,
    so the relative tolerance holds at any scale.  Rows here also differ from
    each other by up to 2^6, and all five widths are present."""
    M, N, K, seed = 300, 300, 1100, 59
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed)
    _, X = synth.activations(a, M, seed)
    f = 2.0 ** (scale_exp + (np.arange(M) % 7) - 3)
    Xs = X * f[:, None]
    Xb = synth.bf16_bits(Xs.astype(np.float32))
    assert np.array_equal(synth.bf16_to_f64(Xb), Xs)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    ref = O.pack_layer(W, a, 3.0, bits=bits)
    Y = polyq_lib.linear_gemm(dev, _x_dev(Xb))
    torch.cuda.synchronize()
    check_tolerance(Y.cpu().numpy(), O.linear(ref, Xs), Xs, K)


def test_gemm_rejects_unaligned_output(polyq_lib):
    W, a = synth.layer_weights(64, 256, 62)
    host = polyq_lib.HostLayer.pack(W, a, 3.0)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    Xb, _ = synth.activations(a, 4, 62)
    Ybuf = torch.zeros(4 * 64 + 1, dtype=torch.float32, device="cuda")
    with pytest.raises(polyq_lib.PolyqError) as ei:
        polyq_lib.linear_gemm(dev, _x_dev(Xb), Y=Ybuf[1:].view(4, 64))
    assert ei.value.code == polyq_lib.POLYQ_EINVAL


def test_gemm_rows_too_wide_to_stage(polyq_lib):
    """Rows of X wider than the pre-pass stages in shared memory (K > 49152)
    are gathered from global memory instead; with activation factors too."""
    M, N, K, seed = 40, 96, 50003, 63
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed)
    Xb, X = synth.activations(a, M, seed)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
    dev = polyq_lib.DeviceLayer(host, "cuda")
    ref = O.pack_layer(W, a, 3.0, bits=bits)
    Y = polyq_lib.linear_gemm(dev, _x_dev(Xb))
    torch.cuda.synchronize()
    check_tolerance(Y.cpu().numpy(), O.linear(ref, X), X, K)
