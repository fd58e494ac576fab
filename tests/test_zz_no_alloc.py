"""polyq_linear_gemv_noalloc: the decode GEMV on the library's own fixed scratch.

Some callers cannot allocate device memory (a plugin inside a host program
whose memory pool owns the device, or a loop that cannot take the device-wide
synchronisation cudaMalloc/cudaFree may cause), so this entry point takes no
workspace.  Its results must match polyq_linear_gemv's on the same inputs,
call after call, although every call reuses the same scratch array.  The file
name makes pytest collect it last.
"""
import numpy as np
import pytest

from paper_2607_14618_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _x_dev(xb):
    return torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).cuda().view(torch.bfloat16)


def _same(got, ref):
    # two runs of the GEMV differ only in the order of the fp32 additions of
    # split rows: the run-to-run tolerance of the GEMV tests
    assert torch.allclose(got, ref, rtol=1e-5, atol=1e-5 * float(ref.abs().max()))


def test_noalloc_matches_workspace_entry_on_two_calls(polyq_lib):
    # call 1: a layer with all five widths at batch 4, no residual
    W1, a1 = synth.layer_weights(1000, 3000, 71)
    bits1 = synth.random_codes_layer_bits(3000, 71)
    dev1 = polyq_lib.DeviceLayer(polyq_lib.HostLayer.pack(W1, a1, 3.0, forced_bits=bits1), "cuda")
    xb1, _ = synth.activations(a1, 4, 71)
    x1 = _x_dev(xb1)
    # call 2: another layer at batch 1 with a residual, so that records left by
    # call 1 (other shape, other batch) would show if they leaked through
    W2, a2 = synth.layer_weights(2048, 2048, 72)
    dev2 = polyq_lib.DeviceLayer(polyq_lib.HostLayer.pack(W2, a2, 3.0), "cuda")
    xb2, _ = synth.activations(a2, 1, 72)
    x2 = _x_dev(xb2)
    res2 = torch.randn(1, 2048, device="cuda", dtype=torch.float32)

    ref1 = polyq_lib.linear_gemv(dev1, x1)
    ref2 = polyq_lib.linear_gemv(dev2, x2, residual=res2)
    torch.cuda.synchronize()

    y1 = torch.full((4, 1000), float("nan"), device="cuda")
    y2 = torch.full((1, 2048), float("nan"), device="cuda")
    polyq_lib.linear_gemv_noalloc(dev1, x1, y1)
    polyq_lib.linear_gemv_noalloc(dev2, x2, y2, residual=res2)
    torch.cuda.synchronize()
    _same(y1, ref1)
    _same(y2, ref2)

    # the same two calls again, in the other order, on the now-used scratch
    y2b = torch.full_like(y2, float("nan"))
    y1b = torch.full_like(y1, float("nan"))
    polyq_lib.linear_gemv_noalloc(dev2, x2, y2b, residual=res2)
    polyq_lib.linear_gemv_noalloc(dev1, x1, y1b)
    torch.cuda.synchronize()
    _same(y1b, ref1)
    _same(y2b, ref2)
    # no bounded wait gave up: the scratch's status word reads zero
    assert polyq_lib.noalloc_status() == 0


def _wide_layer(polyq_lib, K):
    # one 64-row tile (16 rows) of K all-8-bit channels
    N = 16
    W, a = synth.layer_weights(N, K, 74)
    bits = np.full(K, 8, dtype=np.uint8)
    dev = polyq_lib.DeviceLayer(polyq_lib.HostLayer.pack(W, a, 8.0, forced_bits=bits), "cuda")
    return dev, a


def test_noalloc_rejects_layers_beyond_the_scratch(polyq_lib):
    # At batch 4 a step covers 128 channels, so K = 131072 has 1024 steps whose
    # activation records (1376 bytes each) do not fit the fixed 1 MiB.
    dev, a = _wide_layer(polyq_lib, 131072)
    assert polyq_lib.gemv_workspace_bytes(dev, 4) > polyq_lib.NOALLOC_SCRATCH_BYTES
    xb, _ = synth.activations(a, 4, 74)
    y = torch.full((4, dev.N), 7.0, device="cuda")
    with pytest.raises(polyq_lib.PolyqError) as e:
        polyq_lib.linear_gemv_noalloc(dev, _x_dev(xb), y)
    assert e.value.code == polyq_lib.POLYQ_ENOMEM
    assert "scratch" in str(e.value)
    torch.cuda.synchronize()
    assert bool((y == 7.0).all())  # rejected before anything was launched


def test_noalloc_wide_layer_many_pieces(polyq_lib):
    # K = 65536 fits at batch 4 (512 steps of 128 channels).  Its one tile is
    # split over hundreds of CTAs, each adding its piece into y.
    dev, a = _wide_layer(polyq_lib, 65536)
    assert polyq_lib.gemv_workspace_bytes(dev, 4) <= polyq_lib.NOALLOC_SCRATCH_BYTES
    xb, _ = synth.activations(a, 4, 74)
    x = _x_dev(xb)
    ref = polyq_lib.linear_gemv(dev, x)
    y = torch.empty(4, dev.N, device="cuda")
    for _ in range(2):
        y.fill_(float("nan"))
        polyq_lib.linear_gemv_noalloc(dev, x, y)
        torch.cuda.synchronize()
        _same(y, ref)
