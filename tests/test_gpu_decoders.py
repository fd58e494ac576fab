"""The hot decoders checked bit for bit (debug build, libpolyq_debug.so):
every code the decode GEMV's MMA steps extract from the TMA-staged packed
rows, and every fp16 weight the prefill GEMM's dequantisers write into the
tensor cores' operand tile, against the oracle's unpacking of the same packed
layer (Section 4.2 packing, R1 dequantisation).  The cases cover all five
widths, ragged blocks (the last, partial group of every block), every 3-bit
pair window, and the batch-1 (two boxes per step) and batch 2-4 (one box,
paired steps) geometries."""
import ctypes as C

import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def dbg(polyq_lib):
    from paper_2607_14618_gb300 import build
    lib = C.CDLL(build.build_library(debug=True))
    P = C.c_void_p
    lib.polyq_debug_gemv_codes.argtypes = [C.POINTER(polyq_lib.DevLayer), P, C.c_int, P, P,
                                           C.c_size_t, P, P]
    lib.polyq_debug_gemm_weights.argtypes = [C.POINTER(polyq_lib.DevLayer), P, C.c_int64, P, P,
                                             C.c_size_t, P, P]
    lib.polyq_last_error.restype = C.c_char_p
    return lib


def _x_dev(xb):
    return torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).cuda().view(torch.bfloat16)


def _layer(polyq_lib, N, K, B, seed, forced):
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed) if forced else None
    host = polyq_lib.HostLayer.pack(W, a, B, forced_bits=bits)
    return polyq_lib.DeviceLayer(host, "cuda"), O.pack_layer(W, a, B, bits=bits), a


@pytest.mark.parametrize("batch", [1, 2, 4])
@pytest.mark.parametrize("N,K,B,seed,forced", [
    (130, 3001, 3.0, 81, True),    # all five widths, ragged blocks
    (64, 2048, 3.0, 82, False),    # the allocation at B = 3
    (70, 700, 6.0, 83, False),     # many 8-bit channels
])
def test_gemv_decoder_codes_bit_exact(polyq_lib, dbg, batch, N, K, B, seed, forced):
    dev, ref, a = _layer(polyq_lib, N, K, B, seed, forced)
    xb, _ = synth.activations(a, batch, seed)
    x = _x_dev(xb)
    y = torch.empty((batch, N), dtype=torch.float32, device="cuda")
    ws = torch.zeros(polyq_lib.gemv_workspace_bytes(dev, batch), dtype=torch.uint8, device="cuda")
    out = torch.full((N, K), -1, dtype=torch.int16, device="cuda")  # 0xFFFF: not decoded
    rc = dbg.polyq_debug_gemv_codes(C.byref(dev.desc), x.data_ptr(), batch, y.data_ptr(),
                                    ws.data_ptr(), ws.numel(), out.data_ptr(), None)
    assert rc == 0, dbg.polyq_last_error()
    torch.cuda.synchronize()
    got = out.cpu().numpy().view(np.uint16).astype(np.int64)
    want = O.unpack_codes(ref)
    bad = np.argwhere(got != want)
    assert bad.size == 0, f"{len(bad)} codes differ, first (row, pos) {bad[:4].tolist()}"


def _oracle_fp16_weights(ref):
    """fp16 bits of (q - z) * s rounded once to fp16 (b < 16), or the stored
    fp16 (b = 16), at every (row, clustered position)."""
    codes = O.unpack_codes(ref)
    out = np.zeros(codes.shape, np.uint16)
    for blk in ref["blocks"]:
        b, kb, p0, g0 = blk["bits"], blk["n_ch"], blk["pos0"], blk["grp_off"]
        c = codes[:, p0:p0 + kb]
        if b == 16:
            out[:, p0:p0 + kb] = c.astype(np.uint16)
            continue
        for g in range(blk["n_grp"]):
            cols = slice(g * O.GROUP, min((g + 1) * O.GROUP, kb))
            s = ref["meta"][:, g0 + g, 0].view(np.float16).astype(np.float64)
            z = ref["meta"][:, g0 + g, 1].view(np.float16).astype(np.float64)
            w = (c[:, cols] - z[:, None]) * s[:, None]
            out[:, p0 + cols.start:p0 + cols.stop] = w.astype(np.float16).view(np.uint16)
    return out


@pytest.mark.parametrize("M,N,K,B,seed,forced", [
    (16, 300, 1100, 3.0, 84, True),    # all five widths, two N tiles, ragged
    (64, 256, 2048, 3.0, 85, False),   # the allocation at B = 3
    (8, 520, 2100, 6.0, 86, False),    # many 8-bit channels; stream-K
])
def test_gemm_dequantised_weights_bit_exact(polyq_lib, dbg, M, N, K, B, seed, forced):
    dev, ref, a = _layer(polyq_lib, N, K, B, seed, forced)
    Xb, _ = synth.activations(a, M, seed)
    X = _x_dev(Xb)
    Y = torch.empty((M, N), dtype=torch.float32, device="cuda")
    ws = torch.empty(polyq_lib.gemm_workspace_bytes(dev, M), dtype=torch.uint8, device="cuda")
    out = torch.full((N, K), -1, dtype=torch.int16, device="cuda")
    rc = dbg.polyq_debug_gemm_weights(C.byref(dev.desc), X.data_ptr(), M, Y.data_ptr(),
                                      ws.data_ptr(), ws.numel(), out.data_ptr(), None)
    assert rc == 0, dbg.polyq_last_error()
    torch.cuda.synchronize()
    got = out.cpu().numpy().view(np.uint16)
    want = _oracle_fp16_weights(ref)
    bad = np.argwhere(got != want)
    assert bad.size == 0, f"{len(bad)} weights differ, first (row, pos) {bad[:4].tolist()}"
