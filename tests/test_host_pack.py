"""Host-side parity: the library's packer (C++) against the oracle (NumPy),
bit for bit, plus the C-ABI surface and argument validation.  No GPU."""
import ctypes as C
import os
import re

import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth

HEADER = os.path.join(os.path.dirname(os.path.dirname(__file__)), "include", "polyq.h")


def _declared_functions(header=HEADER):
    text = open(header).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(polyq_[a-z0-9_]+)\s*\(", text)))


def test_debug_library_exports_its_declared_symbols(polyq_lib):
    """The debug build (a test aid) exports what include/polyq_debug.h
    declares, besides everything the product exports; the product library
    exports none of the debug calls."""
    from paper_2607_14618_gb300 import build
    names = _declared_functions(os.path.join(os.path.dirname(HEADER), "polyq_debug.h"))
    assert names == ["polyq_debug_gemm_weights", "polyq_debug_gemv_codes"]
    dbg = C.CDLL(build.build_library(debug=True))
    for n in names + _declared_functions():
        assert hasattr(dbg, n), n
    lib = C.CDLL(polyq_lib.LIB_PATH)
    for n in names:
        assert not hasattr(lib, n), n


def test_library_exports_every_declared_symbol(polyq_lib):
    names = _declared_functions()
    assert len(names) >= 15
    lib = C.CDLL(polyq_lib.LIB_PATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) <= set(polyq_lib.exported_symbols())


def test_f64_to_f16_matches_numpy(polyq_lib):
    rng = np.random.default_rng(0)
    vals = list(rng.normal(0, 1, 2000) * 10.0 ** rng.integers(-9, 5, 2000))
    vals += [0.0, -0.0, 1.0, 65504.0, 65519.99, 2.0 ** -24, 2.0 ** -25, 3 * 2.0 ** -26,
             2.0 ** -14, 2.0 ** -14 - 2.0 ** -25, 1 + 2.0 ** -11, 1 + 2.0 ** -11 + 2.0 ** -40,
             1 + 3 * 2.0 ** -11, 6.1e-5, 0.0123]
    for v in vals:
        got = polyq_lib.f64_to_f16(v)
        ref = int(np.array([v], np.float64).astype(np.float16).view(np.uint16)[0])
        assert got == ref, (v, hex(got), hex(ref))


def _compare(host, ref):
    ex = host.export()
    inf = ex["info"]
    assert inf["N"] == ref["N"] and inf["K"] == ref["K"]
    assert np.array_equal(ex["bits"], ref["bits"].astype(np.uint8))
    assert np.array_equal(ex["perm"], ref["perm"].astype(np.int32))
    assert inf["row_stride"] == ref["row_stride"] and inf["n_groups"] == ref["n_groups"]
    assert inf["blocks"] == ref["blocks"]
    assert np.array_equal(ex["packed"], ref["packed"])
    meta_ref = ref["meta"][:, :, 0].astype(np.uint32) | (ref["meta"][:, :, 1].astype(np.uint32) << 16)
    assert np.array_equal(ex["meta"], meta_ref)
    assert inf["b_real"] == O.realized_budget(ref)
    ms = inf["meta_stride"]
    assert ms % 4 == 0 and ms >= inf["n_groups"]
    padded = host.export(meta_stride=ms)["meta"]
    assert np.array_equal(padded[:, :inf["n_groups"]], meta_ref)
    assert np.all(padded[:, inf["n_groups"]:] == 0)


@pytest.mark.parametrize("N,K,B,seed", [
    (2048, 2048, 3.0, 1001),   # the 2048 x 2048, B = 3.0 decode layer
    (64, 5120, 4.5, 2001),
    (48, 5120, 6.0, 3003),
    (96, 1000, 2.0, 5),
    (33, 777, 2.7, 6),
    (7, 129, 16.0, 7),
    (5, 64, 3.3, 8),
])
def test_pack_matches_oracle(polyq_lib, N, K, B, seed):
    W, a = synth.layer_weights(N, K, seed)
    host = polyq_lib.HostLayer.pack(W, a, B)
    _compare(host, O.pack_layer(W, a, B))


@pytest.mark.parametrize("seed", [11, 12, 13])
def test_pack_forced_widths_matches_oracle(polyq_lib, seed):
    rng = np.random.default_rng(seed)
    K = int(rng.integers(5, 700))
    N = int(rng.integers(1, 40))
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
    _compare(host, O.pack_layer(W, a, 3.0, bits=bits))


def test_pack_edge_weights_match_oracle(polyq_lib):
    # constant groups, zeros, tiny and large magnitudes, fp16 subnormal scales
    W = np.zeros((6, 200), np.float32)
    W[1] = 1e-7
    W[2] = np.linspace(-3e-6, 5e-6, 200, dtype=np.float32)
    W[3] = 60000.0
    W[4, ::3] = -65504.0
    W[5] = np.random.default_rng(1).normal(0, 100, 200).astype(np.float32)
    a = np.ones(200, np.float32)
    bits = synth.random_codes_layer_bits(200, 4)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
    _compare(host, O.pack_layer(W, a, 3.0, bits=bits))


def test_ladder_and_palette_match_oracle(polyq_lib):
    W, a = synth.layer_weights(40, 900, 21)
    host = polyq_lib.HostLayer.pack(W, a, 3.4, rule=polyq_lib.ALLOC_LADDER)
    ref_bits = O.allocate_bits(O.saliency(W, a), 3.4, rule=O.SALIENCY_LADDER)
    assert np.array_equal(host.export()["bits"], ref_bits.astype(np.uint8))
    host = polyq_lib.HostLayer.pack(W, a, 3.4, palette=(2, 4, 8))
    ref_bits = O.allocate_bits(O.saliency(W, a), 3.4, palette=(2, 4, 8))
    assert np.array_equal(host.export()["bits"], ref_bits.astype(np.uint8))


def test_thread_count_does_not_change_result(polyq_lib):
    W, a = synth.layer_weights(300, 1500, 9)
    e1 = polyq_lib.HostLayer.pack(W, a, 3.7, n_threads=1).export()
    e8 = polyq_lib.HostLayer.pack(W, a, 3.7, n_threads=8).export()
    for k in ("packed", "meta", "perm", "bits"):
        assert np.array_equal(e1[k], e8[k])


def test_permute_merge_matches_oracle(polyq_lib):
    rng = np.random.default_rng(3)
    for n in (1, 5, 1000):
        beta, pc = rng.permutation(n), rng.permutation(n)
        assert np.array_equal(polyq_lib.permute_merge(beta, pc), O.permute_merge(beta, pc))
    with pytest.raises(polyq_lib.PolyqError) as ei:
        polyq_lib.permute_merge([0, 0, 2], [0, 1, 2])
    assert ei.value.code == polyq_lib.POLYQ_EINVAL


def test_permute_rows_matches_oracle(polyq_lib):
    Wp, ap = synth.layer_weights(150, 80, 41)
    host = polyq_lib.HostLayer.pack(Wp, ap, 3.0)
    ref = O.pack_layer(Wp, ap, 3.0)
    rp = np.random.default_rng(0).permutation(150)
    host.permute_rows(rp)
    ref = O.permute_rows(ref, rp)
    _compare(host, ref)
    assert np.array_equal(host.export()["out_perm"], ref["out_perm"])
    with pytest.raises(polyq_lib.PolyqError):
        host.permute_rows(np.zeros(150, np.int32))


def test_pack_rejects_bad_arguments(polyq_lib):
    W, a = synth.layer_weights(4, 16, 1)
    for B in (1.9, 16.5, float("nan")):
        with pytest.raises(polyq_lib.PolyqError) as ei:
            polyq_lib.HostLayer.pack(W, a, B)
        assert ei.value.code == polyq_lib.POLYQ_EINVAL
    Wbad = W.copy()
    Wbad[0, 0] = np.inf
    with pytest.raises(polyq_lib.PolyqError):
        polyq_lib.HostLayer.pack(Wbad, a, 3.0)
    Wbad[0, 0] = 70000.0
    with pytest.raises(polyq_lib.PolyqError):
        polyq_lib.HostLayer.pack(Wbad, a, 3.0)
    with pytest.raises(polyq_lib.PolyqError):
        polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=np.full(16, 5))
    with pytest.raises(polyq_lib.PolyqError):
        polyq_lib.HostLayer.pack(W, a, 3.0, palette=(5,))


def _desc_from(polyq_lib, host):
    """A descriptor with fake (never dereferenced) aligned device addresses."""
    d = polyq_lib.DevLayer()
    rc = polyq_lib._lib.polyq_dev_layer_fill(host._h, C.c_void_p(0x100000), C.c_void_p(0x200000),
                                            None, C.byref(d))
    assert rc == 0
    return d


def test_corrupt_descriptors_rejected_before_launch(polyq_lib):
    """Host-side fault injection: every corrupted descriptor is refused with
    POLYQ_EINVAL before any device work is queued."""
    W, a = synth.layer_weights(8, 300, 2)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=synth.random_codes_layer_bits(300, 2))
    L = polyq_lib._lib

    def gemv(d, batch=1):
        return L.polyq_linear_gemv(C.byref(d), C.c_void_p(0x300000), batch, C.c_void_p(0x400000),
                                   None, None, 0, None)

    def mutate(f):
        d = _desc_from(polyq_lib, host)
        f(d)
        return d

    cases = [
        lambda d: setattr(d, "row_stride", d.row_stride + 8),
        lambda d: setattr(d, "K", d.K + 1),
        lambda d: setattr(d, "N", 0),
        lambda d: setattr(d, "n_blocks", 0),
        lambda d: setattr(d, "n_blocks", 6),
        lambda d: setattr(d, "packed", 0x100001),
        lambda d: setattr(d, "meta", None),
        lambda d: setattr(d.blocks[1], "bits", 5),
        lambda d: setattr(d.blocks[2], "n_ch", d.blocks[2].n_ch + 1),
        lambda d: setattr(d.blocks[0], "seg_bytes", d.blocks[0].seg_bytes + 16),
        lambda d: setattr(d.blocks[3], "grp_off", 0),
        lambda d: setattr(d, "n_groups", d.n_groups - 1),
        lambda d: setattr(d, "meta_stride", d.meta_stride + 1),
        lambda d: setattr(d, "xscale", 0x500004),
        lambda d: setattr(d, "meta_stride", d.n_groups - 1),
    ]
    for f in cases:
        d = mutate(f)
        assert gemv(d) == polyq_lib.POLYQ_EINVAL, polyq_lib.last_error()
        codes_rc = L.polyq_unpack_codes(C.byref(d), C.c_void_p(0x500000), None)
        assert codes_rc == polyq_lib.POLYQ_EINVAL
    d = _desc_from(polyq_lib, host)
    assert gemv(d, batch=0) == polyq_lib.POLYQ_EUNSUPPORTED
    assert gemv(d, batch=5) == polyq_lib.POLYQ_EUNSUPPORTED
    assert L.polyq_linear_gemv(C.byref(d), None, 1, C.c_void_p(0x400000), None, None, 0,
                               None) == polyq_lib.POLYQ_EINVAL


# ---------------------------------------------------------------------------
# Section 3.1 quantiser proxy, Section 3.3 quanta matching, Section 3.4
# scaling: the library against the oracle, bit for bit
# ---------------------------------------------------------------------------
def _x2(a):
    return np.asarray(a, np.float32).astype(np.float64) ** 2


@pytest.mark.parametrize("N,K,B,seed", [
    (256, 2048, 3.0, 1000),   # the 2048-channel decode layer's shape at B = 3
    (64, 5120, 4.5, 2001),
    (40, 1000, 3.7, 5),       # K a multiple of 8 only
    (33, 777, 2.6, 6),        # no exact sum: the 2-bit block fills
    (16, 13824, 3.0, 2006),
])
def test_snap_to_quanta_matches_oracle(polyq_lib, N, K, B, seed):
    W, a = synth.layer_weights(N, K, seed)
    host = polyq_lib.HostLayer.pack(W, a, B, snap_quanta=True)
    sal = O.saliency(W, a)
    bits = O.snap_to_quanta(O.allocate_bits(sal, B), O.saliency_error_table(sal), B)
    _compare(host, O.pack_layer(W, a, B, bits=bits))
    inf = host.info()
    assert inf["pad_bytes"] == O.padding_bytes_per_row(bits)
    if K % 128 == 0:
        assert inf["pad_bytes"] == 0


def test_snap_with_custom_quanta_and_ladder_matches_oracle(polyq_lib):
    W, a = synth.layer_weights(24, 3000, 31)
    q = {2: 96, 3: 32, 4: 48, 8: 8, 16: 8}
    host = polyq_lib.HostLayer.pack(W, a, 3.3, snap_quanta=True, quanta=q,
                                    rule=polyq_lib.ALLOC_LADDER)
    sal = O.saliency(W, a)
    bits = O.snap_to_quanta(O.allocate_bits(sal, 3.3, rule=O.SALIENCY_LADDER),
                            O.saliency_error_table(sal), 3.3, quanta=q)
    assert np.array_equal(host.export()["bits"], bits.astype(np.uint8))


@pytest.mark.parametrize("N,K,B,seed", [
    (128, 2048, 3.0, 1000),
    (50, 777, 4.2, 7),
    (20, 64, 2.5, 8),
])
def test_quant_proxy_allocation_matches_oracle(polyq_lib, N, K, B, seed):
    W, a = synth.layer_weights(N, K, seed)
    host = polyq_lib.HostLayer.pack(W, a, B, proxy=polyq_lib.PROXY_QUANT)
    bits = O.allocate_from_table(O.quant_error_table(W, _x2(a)), B)
    _compare(host, O.pack_layer(W, a, B, bits=bits))


def test_quant_proxy_with_explicit_second_moments(polyq_lib):
    W, a = synth.layer_weights(40, 900, 12)
    x2 = (np.random.default_rng(1).random(900) * 3).astype(np.float32)
    host = polyq_lib.HostLayer.pack(W, a, 3.2, proxy=polyq_lib.PROXY_QUANT, act_sqmean=x2)
    bits = O.allocate_from_table(O.quant_error_table(W, x2.astype(np.float64)), 3.2)
    assert np.array_equal(host.export()["bits"], bits.astype(np.uint8))


def _compare_scaled(host, W, a, bits, x2):
    alphas, t = O.choose_alphas(W, bits, a, x2)
    ref = O.pack_layer_scaled(W, bits, t)
    _compare(host, ref)
    inf = host.info()
    assert inf["has_xscale"] == 1
    for b in O.PALETTE:
        assert inf["alpha"][b] == (alphas[b] if b in alphas else -1.0)
    assert np.array_equal(host.xscale(), ref["xscale"].astype(np.float32))


@pytest.mark.parametrize("N,K,B,seed", [
    (96, 2048, 3.0, 1000),
    (40, 1000, 4.5, 9),
])
def test_scaled_pack_matches_oracle(polyq_lib, N, K, B, seed):
    W, a = synth.layer_weights(N, K, seed)
    host = polyq_lib.HostLayer.pack(W, a, B, proxy=polyq_lib.PROXY_QUANT, snap_quanta=True,
                                    act_scaling=True)
    E = O.quant_error_table(W, _x2(a))
    bits = O.snap_to_quanta(O.allocate_from_table(E, B), E, B)
    _compare_scaled(host, W, a, bits, _x2(a))


def test_scaled_pack_with_forced_widths_matches_oracle(polyq_lib):
    W, a = synth.layer_weights(30, 3001, 13)
    bits = synth.random_codes_layer_bits(3001, 13)
    host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits, act_scaling=True)
    _compare_scaled(host, W, a, bits, _x2(a))


def test_scaled_pack_finds_the_hand_worked_exponent(polyq_lib):
    # The one-row 2-bit block of the Section 3.4 oracle pins: only alpha = 1/2
    # puts every scaled weight on the 2-bit grid (worked by hand there), and
    # then the packed layer reproduces W exactly.
    m = np.array([4.0, 0.25, 0.25, 0.25, 0.25, 1.0], np.float32)
    W = np.array([[3 / 16, 0.25, 0.5, 0.5, 0.25, 0.0]], np.float32)
    host = polyq_lib.HostLayer.pack(W, m, 2.0, forced_bits=np.full(6, 2), act_scaling=True,
                                    act_sqmean=np.ones(6, np.float32))
    inf = host.info()
    assert inf["alpha"][2] == 0.5
    ex = host.export()
    assert host.xscale().tolist() == [0.5, 2.0, 2.0, 2.0, 2.0, 1.0]  # perm is the identity
    assert ex["perm"].tolist() == list(range(6))
    ref = O.pack_layer_scaled(W, np.full(6, 2), np.array([0.5, 2, 2, 2, 2, 1.0]))
    assert np.array_equal(ex["packed"], ref["packed"])
    meta_ref = ref["meta"][:, :, 0].astype(np.uint32) | (ref["meta"][:, :, 1].astype(np.uint32) << 16)
    assert np.array_equal(ex["meta"], meta_ref)
    assert np.array_equal(O.dequant(ref) * ref["xscale"][None, :], W.astype(np.float64))


def test_unscaled_layer_reports_no_factors(polyq_lib):
    W, a = synth.layer_weights(8, 300, 14)
    host = polyq_lib.HostLayer.pack(W, a, 3.0)
    inf = host.info()
    assert inf["has_xscale"] == 0 and all(v == -1.0 for v in inf["alpha"].values())
    assert np.all(host.xscale() == 1.0)


def test_new_pack_options_are_validated(polyq_lib):
    W, a = synth.layer_weights(4, 128, 1)
    bad = [
        dict(snap_quanta=True, forced_bits=np.full(128, 3)),
        dict(proxy=polyq_lib.PROXY_QUANT, rule=polyq_lib.ALLOC_LADDER),
        dict(proxy=7),
        dict(act_sqmean=np.full(128, -1.0, np.float32), proxy=polyq_lib.PROXY_QUANT),
        dict(act_sqmean=np.full(128, np.nan, np.float32), act_scaling=True),
    ]
    for kw in bad:
        with pytest.raises(polyq_lib.PolyqError) as ei:
            polyq_lib.HostLayer.pack(W, a, 3.0, **kw)
        assert ei.value.code == polyq_lib.POLYQ_EINVAL, kw
    opts = polyq_lib.PackOpts()
    polyq_lib._lib.polyq_pack_opts_default(C.byref(opts))
    opts.snap_quanta = 1
    opts.quanta[0] = 64  # one quantum set, the others zero
    h = C.c_void_p()
    W32 = np.ascontiguousarray(W, np.float32)
    a32 = np.ascontiguousarray(a, np.float32)
    rc = polyq_lib._lib.polyq_pack(W32.ctypes.data, 4, 128, a32.ctypes.data, 3.0,
                                   C.byref(opts), C.byref(h))
    assert rc == polyq_lib.POLYQ_EINVAL
    with pytest.raises(polyq_lib.PolyqError):
        polyq_lib.HostLayer.pack(W, None, 3.0, forced_bits=np.full(128, 3), act_scaling=True)


def test_chain_overlap_rules_checked_before_any_device_work(polyq_lib):
    """polyq_gemv_chain_create rejects hazards between and inside phases on
    the host (fake, never dereferenced device addresses)."""
    W, a = synth.layer_weights(64, 128, 3)
    host = polyq_lib.HostLayer.pack(W, a, 3.0)
    d = _desc_from(polyq_lib, host)
    L = polyq_lib._lib
    base = 0x10000000

    def phase(x, y, res=None, kind=polyq_lib.X_F32):
        ph = polyq_lib.GemvPhase()
        ph.n_layers = 1
        ph.layers[0] = C.pointer(d)
        ph.in_ = polyq_lib.GemvInput(kind, 1e-6, x, None, None)
        ph.ys[0] = y
        ph.residuals[0] = res
        return ph

    def create(*phs):
        arr = (polyq_lib.GemvPhase * len(phs))(*phs)
        h = C.c_void_p()
        rc = L.polyq_gemv_chain_create(arr, len(phs), 1, C.byref(h))
        if rc == 0:
            L.polyq_gemv_chain_free(h)
        return rc

    x0, y0, y1 = base, base + 0x10000, base + 0x20000
    # output overlapping its own input
    assert create(phase(x0, x0 + 256)) == polyq_lib.POLYQ_EINVAL
    # phase 1's fresh output overlapping phase 0's input
    assert create(phase(x0, y0), phase(y0, x0)) == polyq_lib.POLYQ_EINVAL
    # phase 1's fresh output overlapping phase 0's output
    assert create(phase(x0, y0), phase(x0, y0 + 64)) == polyq_lib.POLYQ_EINVAL
    # a residual overlapping (but not equal to) its output
    assert create(phase(x0, y0, y0 + 4)) == polyq_lib.POLYQ_EINVAL
    # bad phase count and batch
    assert L.polyq_gemv_chain_create(None, 0, 1, C.byref(C.c_void_p())) == polyq_lib.POLYQ_EINVAL
    # a legal chain passes the host checks: in place (y == residual) after a
    # phase that read y, then a fresh output elsewhere.  Without a GPU the
    # first device query fails instead.
    rc = create(phase(x0, y0), phase(y0, x0, x0), phase(y0, y1))
    assert rc in (0, polyq_lib.POLYQ_ECUDA)


def test_binding_rejects_wrong_buffers_before_the_library(polyq_lib):
    """The binding checks every buffer it hands to the library as a raw
    pointer: dtype, shape, device and contiguity (CPU tensors here; on a GPU
    the same checks compare against the input's CUDA device)."""
    import torch
    cpu = torch.device("cpu")
    ok = torch.zeros(2, 8)
    polyq_lib._require(ok, "y", torch.float32, (2, 8), cpu)
    bad = [torch.zeros(2, 8, dtype=torch.float16), torch.zeros(8, 2), torch.zeros(2, 9),
           torch.zeros(8, 2).t(), torch.zeros(2, 16)[:, ::2], np.zeros((2, 8), np.float32)]
    for t in bad:
        with pytest.raises(ValueError):
            polyq_lib._require(t, "y", torch.float32, (2, 8), cpu)
    # inputs must be CUDA tensors of the right dtype and width
    for x in (torch.zeros(1, 16, dtype=torch.bfloat16), torch.zeros(1, 16)):
        with pytest.raises(ValueError):
            polyq_lib._cuda_input(x, "x", torch.bfloat16, 16)


def test_gemm_rejects_unaligned_output_on_the_host(polyq_lib):
    W, a = synth.layer_weights(64, 256, 62)
    host = polyq_lib.HostLayer.pack(W, a, 3.0)
    d = _desc_from(polyq_lib, host)
    L = polyq_lib._lib
    rc = L.polyq_linear_gemm(C.byref(d), C.c_void_p(0x300000), 4, C.c_void_p(0x400004),
                             C.c_void_p(0x500000), 1 << 24, None)
    assert rc == polyq_lib.POLYQ_EINVAL
    assert "16-byte" in polyq_lib.last_error()
