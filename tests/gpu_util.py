"""Helpers shared by the GPU parity tests (inputs, oracle references,
tolerances).  The reference values always come from the oracle."""
import numpy as np

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth


def rel_l2(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return float(np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300))


def check_tolerance(y_gpu, y_ref, x, K, rel=1e-3, absk=2e-3):
    """rel-L2 <= 1e-3 and max-abs <= 2e-3 * ||x||_inf * sqrt(K), per batch
    row, against the fp64 oracle."""
    y_gpu = np.atleast_2d(np.asarray(y_gpu, np.float64))
    y_ref = np.atleast_2d(np.asarray(y_ref, np.float64))
    x = np.atleast_2d(np.asarray(x, np.float64))
    assert y_gpu.shape == y_ref.shape
    assert np.all(np.isfinite(y_gpu))
    for b in range(y_ref.shape[0]):
        r = rel_l2(y_gpu[b], y_ref[b])
        bound = absk * np.max(np.abs(x[b])) * np.sqrt(K)
        err = float(np.max(np.abs(y_gpu[b] - y_ref[b])))
        assert r <= rel, f"batch row {b}: rel-L2 {r:.3e} > {rel}"
        assert err <= bound, f"batch row {b}: max-abs {err:.3e} > {bound:.3e}"


def make_case(N, K, B, seed, forced=False, batch=1):
    W, a = synth.layer_weights(N, K, seed)
    bits = synth.random_codes_layer_bits(K, seed) if forced else None
    xb, x = synth.activations(a, batch, seed)
    return W, a, bits, xb, x


def oracle_layer(W, a, B, bits=None):
    return O.pack_layer(W, a, B, bits=bits)


def oracle_rows(W, a, B, rows, bits_full=None):
    """Oracle layer restricted to ``rows`` (widths from the full layer's
    saliency, quantisation per row)."""
    if bits_full is None:
        bits_full = O.allocate_bits(O.saliency(W, a), B)
    return O.pack_layer(W[rows], a, B, bits=bits_full), bits_full
