"""Seeded synthetic inputs shaped like the paper's workloads.

This module only draws random numbers; it holds none of the method's
arithmetic.  Both the tests (oracle side) and the benchmarks (CUDA side) take
their inputs from here.

Recipe (stand-in for calibrated Falcon-H1-3B / Llama2-13B / Qwen3-32B layers,
whose weights and calibration data are not available):

* ``numpy.random.Generator(PCG64(seed))``, one seed per layer;
* W[n,k] ~ N(0, 0.02^2) in fp32; round(0.01*K) columns drawn without
  replacement are multiplied by 10 (weight-outlier channels);
* channel magnitudes m_k ~ lognormal(0, 1); an independent round(0.01*K)
  channels are multiplied by 20 (activation-outlier channels);
  ``act_absmean = m`` (fp32);
* activations x[b,k] = bf16_rn(m_k * zeta[b,k]), zeta ~ N(0, 1), drawn from a
  second generator seeded ``seed + 7919``.
"""
from __future__ import annotations

import numpy as np


def _rng(seed):
    return np.random.Generator(np.random.PCG64(int(seed)))


def layer_weights(N, K, seed):
    """(W fp32 [N][K], act_absmean fp32 [K]) for one synthetic linear layer."""
    rng = _rng(seed)
    W = rng.standard_normal((N, K), dtype=np.float32)
    W *= np.float32(0.02)
    n_out = int(round(0.01 * K))
    if n_out:
        cols = rng.choice(K, size=n_out, replace=False)
        W[:, cols] *= np.float32(10.0)
    m = rng.lognormal(0.0, 1.0, size=K)
    if n_out:
        ch = rng.choice(K, size=n_out, replace=False)
        m[ch] *= 20.0
    return W, m.astype(np.float32)


def bf16_bits(v):
    """Round float32 values to bf16 (ties to even); returns uint16 bit
    patterns.  Input values must be finite."""
    f = np.ascontiguousarray(np.asarray(v, dtype=np.float32))
    u = f.view(np.uint32).astype(np.uint64)
    r = (u + 0x7FFF + ((u >> 16) & 1)) >> 16
    return r.astype(np.uint16)


def bf16_to_f64(bits):
    """fp64 values of bf16 bit patterns (exact)."""
    u = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return u.view(np.float32).astype(np.float64)


def activations(act_absmean, batch, seed):
    """bf16 activations [batch][K] as (uint16 bits, fp64 values)."""
    rng = _rng(int(seed) + 7919)
    m = np.asarray(act_absmean, dtype=np.float64)
    zeta = rng.standard_normal((batch, m.shape[0]))
    bits = bf16_bits((m[None, :] * zeta).astype(np.float32))
    return bits, bf16_to_f64(bits)


def random_codes_layer_bits(K, seed, widths=(2, 3, 4, 8, 16)):
    """A width map that contains every width in ``widths`` (tests that must
    reach all five code paths regardless of the allocation)."""
    rng = _rng(seed)
    bits = rng.choice(np.asarray(widths), size=K)
    bits[: len(widths)] = widths
    rng.shuffle(bits)
    return bits.astype(np.int64)


def seed_for(config, layer_index):
    """Per-layer seed: 1000 * config + layer index."""
    return 1000 * int(config) + int(layer_index)
