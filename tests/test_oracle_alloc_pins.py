"""Pins of the oracle's quanta matching (Section 3.3), quantiser-in-the-loop
proxy (Section 3.1) and bit-specific scaling (Section 3.4) against values
worked out by hand, brute force and invariants.  CPU only."""
import itertools

import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth


# ---------------------------------------------------------------------------
# Section 3.3 step 1: target counts
# ---------------------------------------------------------------------------
def test_gpu_quanta_are_whole_16_byte_chunks():
    for b, q in O.GPU_QUANTA.items():
        assert (q * b) % 128 == 0 and q * b <= 384


def test_quanta_targets_worked_example():
    # K = 256, B = 3: the widths above 2 must add sum (b-2)*c = 768 - 512 =
    # 256 extra bits.  Candidates: c2 in {0,64,128,192}, c3 in {0,128,256},
    # c4 in {0,32,64,96}, c8 in {0,16,32}, c16 in {0,8,16}.  c3 + 2 c4 +
    # 6 c8 + 14 c16 = 256 with the counts summing to 256 has exactly these
    # solutions: (64,128,64,0,0) moving 36+28+14+6 = 84 channels,
    # (192,0,32,32,0) moving 236 and (0,256,0,0,0) moving 312.
    counts = {2: 100, 3: 100, 4: 50, 8: 6, 16: 0}
    t = O.quanta_targets(counts, O.GPU_QUANTA, 3.0, 256)
    assert t == {2: 64, 3: 128, 4: 64, 8: 0, 16: 0}


def test_quanta_targets_narrowest_width_fills_when_no_sum_fits():
    # K = 100 is no sum of multiples of 64, 128, 32 inside the candidate
    # windows c2 in {0,64}, c3 in {0}, c4 in {0,32,64}.  The 2-bit block takes
    # the rest: c4 = 0 -> 200 bits, 32 -> 264, 64 -> 328 against
    # round(2.5 * 100) = 250, so c4 = 32 and c2 = 68.
    counts = {2: 60, 3: 30, 4: 10}
    t = O.quanta_targets(counts, {2: 64, 3: 128, 4: 32}, 2.5, 100)
    assert t == {2: 68, 3: 0, 4: 32}


@pytest.mark.parametrize("seed", range(6))
def test_quanta_targets_are_multiples_summing_to_k(seed):
    rng = np.random.default_rng(seed)
    K = 128 * int(rng.integers(16, 40))
    cuts = np.sort(rng.integers(0, K + 1, 4))
    c = np.diff(np.concatenate([[0], cuts, [K]]))
    counts = dict(zip(O.PALETTE, (int(v) for v in c)))
    B = sum(b * v for b, v in counts.items()) / K
    t = O.quanta_targets(counts, O.GPU_QUANTA, B, K)
    assert sum(t.values()) == K
    for b in O.PALETTE:
        assert t[b] % O.GPU_QUANTA[b] == 0
        assert abs(t[b] - counts[b]) <= 2 * O.GPU_QUANTA[b]
    # the realised mean width stays within the paper's largest mismatch
    assert abs(sum(b * v for b, v in t.items()) / K - B) <= 0.045


# ---------------------------------------------------------------------------
# Section 3.3 step 2: reassignment
# ---------------------------------------------------------------------------
def _random_table(K, seed, palette=O.PALETTE):
    rng = np.random.default_rng(seed)
    return {b: rng.random(K) * (16 - b) for b in palette}


@pytest.mark.parametrize("seed", range(5))
def test_single_boundary_promotion_is_the_best_subset(seed):
    # Moving f channels from 2 to 3 bits: the chosen set must give the
    # smallest total error of all C(n, f) choices.
    K = 10
    E = _random_table(K, seed, (2, 3))
    bits = np.array([2] * 7 + [3] * 3)
    f = 3
    got = O.reassign_to_targets(bits, E, {2: 7 - f, 3: 3 + f})

    def total(bm):
        return sum(E[int(bm[k])][k] for k in range(K))

    best = None
    for sub in itertools.combinations(range(7), f):
        bm = bits.copy()
        bm[list(sub)] = 3
        v = total(bm)
        best = v if best is None else min(best, v)
    assert total(got) == pytest.approx(best, rel=0, abs=1e-12)


@pytest.mark.parametrize("seed", range(5))
def test_single_boundary_demotion_is_the_best_subset(seed):
    K = 9
    E = _random_table(K, 100 + seed, (4, 8))
    bits = np.array([4] * 3 + [8] * 6)
    f = 4
    got = O.reassign_to_targets(bits, E, {4: 3 + f, 8: 6 - f})

    def total(bm):
        return sum(E[int(bm[k])][k] for k in range(K))

    best = None
    for sub in itertools.combinations(range(3, 9), f):
        bm = bits.copy()
        bm[list(sub)] = 4
        v = total(bm)
        best = v if best is None else min(best, v)
    assert total(got) == pytest.approx(best, rel=0, abs=1e-12)


@pytest.mark.parametrize("seed", range(8))
def test_reassignment_reaches_targets_through_neighbours(seed):
    rng = np.random.default_rng(seed)
    K = 300
    bits = rng.choice(O.PALETTE, K, p=[0.4, 0.3, 0.2, 0.08, 0.02])
    E = _random_table(K, seed)
    cuts = np.sort(rng.integers(0, K + 1, 4))
    tc = np.diff(np.concatenate([[0], cuts, [K]]))
    targets = dict(zip(O.PALETTE, (int(v) for v in tc)))
    got = O.reassign_to_targets(bits, E, targets)
    for b in O.PALETTE:
        assert int(np.sum(got == b)) == targets[b]
    # a channel moves in the direction of the flow across every boundary it
    # crosses: with all flows upward no width decreases, and vice versa
    flows = np.cumsum([int(np.sum(bits == b)) - targets[b] for b in O.PALETTE])[:-1]
    if np.all(flows >= 0):
        assert np.all(got >= bits)
    if np.all(flows <= 0):
        assert np.all(got <= bits)


def test_saliency_promotions_take_the_most_salient():
    # With the saliency proxy every gain grows with saliency, so a promotion
    # 2 -> 3 takes the most salient 2-bit channels (lowest index on ties).
    sal = np.array([5.0, 1.0, 3.0, 3.0, 0.5, 9.0])
    E = O.saliency_error_table(sal, (2, 3))
    bits = np.array([2, 2, 2, 2, 2, 3])
    got = O.reassign_to_targets(bits, E, {2: 3, 3: 3})
    assert list(got) == [3, 2, 3, 2, 2, 3]


# ---------------------------------------------------------------------------
# Section 3.1: quantiser in the loop
# ---------------------------------------------------------------------------
def test_quant_error_closed_form_one_group():
    # One row, one group w = (0, 0.1, 0.2, 0.3) at 2 bits: s = fp16(0.1) =
    # 1638 / 16384, z = 0, q = (0, 1, 2, 3); the error of each channel is
    # (q*s - w)^2, multiplied by E[x^2] = (1, 2, 3, 4).
    W = np.array([[0.0, 0.1, 0.2, 0.3]], dtype=np.float32)
    x2 = np.array([1.0, 2.0, 3.0, 4.0])
    E = O.quant_error_table(W, x2, (2,))
    s = 1638.0 / 16384.0
    w = W[0].astype(np.float64)
    ref = (np.arange(4) * s - w) ** 2 * x2
    assert np.array_equal(E[2], ref)


def test_quant_error_zero_on_the_grid_and_for_16_bits():
    # Every group holds codes 0..7 times a power-of-two scale, shifted by the
    # zero point: 3-bit quantisation reproduces it exactly.
    rng = np.random.default_rng(3)
    N, K = 6, 128
    s = 2.0 ** -6
    q = rng.integers(0, 8, (N, K))
    q[:, ::64] = 0
    q[:, 1::64] = 7
    z = rng.integers(0, 8, (N, K // 64)).repeat(64, axis=1)
    W = ((q - z) * s).astype(np.float32)
    E = O.quant_error_table(W, np.ones(K), (3, 4, 16))
    assert np.all(E[3] == 0.0)
    assert np.all(E[16] == 0.0)
    assert np.any(E[4] > 0.0)  # the 4-bit grid (hi-lo)/15 misses these points


def test_quant_error_adds_over_rows():
    W, a = synth.layer_weights(40, 200, 5)
    x2 = a.astype(np.float64) ** 2
    E1 = O.quant_error_table(W, x2, (2, 4))
    E2 = O.quant_error_table(np.concatenate([W, W]), x2, (2, 4))
    for b in (2, 4):
        assert np.allclose(E2[b], 2 * E1[b], rtol=1e-14, atol=0)


def test_table_waterfilling_equals_saliency_waterfilling():
    W, a = synth.layer_weights(64, 700, 9)
    sal = O.saliency(W, a)
    for B in (2.4, 3.0, 4.1, 7.0):
        assert np.array_equal(O.allocate_from_table(O.saliency_error_table(sal), B),
                              O.allocate_bits(sal, B))


# ---------------------------------------------------------------------------
# Section 3.4: bit-specific scaling
# ---------------------------------------------------------------------------
def test_uniform_activations_keep_alpha_zero():
    # m_k = 1 for every channel: every alpha gives t = 1 and the same error,
    # and the tie goes to alpha = 0.
    W, _ = synth.layer_weights(32, 256, 4)
    a = np.full(256, 0.7, dtype=np.float32)
    bits = synth.random_codes_layer_bits(256, 4)
    alphas, t = O.choose_alphas(W, bits, a, a.astype(np.float64) ** 2)
    assert all(v == 0.0 for v in alphas.values())
    assert np.all(t == 1.0)


def test_unscaled_block_error_is_the_table_mean():
    # One width only: the block is the layer in its own order, so the
    # block's groups are the table's groups.
    W, a = synth.layer_weights(24, 300, 6)
    x2 = a.astype(np.float64) ** 2
    for b in (2, 3, 8):
        e = O.block_scaled_error(W.astype(np.float64), x2, np.ones(300), b)
        assert e == pytest.approx(float(np.mean(O.quant_error_table(W, x2, (b,))[b])),
                                  rel=1e-13)


def test_scaled_layer_computes_x_times_dequantised_scaled_weights():
    # A single-width layer: y = (x * t) Q(W / t)^T, written here with the
    # group quantiser directly instead of through the packed bytes.
    W, a = synth.layer_weights(20, 192, 8)
    bits = np.full(192, 4)
    m = O.act_metric(a)
    t = O.act_factor(m, 0.5)
    lay = O.pack_layer_scaled(W, bits, t)
    xb, x = synth.activations(a, 2, 8)
    Wq = O.dequant_rows(W.astype(np.float64) / t[None, :], 4)
    ref = (x * t[None, :]) @ Wq.T
    assert np.allclose(O.linear_scaled(lay, x), ref, rtol=1e-12, atol=1e-12)


def test_activation_factor_direction_on_hand_values():
    # Section 3.4 defines s_j = m_j^alpha and Section 3.1 packs diag(s) W and
    # multiplies the activation by 1/s.  The layer carries t = 1/s = m^-alpha:
    # m = (4, 1/4) at alpha = 1/2 gives t = (1/2, 2), so the salient channel
    # (m = 4) has its weights scaled up by 2 before quantisation.
    t = O.act_factor(np.array([4.0, 0.25]), 0.5)
    assert t.tolist() == [0.5, 2.0]
    assert O.act_factor(np.array([4.0, 0.25]), 0.0).tolist() == [1.0, 1.0]
    assert O.act_factor(np.array([16.0, 1.0]), 1.0).tolist() == [0.0625, 1.0]
    # m_k = a_k / mean(a): hand values
    assert O.act_metric(np.array([4.0, 0.25, 0.25, 0.25, 0.25, 1.0], np.float32)).tolist() == \
        [4.0, 0.25, 0.25, 0.25, 0.25, 1.0]
    assert O.act_metric(np.array([1.0, 3.0], np.float32)).tolist() == [0.5, 1.5]


# A one-row 2-bit block of six channels, built so that its scaled weights
# u_j = w_j * m_j^alpha land exactly on the 2-bit grid {0, 1, 2, 3}/8 at
# alpha = 1/2 and at no other alpha (worked by hand):
#   m = (4, 1/4, 1/4, 1/4, 1/4, 1), w = (3/16, 1/4, 1/2, 1/2, 1/4, 0).
#   u = (3/16 * 4^a, 1/4 * 4^-a, 1/2 * 4^-a, 1/2 * 4^-a, 1/4 * 4^-a, 0).
#   lo = 0, hi = max(u_0, u_2), scale = hi / 3.  Channels 1 and 2 have the
#   ratio 1/2 at every alpha, so both sit on the grid only as hi/3 and 2hi/3,
#   i.e. hi = 3 u_1 = (3/4) 4^-a; hi must also be u_0, so 4^(2a) = 4: a = 1/2.
# At alpha = 1/2 the quantised layer reproduces w exactly; at every other
# grid alpha some channel is off the grid and its error is positive.
_E8_M = np.array([4.0, 0.25, 0.25, 0.25, 0.25, 1.0], np.float32)
_E8_W = np.array([[3 / 16, 0.25, 0.5, 0.5, 0.25, 0.0]], np.float32)


def test_alpha_search_finds_the_only_exact_exponent():
    bits = np.full(6, 2)
    x2 = np.ones(6)
    alphas, t = O.choose_alphas(_E8_W, bits, _E8_M, x2)
    assert alphas == {2: 0.5}
    assert t.tolist() == [0.5, 2.0, 2.0, 2.0, 2.0, 1.0]  # original channel order
    # the packed scaled layer reproduces W exactly (dequant(Q(W/t)) * t = W)
    lay = O.pack_layer_scaled(_E8_W, bits, t)
    assert np.array_equal(O.dequant(lay) * lay["xscale"][None, :],
                          _E8_W.astype(np.float64)[:, lay["perm"]])
    # hand check of the unscaled layer (alpha = 0): lo = 0, hi = 1/2, scale =
    # fp16(1/6) = 1365/8192, zero 0; codes rint(w/scale) = (1, 2, 3, 3, 2, 0)
    # (1/4 is 1.5004 steps), so in units of 1/8192 the errors are
    # (171, 682, 1, 1, 682, 0) and the block mean is 959491 / (6 * 8192^2)
    e0 = O.block_scaled_error(_E8_W.astype(np.float64), x2, np.ones(6), 2)
    assert e0 == pytest.approx(959491.0 / (6 * 8192.0 ** 2), rel=1e-12)
    assert O.block_scaled_error(_E8_W.astype(np.float64), x2, t, 2) == 0.0


def test_alpha_search_would_fail_with_the_exponent_sign_flipped():
    # With t = m^+alpha (the flipped reading) the exact point would need
    # 4^(-2a) = 4, i.e. a = -1/2, which is off the grid: no grid alpha then
    # reproduces W.  Evaluated through the block error with t built by hand.
    x2 = np.ones(6)
    for j in range(11):
        a = j / 10
        t_flip = (_E8_M.astype(np.float64) ** a).astype(np.float32).astype(np.float64)
        assert O.block_scaled_error(_E8_W.astype(np.float64), x2, t_flip, 2) > 0.0


def test_scaling_never_raises_the_block_error():
    W, a = synth.layer_weights(48, 512, 10)
    x2 = a.astype(np.float64) ** 2
    bits = O.allocate_bits(O.saliency(W, a), 3.0)
    alphas, t = O.choose_alphas(W, bits, a, x2)
    for b, al in alphas.items():
        if b == 16:
            continue
        idx = np.where(bits == b)[0]
        e0 = O.block_scaled_error(W[:, idx].astype(np.float64), x2[idx], np.ones(len(idx)), b)
        e1 = O.block_scaled_error(W[:, idx].astype(np.float64), x2[idx], t[idx], b)
        assert e1 <= e0


# ---------------------------------------------------------------------------
# Section 5.3 (Figure 7): budget kept after snapping, padding removed
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("B", [3.0, 3.5, 4.0, 5.0, 6.0])
def test_snapped_budget_stays_within_the_papers_mismatch(B):
    W, a = synth.layer_weights(256, 2048, 1000)
    sal = O.saliency(W, a)
    bits = O.allocate_bits(sal, B)
    snapped = O.snap_to_quanta(bits, O.saliency_error_table(sal), B)
    assert abs(float(np.mean(snapped)) - B) <= 0.045  # the paper's largest mismatch
    assert O.padding_bytes_per_row(snapped) == 0
    for b in O.PALETTE:
        assert int(np.sum(snapped == b)) % O.GPU_QUANTA[b] == 0
