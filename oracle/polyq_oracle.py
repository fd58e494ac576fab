"""PolyQ reference oracle: a plain, slow, fp64 CPU restatement of the method.

TEST INFRASTRUCTURE ONLY.  Only ``tests/``, ``__graft_entry__.smoke()`` and the
``cpu_baseline`` / ``--impl reference`` legs of ``bench.py`` may import this
module.  The product (the C-ABI library under ``paper_2607_14618_gb300``) never
imports, links or calls it, and this module shares no code with it.

What is restated here (PolyQ, arXiv 2607.14618):

* §3.1  activation-aware per-channel error proxy (E_16 = 0); the proxy is
        instantiated from the channel saliency ``a_k * ||W[:,k]||`` (reading
        R3 below).
* §3.2  layer-wise fractional budget, the residual budget
        ``Delta = round(B*K) - b_min*K``, the gain-per-bit ``G_{b->b'}`` and the
        greedy max-heap waterfilling.
* §3.4 / §3.1 group-wise uniform quantisation at each channel's width
        (reading R1: asymmetric, fp16 scale/zero per output row per
        64-channel group; 16-bit channels stored as fp16).
* §4.1  channel permutation/clustering ``O = (A P^T)(P W)``: only the
        clustered weight is materialised; the activation is gathered.
* §4.2  bit-homogeneous blocks (one segment per width per row).
* §4.3  the merge rule ``O' = A (W P^T)(P W')``: the producer emits its
        outputs in the consumer's basis, so the consumer's gather becomes the
        identity.
* §5.4  the per-token reorder-traffic model (A16 read+write bytes of explicit
        activation shuffles).

Readings taken where the paper is silent:

R1 quantiser: per (row n, block, 64-position group of the clustered order),
   lo=min w, hi=max w, qmax=2^b-1, s=fp16_rn((hi-lo)/qmax), if s==0 then
   s=fp16_rn(max(|lo|,|hi|,2^-14)); z=clamp(rint(-lo/s),0,qmax);
   q=clamp(rint(w/s)+z,0,qmax); dequant w'=(q-z)*s.  rint = half-to-even.
   16-bit channels: w' = fp16_rn(w).  |W| must be finite and <= 65504.
R2 saliency: sal_k = a_k * sqrt(sum_n W[n,k]^2), the sum taken in fp64 in row
   order n = 0..N-1.
R3 allocation (WATERFILL_SALIENCY): E_b[k] = (sal_k/(2^b-1))^2 for b<16,
   E_16 = 0; max-heap keyed by (gain desc, channel index asc); a popped step
   that does not fit the residual budget is dropped (the channel stops).
   SALIENCY_LADDER (option): channels in descending saliency each climb the
   palette while the next step fits.
R4 permutation: blocks in ascending width; inside a block ascending channel.
R5 packing: per (row, block) an LSB-first bitstream (code p at bits
   [p*b, p*b+b), little-endian bytes), zero-padded to a multiple of 16 bytes;
   16-bit segments are little-endian fp16 padded with +0.0.  A row is the
   concatenation of its segments in block order.  meta[n][g] = (scale, zero)
   as two fp16, groups ordered by block then position.
R6 merge: a producer basis beta means emitted[i] = y_orig[beta[i]]; the
   consumer gather is r = beta^-1 o P_c, i.e. xs[p] = x_emitted[r[p]].
R13 quanta targets (§3.3): for each palette width b the candidates are the
   multiples q_b*(floor(c_b/q_b)+d), d in {-1,0,1,2}, inside [0, K]; among
   the combinations that sum to K, take the smallest |sum b*c^_b -
   round(B*K)|, then the smallest sum |c^_b - c_b|, then the
   lexicographically smallest count vector (widths ascending).  When no
   combination sums to K (K not a multiple of the quanta's gcd, or the window
   is too narrow), the narrowest width takes K minus the others' counts.
R14 reassignment (§3.3): moves only between neighbouring palette widths.  The
   net flow across boundary i (between widths w_i < w_{i+1}) is f_i =
   sum_{j<=i} (c_j - c^_j).  Upward flows are applied boundary by boundary
   from the bottom, each promoting the f_i channels of width w_i with the
   largest gain G_{w_i->w_{i+1}} (ties: lower index); then downward flows from
   the top, each demoting the |f_i| channels of width w_{i+1} with the
   smallest gain (ties: higher index).
R15 quantiser-in-the-loop proxy (§3.1, Eq. for E_b[j]): E_b[k] =
   sum_n (Q_b(W)[n,k] - W[n,k])^2 * E[x_k^2] with Q_b the R1 quantiser applied
   to the whole layer at width b, groups = 64 consecutive original channels of
   a row; E_16 = 0.  The sum over n runs in row order in fp64.
R17 graph planning (§4.4): edges carry a channel basis; linears absorb any
   input basis into their gather and emit any output basis by permuting
   rows; elementwise nodes (norms, activations, products, residual adds)
   keep one basis for all their inputs and their output; attention passes
   v's basis to its output when they have the same width (the kernel reads
   the head of each channel from the basis) and otherwise, like graph
   outputs and q/k under rotary embedding, needs the natural basis.  The
   edges joined by basis-keeping nodes form regions; each region takes the
   candidate basis (natural, or a consuming linear's permutation) with the
   smallest modelled traffic, where one explicit shuffle of an edge into a
   basis costs 4 bytes per channel (A16 read + write, §5.4) and is shared
   by every consumer of that edge wanting that basis; ties go to natural,
   then to the lowest permutation id.
R16 bit-specific scaling (§3.4): m_k = a_k / mean(a) (a = the activation
   magnitude, mean summed in channel order) and, for the channels of width b,
   the activation factor t_k = fp32_rn(m_k^-alpha_b), i.e. s_k = 1/t_k.  A
   block is quantised as Q_b(W / t) (one fp64 division per weight), so its
   effective weight is Q_b(W/t) * t, and the layer multiplies its gathered
   activation by t at each clustered position.  alpha_b is the grid value
   j/10, j = 0..10, with the smallest mean of E_b over the block's channels,
   evaluated with the block's own groups (64 consecutive clustered
   positions); ties take the smaller alpha.  A value of alpha for which some
   t_k is not finite and positive, or W/t leaves the fp16 range, is skipped
   (alpha = 0 gives t = 1 and is always allowed).
"""
from __future__ import annotations

import heapq
import itertools
import math

import numpy as np

PALETTE = (2, 3, 4, 8, 16)
GROUP = 64
FP16_MAX = 65504.0
WATERFILL_SALIENCY = 0
SALIENCY_LADDER = 1


# ---------------------------------------------------------------------------
# scalar helpers
# ---------------------------------------------------------------------------
def fp16_rn(v):
    """Round fp64 values to the nearest fp16 (ties to even), returned as fp64.

    NumPy converts float64 -> float16 directly (no float32 step), so this is a
    single correctly rounded conversion."""
    return np.asarray(v, dtype=np.float64).astype(np.float16).astype(np.float64)


def _check_weights(W):
    W = np.asarray(W)
    if W.ndim != 2:
        raise ValueError("W must be 2-D [N][K]")
    if not np.all(np.isfinite(W)) or (W.size and np.max(np.abs(W)) > FP16_MAX):
        raise ValueError("W must be finite with |W| <= 65504 (R1)")
    return W


# ---------------------------------------------------------------------------
# §3.1 (R1): group-wise asymmetric uniform quantiser
# ---------------------------------------------------------------------------
def quantize_group(w, b):
    """Quantise one group of weights (1-D, fp64) to ``b`` bits (R1, §3.1/§3.4).

    Returns (s, z, q): the fp16-representable scale and zero (as floats) and
    the integer codes."""
    w = np.asarray(w, dtype=np.float64)
    qmax = (1 << b) - 1
    lo = float(w.min())
    hi = float(w.max())
    s = float(fp16_rn((hi - lo) / qmax))
    if s == 0.0:
        s = float(fp16_rn(max(abs(lo), abs(hi), 2.0 ** -14)))
    z = float(min(max(np.rint(-lo / s), 0.0), float(qmax)))
    q = np.clip(np.rint(w / s) + z, 0.0, float(qmax)).astype(np.int64)
    return s, z, q


def quantize_rows(Wb, b):
    """Quantise a block ``Wb`` (N x K_b, fp64) group by group along columns.

    Each row and each run of 64 consecutive columns (the last run may be
    shorter) is one group.  Same arithmetic as :func:`quantize_group`,
    evaluated for all rows of a group at once.  Returns (scale[N,G],
    zero[N,G], codes[N,K_b])."""
    N, Kb = Wb.shape
    qmax = float((1 << b) - 1)
    ng = -(-Kb // GROUP)
    S = np.zeros((N, ng))
    Z = np.zeros((N, ng))
    Q = np.zeros((N, Kb), dtype=np.int64)
    for g in range(ng):
        cols = slice(g * GROUP, min((g + 1) * GROUP, Kb))
        w = Wb[:, cols]
        lo = w.min(axis=1)
        hi = w.max(axis=1)
        s = fp16_rn((hi - lo) / qmax)
        fb = s == 0.0
        if np.any(fb):
            alt = np.maximum(np.maximum(np.abs(lo), np.abs(hi)), 2.0 ** -14)
            s = np.where(fb, fp16_rn(alt), s)
        z = np.clip(np.rint(-lo / s), 0.0, qmax)
        q = np.clip(np.rint(w / s[:, None]) + z[:, None], 0.0, qmax)
        S[:, g] = s
        Z[:, g] = z
        Q[:, cols] = q.astype(np.int64)
    return S, Z, Q


# ---------------------------------------------------------------------------
# §3.1 / §3.2 (R2, R3): saliency, error proxy, greedy waterfilling
# ---------------------------------------------------------------------------
def saliency(W, act_absmean):
    """sal_k = a_k * sqrt(sum_n W[n,k]^2) in fp64, rows summed in order (R2)."""
    W = np.asarray(W)
    acc = np.zeros(W.shape[1], dtype=np.float64)
    for n in range(W.shape[0]):
        row = W[n].astype(np.float64)
        acc = acc + row * row
    return np.asarray(act_absmean, dtype=np.float64) * np.sqrt(acc)


def proxy_error(sal_k, b):
    """E_b[k] from saliency: (sal/(2^b-1))^2, and E_16 = 0 (§3.1, R3)."""
    if b == 16:
        return 0.0
    e = sal_k / float((1 << b) - 1)
    return e * e


def gain(sal_k, b, b_next):
    """Gain per extra bit G_{b->b'} = (E_b - E_b') / (b' - b) (§3.2)."""
    return (proxy_error(sal_k, b) - proxy_error(sal_k, b_next)) / float(b_next - b)


def palette_from_mask(mask):
    pal = tuple(b for b in PALETTE if mask & (1 << b))
    if not pal:
        raise ValueError("empty palette")
    return pal


def residual_budget(B, K, b_min):
    """Delta = round(B*K) - b_min*K, round half up (§3.2)."""
    return int(math.floor(B * K + 0.5)) - b_min * K


def allocate_bits(sal, B, palette=PALETTE, rule=WATERFILL_SALIENCY):
    """Per-channel widths under the average budget B (§3.2, R3).

    Every channel starts at the smallest palette width; upgrades to the next
    palette width are taken greedily by gain per bit from a max-heap until
    the residual budget is spent or no step fits."""
    sal = [float(v) for v in sal]
    K = len(sal)
    pal = tuple(sorted(palette))
    b_min = pal[0]
    nxt = {pal[i]: pal[i + 1] for i in range(len(pal) - 1)}
    bits = [b_min] * K
    delta = residual_budget(B, K, b_min)
    if delta <= 0 or len(pal) == 1:
        return np.array(bits, dtype=np.int64)
    if rule == SALIENCY_LADDER:
        order = sorted(range(K), key=lambda k: (-sal[k], k))
        for k in order:
            if delta == 0:
                break
            while bits[k] in nxt and nxt[bits[k]] - bits[k] <= delta:
                delta -= nxt[bits[k]] - bits[k]
                bits[k] = nxt[bits[k]]
        return np.array(bits, dtype=np.int64)
    heap = [(-gain(sal[k], b_min, nxt[b_min]), k, nxt[b_min]) for k in range(K)]
    heapq.heapify(heap)
    while delta > 0 and heap:
        _, k, b_new = heapq.heappop(heap)
        cost = b_new - bits[k]
        if cost > delta:
            continue  # can never fit later: Delta only shrinks
        bits[k] = b_new
        delta -= cost
        if b_new in nxt:
            heapq.heappush(heap, (-gain(sal[k], b_new, nxt[b_new]), k, nxt[b_new]))
    return np.array(bits, dtype=np.int64)


# ---------------------------------------------------------------------------
# §4.1 / §4.2 (R4, R5): permutation, blocks, packing
# ---------------------------------------------------------------------------
def cluster_perm(bits):
    """perm[p] = original channel at clustered position p (R4, §4.1)."""
    bits = np.asarray(bits)
    return np.argsort(bits, kind="stable").astype(np.int64)


def seg_bytes(b, kb):
    raw = kb * 2 if b == 16 else (kb * b + 7) // 8
    return -(-raw // 16) * 16


def make_blocks(bits):
    """Block table: one entry per width present, ascending (§4.2)."""
    bits = np.asarray(bits)
    blocks = []
    pos = 0
    off = 0
    goff = 0
    for b in PALETTE:
        kb = int(np.sum(bits == b))
        if kb == 0:
            continue
        ng = 0 if b == 16 else -(-kb // GROUP)
        sb = seg_bytes(b, kb)
        blocks.append(dict(bits=b, n_ch=kb, pos0=pos, seg_off=off,
                           seg_bytes=sb, grp_off=goff, n_grp=ng))
        pos += kb
        off += sb
        goff += ng
    return blocks, off, goff


def pack_codes(codes, b, nbytes):
    """LSB-first bitstream of ``codes`` (N x K_b) padded to ``nbytes`` (R5)."""
    N, Kb = codes.shape
    planes = (codes[:, :, None] >> np.arange(b)[None, None, :]) & 1
    stream = planes.reshape(N, Kb * b).astype(np.uint8)
    pad = nbytes * 8 - Kb * b
    stream = np.concatenate([stream, np.zeros((N, pad), np.uint8)], axis=1)
    return np.packbits(stream, axis=1, bitorder="little")


def unpack_codes_from_bytes(seg, b, kb):
    """Inverse of :func:`pack_codes` for one block segment (N x bytes)."""
    bitsarr = np.unpackbits(seg, axis=1, bitorder="little")[:, : kb * b]
    bitsarr = bitsarr.reshape(seg.shape[0], kb, b).astype(np.int64)
    return (bitsarr << np.arange(b)[None, None, :]).sum(axis=2)


def pack_layer(W, act_absmean, B, palette=PALETTE, rule=WATERFILL_SALIENCY,
               bits=None):
    """Allocation, permutation and packing of one linear layer.

    ``W`` is [N][K] (out x in) float32, ``act_absmean`` the per-input-channel
    activation magnitude.  ``bits`` may force a width map (tests).  Returns a
    dict describing the layer in the R5 format."""
    W = _check_weights(W)
    N, K = W.shape
    if bits is None:
        sal = saliency(W, act_absmean)
        bits = allocate_bits(sal, B, palette, rule)
    bits = np.asarray(bits, dtype=np.int64)
    perm = cluster_perm(bits)
    blocks, S, G = make_blocks(bits)
    packed = np.zeros((N, S), dtype=np.uint8)
    meta = np.zeros((N, G, 2), dtype=np.uint16)
    for blk in blocks:
        b, kb, p0 = blk["bits"], blk["n_ch"], blk["pos0"]
        Wb = W[:, perm[p0:p0 + kb]].astype(np.float64)
        o, sb = blk["seg_off"], blk["seg_bytes"]
        if b == 16:
            h = np.ascontiguousarray(Wb.astype(np.float16)).view("<u2").view(np.uint8)
            packed[:, o:o + h.shape[1]] = h
            continue
        sc, ze, q = quantize_rows(Wb, b)
        packed[:, o:o + sb] = pack_codes(q, b, sb)
        g0, ng = blk["grp_off"], blk["n_grp"]
        meta[:, g0:g0 + ng, 0] = sc.astype(np.float16).view(np.uint16)
        meta[:, g0:g0 + ng, 1] = ze.astype(np.float16).view(np.uint16)
    return dict(N=N, K=K, bits=bits, perm=perm, blocks=blocks, row_stride=S,
                n_groups=G, packed=packed, meta=meta,
                out_perm=np.arange(N, dtype=np.int64), B=float(B))


def realized_budget(layer):
    """B_real = mean width over the input channels (§3.3)."""
    return float(np.mean(layer["bits"]))


def unpack_codes(layer):
    """Integer codes [N][K] in clustered order from the packed bytes.

    For 16-bit positions the value is the fp16 bit pattern."""
    N, K = layer["N"], layer["K"]
    out = np.zeros((N, K), dtype=np.int64)
    for blk in layer["blocks"]:
        b, kb, p0 = blk["bits"], blk["n_ch"], blk["pos0"]
        o, sb = blk["seg_off"], blk["seg_bytes"]
        seg = layer["packed"][:, o:o + sb]
        if b == 16:
            out[:, p0:p0 + kb] = seg[:, : 2 * kb].copy().view("<u2").astype(np.int64)
        else:
            out[:, p0:p0 + kb] = unpack_codes_from_bytes(seg, b, kb)
    return out


def dequant(layer):
    """Dequantised clustered weights W'[N][K] (fp64) from the packed bytes:
    (q - z) * s for b < 16, the stored fp16 value for b = 16 (R1)."""
    N, K = layer["N"], layer["K"]
    codes = unpack_codes(layer)
    Wd = np.zeros((N, K), dtype=np.float64)
    meta = layer["meta"]
    for blk in layer["blocks"]:
        b, kb, p0 = blk["bits"], blk["n_ch"], blk["pos0"]
        c = codes[:, p0:p0 + kb]
        if b == 16:
            Wd[:, p0:p0 + kb] = c.astype(np.uint16).view(np.float16).astype(np.float64)
            continue
        g0 = blk["grp_off"]
        for g in range(blk["n_grp"]):
            cols = slice(g * GROUP, min((g + 1) * GROUP, kb))
            s = meta[:, g0 + g, 0].view(np.float16).astype(np.float64)
            z = meta[:, g0 + g, 1].view(np.float16).astype(np.float64)
            Wd[:, p0 + cols.start:p0 + cols.stop] = (c[:, cols] - z[:, None]) * s[:, None]
    return Wd


def gather_index(layer, producer_basis=None):
    """r[p]: index into the producer-emitted activation for clustered
    position p (R6).  With the natural basis this is ``perm``."""
    perm = layer["perm"]
    if producer_basis is None:
        return perm.copy()
    return permute_merge(producer_basis, perm)


def dense_layer(W, bits):
    """The clustered dequantised weights of a layer with width map ``bits``,
    computed straight from W with the R1 quantiser, block by block, without
    the bitstream (§4.1, §4.2): the same W' as ``dequant(pack_layer(W,
    bits=bits))``, for layers too large to pack here in reasonable time.
    Returns a layer dict with N, K, bits, perm, out_perm and Wd [N][K]."""
    W = _check_weights(W)
    N, K = W.shape
    bits = np.asarray(bits, dtype=np.int64)
    perm = cluster_perm(bits)
    Wd = np.zeros((N, K), dtype=np.float64)
    for blk in make_blocks(bits)[0]:
        b, kb, p0 = blk["bits"], blk["n_ch"], blk["pos0"]
        Wd[:, p0:p0 + kb] = dequant_rows(W[:, perm[p0:p0 + kb]].astype(np.float64), b)
    return dict(N=N, K=K, bits=bits, perm=perm, out_perm=np.arange(N, dtype=np.int64), Wd=Wd)


def linear(layer, x, gather=None):
    """y[b][n'] = sum_p x[b][r[p]] * W'[row(n')][p] in fp64 (§4.1, R6).

    ``x`` is [batch][K] (the activation in its producer's basis, values exact
    in fp64), ``gather`` is r (default: ``perm``, natural producer basis).
    Rows come out in the layer's current output basis (``out_perm``).  W'
    comes from the packed bytes, or from ``Wd`` for a ``dense_layer``."""
    x = np.atleast_2d(np.asarray(x, dtype=np.float64))
    r = layer["perm"] if gather is None else np.asarray(gather)
    xs = x[:, r]
    Wd = layer["Wd"] if "Wd" in layer else dequant(layer)
    return xs @ Wd.T


def linear_natural(layer, x):
    """The same product written without the permutation: W' is scattered
    back to original channel order and x is used as is (§4.1 identity)."""
    x = np.atleast_2d(np.asarray(x, dtype=np.float64))
    Wc = dequant(layer)
    Wn = np.zeros_like(Wc)
    Wn[:, layer["perm"]] = Wc
    return x @ Wn.T


# ---------------------------------------------------------------------------
# §4.3 (R6): permutation merge
# ---------------------------------------------------------------------------
def _check_perm(p, n):
    p = np.asarray(p, dtype=np.int64)
    if p.shape != (n,) or not np.array_equal(np.sort(p), np.arange(n)):
        raise ValueError("not a permutation of 0..n-1")
    return p


def permute_merge(producer_basis, consumer_perm):
    """r = beta^-1 o P_c: r[p] = beta^-1[consumer_perm[p]] (§4.3, R6)."""
    n = len(consumer_perm)
    beta = _check_perm(producer_basis, n)
    pc = _check_perm(consumer_perm, n)
    inv = np.empty(n, dtype=np.int64)
    inv[beta] = np.arange(n)
    return inv[pc]


def permute_rows(layer, row_perm):
    """Make the layer emit output i = y_orig[out_perm[row_perm[i]]] by moving
    whole packed rows and their metadata (§4.3: compile-time permutation of
    the producer's output channels)."""
    rp = _check_perm(row_perm, layer["N"])
    out = dict(layer)
    for key in ("packed", "meta", "Wd"):
        if key in layer:
            out[key] = layer[key][rp].copy()
    out["out_perm"] = layer["out_perm"][rp].copy()
    return out


# ---------------------------------------------------------------------------
# §5.4: reorder-traffic model
# ---------------------------------------------------------------------------
def reorder_traffic_bytes(gathered_k, n_layers):
    """Per-token A16 read+write bytes of explicit activation shuffles: each
    shuffled activation of K channels costs 2 bytes read + 2 bytes written
    per channel (§5.4)."""
    return 4 * int(sum(gathered_k)) * int(n_layers)


def llama_layer_linears(hidden, ffn):
    """(name, N, K) of the seven linears of one Llama-style decoder layer."""
    return [("q", hidden, hidden), ("k", hidden, hidden), ("v", hidden, hidden),
            ("o", hidden, hidden), ("gate", ffn, hidden), ("up", ffn, hidden),
            ("down", hidden, ffn)]


# ---------------------------------------------------------------------------
# decode-step reference for a Llama-shaped stack (the per-layer graph)
# ---------------------------------------------------------------------------
def bf16_rn(v):
    """Round fp64 to bf16 (ties to even) via fp32, returned as fp64.

    Used only where the decode-step graph stores an activation in bf16; the
    fp64 -> fp32 -> bf16 order is the graph's definition, not a shortcut."""
    f = np.asarray(v, dtype=np.float64).astype(np.float32)
    u = f.view(np.uint32).astype(np.uint64)
    r = ((u + 0x7FFF + ((u >> 16) & 1)) >> 16) << 16
    return r.astype(np.uint32).view(np.float32).astype(np.float64)


def rmsnorm(s, eps=1e-6):
    """RMSNorm with unit gain over the last axis: s / sqrt(mean(s^2) + eps)."""
    s = np.asarray(s, dtype=np.float64)
    return s / np.sqrt(np.mean(s * s, axis=-1, keepdims=True) + eps)


def silu(v):
    """SiLU: v * sigmoid(v) = v / (1 + exp(-v))."""
    v = np.asarray(v, dtype=np.float64)
    return v / (1.0 + np.exp(-v))


def row_slice(layer, r0, r1):
    """Rows [r0, r1) of a packed layer as a layer of their own (same channel
    permutation and blocks): a jointly allocated stack of linears, split."""
    out = dict(layer)
    for key in ("packed", "meta", "Wd"):
        if key in layer:
            out[key] = layer[key][r0:r1].copy()
    out["out_perm"] = np.arange(r1 - r0, dtype=np.int64)
    out["N"] = r1 - r0
    return out


def merge_decoder_layer(lin):
    """Apply the §4.3 merges of one decoder layer (reading R11): v emits in
    o's input basis and gate/up emit in down's, so o and down read their
    input without a gather; q, k, v, gate and up gather the natural-basis
    stream.  ``lin`` maps q, k, v, o, gate, up, down to packed layers; the
    result maps each name to (layer, gather) with gather None for identity."""
    out = {}
    for name in ("q", "k"):
        out[name] = (lin[name], lin[name]["perm"])
    out["v"] = (permute_rows(lin["v"], lin["o"]["perm"]), lin["v"]["perm"])
    out["o"] = (lin["o"], None)
    for name in ("gate", "up"):
        out[name] = (permute_rows(lin[name], lin["down"]["perm"]), lin[name]["perm"])
    out["down"] = (lin["down"], None)
    return out


def _linear_g(layer_gather, x):
    layer, gather = layer_gather
    g = np.arange(layer["K"]) if gather is None else gather
    return linear(layer, x, gather=g)


def decode_layer(s, merged, eps=1e-6):
    """One decode step of a Llama-shaped layer at position 0 (reading R11):
    h = bf16(rmsnorm(s)); q, k, v from h; attention over the single cached
    key returns v, so s += o(bf16(v)); h2 = bf16(rmsnorm(s)); s +=
    down(bf16(silu(gate(h2)) * up(h2))).  s is the fp32/fp64 residual stream
    in the natural basis; ``merged`` comes from merge_decoder_layer.  Returns
    the new stream and the intermediate values by name."""
    s = np.asarray(s, dtype=np.float64)
    h = bf16_rn(rmsnorm(s, eps))
    q = _linear_g(merged["q"], h)
    k = _linear_g(merged["k"], h)
    v = _linear_g(merged["v"], h)
    xo = bf16_rn(v)
    s1 = s + _linear_g(merged["o"], xo)
    h2 = bf16_rn(rmsnorm(s1, eps))
    g = _linear_g(merged["gate"], h2)
    u = _linear_g(merged["up"], h2)
    xd = bf16_rn(silu(g) * u)
    s2 = s1 + _linear_g(merged["down"], xd)
    return s2, dict(h=h, q=q, k=k, v=v, xo=xo, s1=s1, h2=h2, gate=g, up=u, xd=xd)


# ---------------------------------------------------------------------------
# §3.1 full proxy (R15), §3.2 waterfilling on an error table, §3.3 quanta
# matching (R13, R14), §3.4 bit-specific scaling (R16)
# ---------------------------------------------------------------------------
GPU_QUANTA = {2: 64, 3: 128, 4: 32, 8: 16, 16: 8}
"""Channels per quantum: one quantum of each width is a whole number of
16-byte chunks (64x2, 128x3, 32x4, 16x8 and 8x16 bits), so blocks whose sizes
are multiples of these need no segment padding."""

ALPHA_GRID = tuple(j / 10.0 for j in range(11))


def saliency_error_table(sal, palette=PALETTE):
    """E[b] = array over channels of the saliency proxy (R3)."""
    return {b: np.array([proxy_error(float(v), b) for v in sal]) for b in palette}


def _col_sq_err(Wq, W):
    """sum_n (Wq[n,k] - W[n,k])^2 for each k, rows added in order, fp64."""
    acc = np.zeros(W.shape[1], dtype=np.float64)
    for n in range(W.shape[0]):
        d = Wq[n] - W[n]
        acc = acc + d * d
    return acc


def dequant_rows(Wb, b):
    """Q_b applied to the columns of ``Wb`` (N x K_b, fp64) in groups of 64
    consecutive columns (R1), dequantised: (q - z) * s, fp16(w) for b = 16."""
    if b == 16:
        return fp16_rn(Wb)
    S, Z, Q = quantize_rows(Wb, b)
    out = np.zeros_like(Wb)
    for g in range(S.shape[1]):
        cols = slice(g * GROUP, min((g + 1) * GROUP, Wb.shape[1]))
        out[:, cols] = (Q[:, cols] - Z[:, g][:, None]) * S[:, g][:, None]
    return out


def quant_error_table(W, act_sqmean, palette=PALETTE):
    """Quantiser-in-the-loop proxy (§3.1 channel-error equation, R15):
    E[b][k] = ||Q_b(W)[:,k] - W[:,k]||^2 * E[x_k^2], the whole layer quantised
    at width b with groups of 64 consecutive original channels; E[16] = 0."""
    W = _check_weights(W).astype(np.float64)
    x2 = np.asarray(act_sqmean, dtype=np.float64)
    E = {}
    for b in palette:
        if b == 16:
            E[b] = np.zeros(W.shape[1])
        else:
            E[b] = _col_sq_err(dequant_rows(W, b), W) * x2
    return E


def allocate_from_table(E, B, palette=PALETTE):
    """§3.2 waterfilling with the gains of an error table: all channels start
    at the narrowest width, Delta = round(B*K) - b_min*K, and the max-heap of
    (gain per bit desc, channel asc) hands out upgrades to the next palette
    width while they fit (a step that does not fit is dropped)."""
    pal = tuple(sorted(palette))
    K = len(E[pal[0]])
    b_min = pal[0]
    nxt = {pal[i]: pal[i + 1] for i in range(len(pal) - 1)}
    bits = [b_min] * K
    delta = residual_budget(B, K, b_min)
    if delta <= 0 or len(pal) == 1:
        return np.array(bits, dtype=np.int64)

    def g(k, b, bn):
        return (float(E[b][k]) - float(E[bn][k])) / float(bn - b)

    heap = [(-g(k, b_min, nxt[b_min]), k, nxt[b_min]) for k in range(K)]
    heapq.heapify(heap)
    while delta > 0 and heap:
        _, k, b_new = heapq.heappop(heap)
        cost = b_new - bits[k]
        if cost > delta:
            continue
        bits[k] = b_new
        delta -= cost
        if b_new in nxt:
            heapq.heappush(heap, (-g(k, b_new, nxt[b_new]), k, nxt[b_new]))
    return np.array(bits, dtype=np.int64)


def quanta_targets(counts, quanta, B, K):
    """§3.3 first step (R13): block sizes that are multiples of the quanta,
    near the waterfilling counts, summing to K, budget kept closest to
    round(B*K).  ``counts`` maps every palette width to its channel count."""
    widths = sorted(counts)
    T = int(math.floor(B * K + 0.5))
    cand = []
    for b in widths:
        q = int(quanta[b])
        base = int(counts[b]) // q
        cand.append(sorted({q * (base + d) for d in (-1, 0, 1, 2) if 0 <= q * (base + d) <= K}))

    def key(combo):
        tb = sum(b * c for b, c in zip(widths, combo))
        mv = sum(abs(c - int(counts[b])) for b, c in zip(widths, combo))
        return (abs(tb - T), mv, tuple(combo))

    best = None
    for combo in itertools.product(*cand):
        if sum(combo) != K:
            continue
        k = key(combo)
        if best is None or k < best:
            best = k
    if best is None:
        # the narrowest width fills the remainder
        for rest in itertools.product(*cand[1:]):
            c0 = K - sum(rest)
            if c0 < 0:
                continue
            k = key((c0,) + tuple(rest))
            if best is None or k < best:
                best = k
    return {b: int(c) for b, c in zip(widths, best[2])}


def reassign_to_targets(bits, E, targets):
    """§3.3 second step (R14): move channels between neighbouring widths until
    the per-width counts equal ``targets``; promotions take the largest gain
    per bit, demotions the smallest."""
    bits = np.array(bits, dtype=np.int64)
    pal = sorted(targets)
    m = len(pal)
    cur = [int(np.sum(bits == b)) for b in pal]
    flow = []
    acc = 0
    for i in range(m - 1):
        acc += cur[i] - int(targets[pal[i]])
        flow.append(acc)

    def g(k, i):
        b, bn = pal[i], pal[i + 1]
        return (float(E[b][k]) - float(E[bn][k])) / float(bn - b)

    for i in range(m - 1):  # upward flows, bottom-up
        if flow[i] > 0:
            members = [k for k in range(len(bits)) if bits[k] == pal[i]]
            members.sort(key=lambda k: (-g(k, i), k))
            for k in members[:flow[i]]:
                bits[k] = pal[i + 1]
    for i in reversed(range(m - 1)):  # downward flows, top-down
        if flow[i] < 0:
            members = [k for k in range(len(bits)) if bits[k] == pal[i + 1]]
            members.sort(key=lambda k: (g(k, i), -k))
            for k in members[:-flow[i]]:
                bits[k] = pal[i]
    return bits


def snap_to_quanta(bits, E, B, quanta=None, palette=PALETTE):
    """Quanta matching (§3.3): R13 targets, then R14 reassignment."""
    quanta = GPU_QUANTA if quanta is None else quanta
    bits = np.asarray(bits, dtype=np.int64)
    K = len(bits)
    counts = {b: int(np.sum(bits == b)) for b in palette}
    t = quanta_targets(counts, quanta, B, K)
    return reassign_to_targets(bits, E, t)


def padding_bytes_per_row(bits):
    """Segment padding of one packed row: sum over blocks of the padded
    segment bytes minus the bytes the codes need (R5)."""
    bits = np.asarray(bits)
    pad = 0
    for b in PALETTE:
        kb = int(np.sum(bits == b))
        if kb:
            raw = kb * 2 if b == 16 else (kb * b + 7) // 8
            pad += seg_bytes(b, kb) - raw
    return pad


def act_metric(act_absmean):
    """m_k = a_k / mean(a), the mean summed in channel order (R16)."""
    a = np.asarray(act_absmean, dtype=np.float64)
    tot = 0.0
    for v in a:
        tot = tot + float(v)
    return a / (tot / len(a))


def act_factor(m, alpha):
    """t_k = fp32_rn(m_k^-alpha) (R16); None when some t_k is unusable."""
    with np.errstate(divide="ignore", over="ignore", invalid="ignore"):
        t = np.power(np.asarray(m, dtype=np.float64), -float(alpha))
    t = t.astype(np.float32).astype(np.float64)
    if not np.all(np.isfinite(t)) or np.any(t <= 0.0):
        return None
    return t


def block_scaled_error(Wb, x2b, tb, b):
    """Mean over the block's channels of ||Q_b(Wb/t)*t - Wb||^2 * E[x^2]
    (R16), the block's groups being 64 consecutive clustered columns.  None
    when Wb/t leaves the fp16 range."""
    Ws = Wb / tb[None, :]
    if np.max(np.abs(Ws)) > FP16_MAX:
        return None
    We = dequant_rows(Ws, b) * tb[None, :]
    e = _col_sq_err(We, Wb) * x2b
    tot = 0.0
    for v in e:
        tot = tot + float(v)
    return tot / len(e)


def choose_alphas(W, bits, act_absmean, act_sqmean, grid=ALPHA_GRID):
    """§3.4 grid search (R16): per width present, the alpha with the smallest
    mean scaled proxy error over the block; returns (alpha by width, t[K] in
    original channel order)."""
    W = _check_weights(W).astype(np.float64)
    bits = np.asarray(bits, dtype=np.int64)
    perm = cluster_perm(bits)
    m = act_metric(act_absmean)
    x2 = np.asarray(act_sqmean, dtype=np.float64)
    t_all = np.ones(len(bits))
    alphas = {}
    for b in PALETTE:
        idx = perm[bits[perm] == b]
        if len(idx) == 0:
            continue
        if b == 16:
            alphas[b] = 0.0  # E_16 = 0 for every alpha: the smallest wins
            continue
        best = None
        for a in grid:
            tb = act_factor(m[idx], a)
            if tb is None:
                continue
            e = block_scaled_error(W[:, idx], x2[idx], tb, b)
            if e is None:
                continue
            if best is None or e < best[0]:
                best = (e, a, tb)
        alphas[b] = best[1]
        t_all[idx] = best[2]
    return alphas, t_all


def pack_layer_scaled(W, bits, t):
    """Pack W / t (R16) with the width map ``bits``; the layer carries the
    activation factors ``xscale`` in clustered order."""
    W = _check_weights(W).astype(np.float64)
    t = np.asarray(t, dtype=np.float64)
    lay = pack_layer(W / t[None, :], None, 0.0, bits=bits)
    lay["xscale"] = t[lay["perm"]]
    return lay


def linear_scaled(layer, x, gather=None):
    """y[b][n'] = sum_p x[b][r[p]] * t[p] * W'[row(n')][p] (R16, fp64)."""
    x = np.atleast_2d(np.asarray(x, dtype=np.float64))
    r = layer["perm"] if gather is None else np.asarray(gather)
    xs = x[:, r] * layer["xscale"][None, :]
    return xs @ dequant(layer).T


# ---------------------------------------------------------------------------
# §4.4 graph-based permutation planning (R17)
# ---------------------------------------------------------------------------
NODE_SOURCE_FIXED = 0   # emits its edge in the natural basis
NODE_SOURCE_FREE = 1    # emits in any basis at no cost (e.g. a permuted embedding)
NODE_LINEAR = 2         # ins = [x]; absorbs its input basis, emits any basis
NODE_ELEMENTWISE = 3    # ins and out share one basis (norm, activation, product, add)
NODE_BOUNDARY = 4       # ins need the natural basis; out (if any) is natural
NODE_ATTENTION = 5      # ins = [q, k, v]: q, k natural; out keeps v's basis if widths match
NATURAL = -1


def _basis_joins(nodes, edge_dims):
    """Pairs of edges that one node forces into the same basis (R17)."""
    joins = []
    for kind, ins, out, _ in nodes:
        if kind == NODE_ELEMENTWISE:
            for e in ins:
                joins.append((e, out))
        elif kind == NODE_ATTENTION and out >= 0 and edge_dims[ins[2]] == edge_dims[out]:
            joins.append((ins[2], out))
    return joins


def plan_regions(nodes, edge_dims):
    """Region id of every edge: connected components of the basis joins."""
    n = len(edge_dims)
    parent = list(range(n))

    def find(i):
        while parent[i] != i:
            i = parent[i]
        return i

    for a, b in _basis_joins(nodes, edge_dims):
        ra, rb = find(a), find(b)
        if ra != rb:
            parent[max(ra, rb)] = min(ra, rb)
    return [find(i) for i in range(n)]


def _requests(nodes, edge_dims):
    """(edge, wanted basis) pairs: what each consumer needs to read without a
    shuffle, and the fixed bases producers emit."""
    want = []   # (edge, basis) consumers
    fixed = []  # (edge, basis) producers that cannot choose
    for kind, ins, out, perm in nodes:
        if kind == NODE_LINEAR:
            want.append((ins[0], perm))
        elif kind == NODE_BOUNDARY:
            want.extend((e, NATURAL) for e in ins)
            if out >= 0:
                fixed.append((out, NATURAL))
        elif kind == NODE_ATTENTION:
            want.append((ins[0], NATURAL))
            want.append((ins[1], NATURAL))
            if out >= 0 and edge_dims[ins[2]] != edge_dims[out]:
                want.append((ins[2], NATURAL))
                fixed.append((out, NATURAL))
        elif kind == NODE_SOURCE_FIXED:
            fixed.append((out, NATURAL))
    return want, fixed


def basis_keys(perms):
    """key[i]: NATURAL if permutation i is the identity, else the smallest id
    whose permutation has the same contents (equal bases compare equal)."""
    keys, seen = [], {}
    for i, p in enumerate(perms):
        p = np.asarray(p)
        if np.array_equal(p, np.arange(len(p))):
            keys.append(NATURAL)
            continue
        t = tuple(int(v) for v in p)
        keys.append(seen.setdefault(t, i))
    return keys


def _key(keys, w):
    return NATURAL if w == NATURAL else keys[w]


def plan_cost(nodes, edge_dims, labels, perms, only_region=None, region=None, keys=None):
    """Modelled bytes per token of the explicit shuffles a labelling needs
    (R17): one shuffle per distinct (edge, wanted basis) that differs from
    the edge's label, and one per fixed producer whose basis differs;
    optionally only for the edges of one region."""
    keys = basis_keys(perms) if keys is None else keys
    want, fixed = _requests(nodes, edge_dims)
    if only_region is not None:
        want = [(e, w) for e, w in want if region[e] == only_region]
        fixed = [(e, w) for e, w in fixed if region[e] == only_region]
    need = set()
    for e, w in want:
        if _key(keys, labels[e]) != _key(keys, w):
            need.add((e, _key(keys, w)))
    cost = 4 * sum(edge_dims[e] for e, _ in need)
    for e, w in fixed:
        if _key(keys, labels[e]) != _key(keys, w):
            cost += 4 * edge_dims[e]
    return cost


def plan_graph(nodes, edge_dims, perms):
    """§4.4 planning (R17): the basis label of every edge.  ``nodes`` are
    (kind, inputs, output edge or -1, permutation id or -1), ``perms[i]``
    a linear's preferred input order (its clustering permutation).  Returns
    (labels, modelled bytes per token)."""
    keys = basis_keys(perms)
    region = plan_regions(nodes, edge_dims)
    want, _ = _requests(nodes, edge_dims)
    labels = [NATURAL] * len(edge_dims)
    for r in sorted(set(region)):
        edges = [e for e in range(len(edge_dims)) if region[e] == r]
        cands = [NATURAL] + sorted({keys[w] for e, w in want
                                    if region[e] == r and w != NATURAL and keys[w] != NATURAL})
        best = None
        for c in cands:
            for e in edges:
                labels[e] = c
            cost = plan_cost(nodes, edge_dims, labels, perms, only_region=r, region=region,
                             keys=keys)
            if best is None or cost < best[0]:
                best = (cost, c)
        for e in edges:
            labels[e] = best[1]
    return labels, plan_cost(nodes, edge_dims, labels, perms, keys=keys)


def no_merge_traffic(nodes, edge_dims):
    """The per-layer-gather baseline of §5.4: every linear input shuffled."""
    return 4 * sum(edge_dims[i[0]] for k, i, o, p in nodes if k == NODE_LINEAR)


def decoder_graph(n_layers, hidden, ffn, kv=None, perm_ids=None, qdim=None, free_source=False,
                  head=None):
    """The decode graph of a Llama/Qwen-style stack (R11 per layer, R17
    kinds): nodes, edge widths and, per layer, the edge ids by name.  ``qdim``
    is the width of q and of the attention output (heads x head width,
    default ``hidden``), ``kv`` the k/v width (grouped-query attention when
    below ``qdim``);
    ``perm_ids(layer, name)`` gives each linear's permutation id.  By default
    the stream enters from a fixed natural source and leaves through a
    boundary (the output head reads natural order).  ``free_source``: the
    stream enters from an embedding table whose columns may be permuted at
    compile time (any order, no cost).  ``head = (perm id, vocab)``: the
    stream ends in a final RMSNorm and an output head that is itself a linear
    (it reads any order through its gather), whose logits leave through a
    boundary."""
    qdim = hidden if qdim is None else qdim
    kv = qdim if kv is None else kv
    nodes, dims, names = [], [], []

    def edge(d):
        dims.append(d)
        return len(dims) - 1

    s = edge(hidden)
    nodes.append((NODE_SOURCE_FREE if free_source else NODE_SOURCE_FIXED, [], s, -1))
    for l in range(n_layers):
        e = {}
        e["h"] = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [s], e["h"], -1))           # RMSNorm
        for nm, w in (("q", qdim), ("k", kv), ("v", kv)):
            e[nm] = edge(w)
            nodes.append((NODE_LINEAR, [e["h"]], e[nm], perm_ids(l, nm)))
        e["att"] = edge(qdim)
        nodes.append((NODE_ATTENTION, [e["q"], e["k"], e["v"]], e["att"], -1))
        e["o"] = edge(hidden)
        nodes.append((NODE_LINEAR, [e["att"]], e["o"], perm_ids(l, "o")))
        e["s1"] = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [s, e["o"]], e["s1"], -1))  # residual add
        e["h2"] = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [e["s1"]], e["h2"], -1))    # RMSNorm
        for nm in ("gate", "up"):
            e[nm] = edge(ffn)
            nodes.append((NODE_LINEAR, [e["h2"]], e[nm], perm_ids(l, nm)))
        e["m"] = edge(ffn)
        nodes.append((NODE_ELEMENTWISE, [e["gate"], e["up"]], e["m"], -1))  # SiLU * up
        e["down"] = edge(hidden)
        nodes.append((NODE_LINEAR, [e["m"]], e["down"], perm_ids(l, "down")))
        e["s2"] = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [e["s1"], e["down"]], e["s2"], -1))
        e["s_in"] = s
        names.append(e)
        s = e["s2"]
    if head is None:
        nodes.append((NODE_BOUNDARY, [s], -1, -1))
    else:
        hf = edge(hidden)
        nodes.append((NODE_ELEMENTWISE, [s], hf, -1))    # final RMSNorm
        logits = edge(head[1])
        nodes.append((NODE_LINEAR, [hf], logits, head[0]))
        nodes.append((NODE_BOUNDARY, [logits], -1, -1))
    return nodes, dims, names


DECODER_LINEAR_EDGES = (("q", "h", "q"), ("k", "h", "k"), ("v", "h", "v"), ("o", "att", "o"),
                        ("gate", "h2", "gate"), ("up", "h2", "up"), ("down", "m", "down"))
"""(linear, input edge, output edge) of one layer of ``decoder_graph``."""


def merge_from_labels(lin, edges, labels, perms):
    """The §4.3 merges a plan implies for one decoder layer (R17): each
    linear's rows are permuted to its output edge's basis and it gathers from
    its input edge's basis (gather None where that is its own order).
    ``lin`` maps names to packed layers, ``edges`` is the layer's entry of
    ``decoder_graph``'s names, ``labels`` and ``perms`` come from
    ``plan_graph``; the result has merge_decoder_layer's form."""
    def basis(e):
        lab = labels[e]
        return None if lab == NATURAL else np.asarray(perms[lab])

    out = {}
    for nm, ein, eout in DECODER_LINEAR_EDGES:
        L = lin[nm]
        bo = basis(edges[eout])
        if bo is not None:
            L = permute_rows(L, bo)
        bi = basis(edges[ein])
        g = L["perm"] if bi is None else permute_merge(bi, L["perm"])
        if np.array_equal(g, np.arange(len(g))):
            g = None
        out[nm] = (L, g)
    return out
