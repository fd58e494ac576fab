"""Pins of the oracle's graph planner (Section 4.4, traffic model of
Section 5.4): the paper's per-layer-gather baselines, hand-worked graphs,
exhaustive search on small graphs, and execution of a planned stack against
the unplanned one.  CPU only."""
import itertools

import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth

MIB = 2.0 ** 20


def _distinct_perms(hidden, ffn, qdim=None, grouped=False, seed=0):
    rng = np.random.default_rng(seed)
    perms, ids = [], {}

    def pid(l, nm):
        key = (l, {"q": "qkv", "k": "qkv", "v": "qkv", "gate": "gu", "up": "gu"}.get(nm, nm)
               if grouped else nm)
        if key not in ids:
            dim = {"o": qdim or hidden, "down": ffn}.get(nm, hidden)
            ids[key] = len(perms)
            perms.append(rng.permutation(dim))
        return ids[key]
    return perms, pid


@pytest.mark.parametrize("layers,hidden,ffn,kv,qdim,paper_mib", [
    (40, 5120, 13824, None, None, 6.80),   # Llama2-13B (§5.4)
    (64, 5120, 25600, 1024, 8192, 14.50),  # Qwen3-32B (§5.4)
])
def test_no_merge_baseline_reproduces_the_papers_traffic(layers, hidden, ffn, kv, qdim,
                                                         paper_mib):
    perms, pid = _distinct_perms(hidden, ffn, qdim)
    nodes, dims, _ = O.decoder_graph(layers, hidden, ffn, kv, pid, qdim)
    assert round(O.no_merge_traffic(nodes, dims) / MIB, 2) == paper_mib


def test_chain_of_two_linears():
    # x (8 channels, fixed natural) -> L1 -> y (6) -> L2 -> z (5) -> output.
    # {x}: L1 wants P1, the source is fixed natural: either costs 8 channels,
    # the tie goes to natural.  {y}: L1 emits L2's order for free.  {z}: the
    # output wants natural, L2 emits it for free.  Total 8 * 4 bytes.
    rng = np.random.default_rng(1)
    perms = [rng.permutation(8), rng.permutation(6)]
    nodes = [(O.NODE_SOURCE_FIXED, [], 0, -1), (O.NODE_LINEAR, [0], 1, 0),
             (O.NODE_LINEAR, [1], 2, 1), (O.NODE_BOUNDARY, [2], -1, -1)]
    labels, cost = O.plan_graph(nodes, [8, 6, 5], perms)
    assert labels == [O.NATURAL, 1, O.NATURAL] and cost == 32
    # a free source emits L1's order: nothing is shuffled
    nodes[0] = (O.NODE_SOURCE_FREE, [], 0, -1)
    labels, cost = O.plan_graph(nodes, [8, 6, 5], perms)
    assert labels == [0, 1, O.NATURAL] and cost == 0


def test_fan_out_shares_one_shuffle_per_order():
    # x (10) feeds four linears: two want P0, one P1 (equal in contents to
    # P0), one P2.  The region takes P0; one shuffle into P2 remains.
    rng = np.random.default_rng(2)
    p0, p2 = rng.permutation(10), rng.permutation(10)
    perms = [p0, p0.copy(), p2]
    nodes = [(O.NODE_SOURCE_FREE, [], 0, -1)]
    for i, pid in enumerate((0, 0, 1, 2)):
        nodes.append((O.NODE_LINEAR, [0], 1 + i, pid))
    labels, cost = O.plan_graph(nodes, [10, 3, 3, 3, 3], perms)
    assert labels[0] == 0 and cost == 40


def test_fan_in_producers_emit_the_consumers_order():
    # a = L0(x), b = L1(x), m = a * b (elementwise), L2(m): L0 and L1 emit
    # L2's order, so the product region costs nothing.
    rng = np.random.default_rng(3)
    perms = [rng.permutation(7), rng.permutation(7), rng.permutation(12)]
    nodes = [(O.NODE_SOURCE_FIXED, [], 0, -1), (O.NODE_LINEAR, [0], 1, 0),
             (O.NODE_LINEAR, [0], 2, 1), (O.NODE_ELEMENTWISE, [1, 2], 3, -1),
             (O.NODE_LINEAR, [3], 4, 2), (O.NODE_BOUNDARY, [4], -1, -1)]
    labels, cost = O.plan_graph(nodes, [7, 12, 12, 12, 9], perms)
    assert labels[1] == labels[2] == labels[3] == 2
    # x: natural (fixed) -> both linears gather: 2 shuffles of 7; P0 or P1
    # -> the source and the other linear: also 2.  Natural wins the tie.
    assert labels[0] == O.NATURAL and cost == 4 * 14


def test_grouped_query_attention_is_a_boundary_for_v():
    # v (4) and the attention output (8) differ in width: o gathers.
    perms, pid = _distinct_perms(16, 24, qdim=8)
    nodes, dims, names = O.decoder_graph(1, 16, 24, 4, pid, 8)
    labels, cost = O.plan_graph(nodes, dims, perms)
    e = names[0]
    assert labels[e["att"]] == O.NATURAL and labels[e["v"]] == O.NATURAL
    # shuffles: q, k, v inputs (h, 3 orders), o's input (8), gate, up (h2, 2)
    assert cost == 4 * (3 * 16 + 8 + 2 * 16)


def _free_cost(nodes, dims, labels, perms):
    """Cost of any labelling: a shuffle for every distinct (edge, order) that
    a consumer needs and the edge does not carry, where elementwise nodes need
    their output's order on every input and attention its output's order on v
    (equal widths), plus fixed producers off their order."""
    keys = O.basis_keys(perms)

    def k(w):
        return O.NATURAL if w == O.NATURAL else keys[w]

    need, cost = set(), 0
    for kind, ins, out, perm in nodes:
        wants = []
        if kind == O.NODE_LINEAR:
            wants = [(ins[0], k(perm))]
        elif kind == O.NODE_ELEMENTWISE:
            wants = [(e, labels[out]) for e in ins]
        elif kind == O.NODE_BOUNDARY:
            wants = [(e, O.NATURAL) for e in ins]
            if out >= 0 and labels[out] != O.NATURAL:
                cost += dims[out]
        elif kind == O.NODE_ATTENTION:
            wants = [(ins[0], O.NATURAL), (ins[1], O.NATURAL)]
            if out >= 0 and dims[ins[2]] == dims[out]:
                wants.append((ins[2], labels[out]))
            else:
                wants.append((ins[2], O.NATURAL))
                if out >= 0 and labels[out] != O.NATURAL:
                    cost += dims[out]
        elif kind == O.NODE_SOURCE_FIXED and labels[out] != O.NATURAL:
            cost += dims[out]
        for e, w in wants:
            if labels[e] != w:
                need.add((e, w))
    return 4 * (cost + sum(dims[e] for e, _ in need))


@pytest.mark.parametrize("seed", range(6))
def test_plan_is_optimal_over_every_labelling(seed):
    # A random graph of 7 edges of width 5 with three orders: the plan's cost
    # equals the minimum over all 4^7 labellings, shuffles at elementwise
    # nodes allowed.
    rng = np.random.default_rng(seed)
    perms = [rng.permutation(5) for _ in range(3)]
    nodes = [(O.NODE_SOURCE_FIXED if seed % 2 else O.NODE_SOURCE_FREE, [], 0, -1),
             (O.NODE_ELEMENTWISE, [0], 1, -1)]
    edge = 2
    avail = [0, 1]
    while edge < 7:
        kind = rng.choice([O.NODE_LINEAR, O.NODE_ELEMENTWISE, O.NODE_LINEAR])
        a = int(rng.choice(avail))
        if kind == O.NODE_LINEAR:
            nodes.append((O.NODE_LINEAR, [a], edge, int(rng.integers(0, 3))))
        else:
            b = int(rng.choice(avail))
            nodes.append((O.NODE_ELEMENTWISE, sorted({a, b}), edge, -1))
        avail.append(edge)
        edge += 1
    nodes.append((O.NODE_LINEAR, [int(rng.choice(avail))], 7, int(rng.integers(0, 3))))
    nodes.append((O.NODE_BOUNDARY, [7], -1, -1))
    dims = [5] * 7 + [3]
    labels, cost = O.plan_graph(nodes, dims, perms)
    assert cost == _free_cost(nodes, dims, labels, perms)
    best = min(_free_cost(nodes, dims, list(lab) + [O.NATURAL], perms)
               for lab in itertools.product([O.NATURAL, 0, 1, 2], repeat=7))
    assert cost == best


def _llama_stack(n_layers, hidden, ffn, seed):
    lins = []
    for l in range(n_layers):
        lin = {}
        for j, (nm, N, K) in enumerate(O.llama_layer_linears(hidden, ffn)):
            W, a = synth.layer_weights(N, K, seed + 10 * l + j)
            lin[nm] = O.pack_layer(W, a, 3.0)
        lins.append(lin)
    return lins


def test_planned_stack_equals_the_unplanned_stack_bit_for_bit():
    hidden, ffn = 64, 160
    lins = _llama_stack(2, hidden, ffn, 700)
    perms, ids = [], {}

    def pid(l, nm):
        ids[(l, nm)] = len(perms)
        perms.append(lins[l][nm]["perm"])
        return ids[(l, nm)]

    nodes, dims, names = O.decoder_graph(2, hidden, ffn, None, pid)
    labels, _ = O.plan_graph(nodes, dims, perms)
    s = np.random.default_rng(4).normal(0, 1, (2, hidden))
    s_plan = s.copy()
    s_nat = s.copy()
    for l in range(2):
        merged = O.merge_from_labels(lins[l], names[l], labels, perms)
        plain = {nm: (lins[l][nm], lins[l][nm]["perm"]) for nm, _, _ in O.DECODER_LINEAR_EDGES}
        s_plan, _ = O.decode_layer(s_plan, merged)
        s_nat, _ = O.decode_layer(s_nat, plain)
        # the plan reproduces the hand-written merge of a Llama layer
        hand = O.merge_decoder_layer(lins[l])
        for nm in merged:
            assert np.array_equal(merged[nm][0]["packed"], hand[nm][0]["packed"])
            g1, g2 = merged[nm][1], hand[nm][1]
            assert (g1 is None) == (g2 is None)
            if g1 is not None:
                assert np.array_equal(g1, g2)
    assert np.array_equal(s_plan, s_nat)


@pytest.mark.parametrize("free_source,head,shuffles,stream_label", [
    (False, None, 2, O.NATURAL),     # q/k/v and gate/up gather the natural stream
    (True, None, 2, O.NATURAL),      # a free source alone changes nothing: the
                                     # boundary still wants natural order
    (False, True, 3, O.NATURAL),     # a linear head adds its own gather
    (True, True, 2, 0),              # the stream takes q/k/v's order from the
                                     # embedding: q/k/v read it as is, gate/up
                                     # and the head gather
])
def test_free_embedding_and_linear_head_hand_worked(free_source, head, shuffles, stream_label):
    # One grouped layer: q/k/v share permutation 0, o has 1, gate/up share 2,
    # down has 3, the head 4.  The residual stream, both RMSNorm outputs and
    # the o/down outputs form one region (joined by elementwise nodes); every
    # other region is free.  Each order wanted from that region costs one
    # shuffle of 64 channels at 4 bytes (Section 5.4); worked by hand.
    rng = np.random.default_rng(9)
    perms = [rng.permutation(64), rng.permutation(64), rng.permutation(64),
             rng.permutation(160), rng.permutation(64)]
    pid = {"q": 0, "k": 0, "v": 0, "o": 1, "gate": 2, "up": 2, "down": 3}
    nodes, dims, names = O.decoder_graph(1, 64, 160, None, lambda l, nm: pid[nm], None,
                                         free_source, (4, 100) if head else None)
    labels, cost = O.plan_graph(nodes, dims, perms)
    assert cost == shuffles * 4 * 64
    assert labels[names[0]["s_in"]] == stream_label
    assert labels[names[0]["h"]] == stream_label and labels[names[0]["s2"]] == stream_label
