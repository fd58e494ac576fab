"""The library's graph planner (C++) against the oracle's: labels and
modelled traffic equal on random graphs and on the Llama2-13B and Qwen3-32B
decode graphs, plus argument validation.  CPU only."""
import numpy as np
import pytest

from oracle import polyq_oracle as O


def _random_graph(seed):
    rng = np.random.default_rng(seed)
    widths = [6, 9, 4]
    perms_by_w = {w: [rng.permutation(w) for _ in range(3)] for w in widths}
    perms, pid_of = [], {}
    for w in widths:
        for i, p in enumerate(perms_by_w[w]):
            pid_of[(w, i)] = len(perms)
            perms.append(p)
    perms.append(np.arange(6))  # an identity permutation counts as natural
    pid_of[(6, 3)] = len(perms) - 1
    perms.append(perms_by_w[9][0].copy())  # equal contents, another id
    pid_of[(9, 3)] = len(perms) - 1
    nodes, dims = [], []

    def edge(w):
        dims.append(w)
        return len(dims) - 1

    avail = []
    for _ in range(2):
        w = int(rng.choice(widths))
        e = edge(w)
        nodes.append((int(rng.choice([O.NODE_SOURCE_FIXED, O.NODE_SOURCE_FREE])), [], e, -1))
        avail.append(e)
    for _ in range(int(rng.integers(8, 20))):
        kind = int(rng.choice([O.NODE_LINEAR, O.NODE_LINEAR, O.NODE_ELEMENTWISE,
                               O.NODE_BOUNDARY, O.NODE_ATTENTION]))
        a = int(rng.choice(avail))
        if kind == O.NODE_LINEAR:
            w_in = dims[a]
            e = edge(int(rng.choice(widths)))
            nodes.append((kind, [a], e, pid_of[(w_in, int(rng.integers(0, 4 if w_in in (6, 9) else 3)))]))
        elif kind == O.NODE_ELEMENTWISE:
            same = [x for x in avail if dims[x] == dims[a]]
            ins = sorted({a, int(rng.choice(same))})
            e = edge(dims[a])
            nodes.append((kind, ins, e, -1))
        elif kind == O.NODE_BOUNDARY:
            e = edge(int(rng.choice(widths))) if rng.random() < 0.5 else -1
            nodes.append((kind, [a], e, -1))
        else:
            q, k, v = (int(rng.choice(avail)) for _ in range(3))
            e = edge(dims[v] if rng.random() < 0.6 else int(rng.choice(widths)))
            nodes.append((kind, [q, k, v], e, -1))
        if nodes[-1][2] >= 0:
            avail.append(nodes[-1][2])
    return nodes, dims, perms


@pytest.mark.parametrize("seed", range(25))
def test_planner_matches_oracle_on_random_graphs(polyq_lib, seed):
    nodes, dims, perms = _random_graph(seed)
    lo, co = O.plan_graph(nodes, dims, perms)
    lc, cc = polyq_lib.plan_graph(nodes, dims, perms)
    assert list(lc) == lo and cc == co


@pytest.mark.parametrize("layers,hidden,ffn,kv,qdim,grouped", [
    (40, 5120, 13824, None, None, False),
    (40, 5120, 13824, None, None, True),
    (64, 5120, 25600, 1024, 8192, True),
])
def test_planner_matches_oracle_on_decoder_graphs(polyq_lib, layers, hidden, ffn, kv, qdim,
                                                  grouped):
    rng = np.random.default_rng(layers)
    perms, ids = [], {}

    def pid(l, nm):
        key = (l, {"q": "qkv", "k": "qkv", "v": "qkv", "gate": "gu", "up": "gu"}.get(nm, nm)
               if grouped else nm)
        if key not in ids:
            ids[key] = len(perms)
            perms.append(rng.permutation({"o": qdim or hidden, "down": ffn}.get(nm, hidden)))
        return ids[key]

    nodes, dims, _ = O.decoder_graph(layers, hidden, ffn, kv, pid, qdim)
    lo, co = O.plan_graph(nodes, dims, perms)
    lc, cc = polyq_lib.plan_graph(nodes, dims, perms)
    assert list(lc) == lo and cc == co
    # the same stack entered from a free-order embedding and left through a
    # linear output head
    perms.append(rng.permutation(hidden))
    nodes, dims, _ = O.decoder_graph(layers, hidden, ffn, kv, pid, qdim, True,
                                     (len(perms) - 1, 32000))
    lo, co = O.plan_graph(nodes, dims, perms)
    lc, cc = polyq_lib.plan_graph(nodes, dims, perms)
    assert list(lc) == lo and cc == co


def test_planner_rejects_bad_graphs(polyq_lib):
    p = [np.arange(4)[::-1].copy()]
    bad = [
        ([(O.NODE_LINEAR, [0], 1, 0)], [5, 3], p),           # permutation width != input
        ([(O.NODE_ELEMENTWISE, [0], 1, -1)], [4, 3], p),     # elementwise width change
        ([(9, [], 0, -1)], [4], p),                           # unknown kind
        ([(O.NODE_LINEAR, [0], 1, 3)], [4, 3], p),            # no such permutation
        ([(O.NODE_LINEAR, [0], 7, 0)], [4, 3], p),            # no such edge
        ([(O.NODE_SOURCE_FREE, [], 0, -1), (O.NODE_SOURCE_FREE, [], 0, -1)], [4], p),
        ([(O.NODE_LINEAR, [0], 1, 0)], [4, 3], [np.array([0, 0, 1, 2])]),  # not a permutation
        ([(O.NODE_ATTENTION, [0, 0], 1, -1)], [4, 4], p),
    ]
    for nodes, dims, perms in bad:
        with pytest.raises(polyq_lib.PolyqError) as ei:
            polyq_lib.plan_graph(nodes, dims, perms)
        assert ei.value.code == polyq_lib.POLYQ_EINVAL


def test_library_decoder_graph_matches_oracle_graph(polyq_lib):
    def pid(l, nm):
        return 7 * l + ["q", "k", "v", "o", "gate", "up", "down"].index(nm)
    for args in ((3, 64, 160, None, None, False, None), (2, 64, 160, 16, 96, False, None),
                 (2, 64, 160, None, None, True, (14, 500)), (1, 64, 160, 16, 96, False, (7, 9))):
        n1, d1, e1 = polyq_lib.decoder_plan_graph(args[0], args[1], args[2], pid, args[3], args[4],
                                                  args[5], args[6])
        n2, d2, e2 = O.decoder_graph(args[0], args[1], args[2], args[3], pid, args[4], args[5],
                                     args[6])
        assert [(k, list(i), o, p) for k, i, o, p in n1] == [(k, list(i), o, p) for k, i, o, p in n2]
        assert list(d1) == list(d2) and e1 == e2
