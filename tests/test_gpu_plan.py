"""A two-layer decode stack whose Section 4.3 merges come from the library's
Section 4.4 planner (polyq_plan_graph): the plan's edge orders become row
permutations (polyq_layer_permute_rows) and gathers (polyq_permute_merge) in
the library, the stack runs on the GPU with the fused glue, and each linear
and the stream are checked against the oracle's stack merged from the
oracle's own plan."""
import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth
from tests.gpu_util import check_tolerance

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _bf16_bits(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


def _bf16_vals(bits):
    return (bits.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


@pytest.mark.parametrize("grouped", [False, True])
def test_planned_stack_runs_on_the_gpu(polyq_lib, grouped):
    hidden, ffn, n_layers, B = 256, 640, 2, 3.0
    names_lin = [n for n, _, _ in O.llama_layer_linears(hidden, ffn)]
    hosts, refs = [], []
    perms, ids = [], {}

    def pid(l, nm):
        key = (l, {"q": "qkv", "k": "qkv", "v": "qkv", "gate": "gu", "up": "gu"}.get(nm, nm)
               if grouped else nm)
        return ids[key]

    for l in range(n_layers):
        W = {nm: synth.layer_weights(N, K, synth.seed_for(7, 10 * l + i))
             for i, (nm, N, K) in enumerate(O.llama_layer_linears(hidden, ffn))}
        if grouped:
            # q/k/v and gate/up allocated jointly; each name gets its rows of
            # the joint layer, all sharing the joint permutation
            h, r = {}, {}
            for grp, members in (("qkv", ("q", "k", "v")), ("gu", ("gate", "up"))):
                Wj = np.vstack([W[m][0] for m in members])
                r[grp] = O.pack_layer(Wj, W[members[0]][1], B)
                ids[(l, grp)] = len(perms)
                perms.append(r[grp]["perm"])
                for i, m in enumerate(members):
                    N = W[m][0].shape[0]
                    h[m] = polyq_lib.HostLayer.pack(W[m][0], W[members[0]][1], B,
                                                    forced_bits=r[grp]["bits"])
                    r[m] = O.pack_layer(W[m][0], None, B, bits=r[grp]["bits"])
            for m in ("o", "down"):
                h[m] = polyq_lib.HostLayer.pack(*W[m], B)
                r[m] = O.pack_layer(*W[m], B)
                ids[(l, m)] = len(perms)
                perms.append(r[m]["perm"])
        else:
            h = {nm: polyq_lib.HostLayer.pack(*W[nm], B) for nm in names_lin}
            r = {nm: O.pack_layer(*W[nm], B) for nm in names_lin}
            for nm in names_lin:
                ids[(l, nm)] = len(perms)
                perms.append(r[nm]["perm"])
        for nm in names_lin:
            assert np.array_equal(h[nm].export()["perm"], r[nm]["perm"].astype(np.int32))
        hosts.append(h)
        refs.append(r)

    nodes, dims, names = polyq_lib.decoder_plan_graph(n_layers, hidden, ffn, pid)
    labels, cost = polyq_lib.plan_graph(nodes, dims, perms)
    o_nodes, o_dims, o_names = O.decoder_graph(n_layers, hidden, ffn, None, pid)
    labels_o, cost_o = O.plan_graph(o_nodes, o_dims, perms)
    assert list(labels) == labels_o and cost == cost_o
    # the plan keeps the residual stream in natural order here, so the fused
    # glue (RMSNorm, SiLU * up, residual adds) runs on natural vectors
    for e in names:
        assert labels[e["s_in"]] == -1 and labels[e["h"]] == -1 and labels[e["h2"]] == -1

    def basis(lab):
        return None if lab == -1 else np.asarray(perms[lab])

    devs = []
    for l in range(n_layers):
        d = {}
        for nm, ein, eout in O.DECODER_LINEAR_EDGES:
            host = hosts[l][nm]
            bo = basis(labels[names[l][eout]])
            if bo is not None:
                host.permute_rows(bo)
            perm = host.export()["perm"]
            bi = basis(labels[names[l][ein]])
            g = perm if bi is None else polyq_lib.permute_merge(bi, perm)
            ident = np.array_equal(g, np.arange(len(g)))
            d[nm] = polyq_lib.DeviceLayer(host, "cuda", gather=None if ident else g,
                                          identity_gather=ident)
        devs.append(d)

    rng = np.random.default_rng(8)
    s0 = rng.standard_normal((1, hidden)).astype(np.float32)
    s = torch.from_numpy(s0).cuda()
    s_ref = s0.astype(np.float64)
    L = polyq_lib
    for l in range(n_layers):
        merged = O.merge_from_labels(refs[l], o_names[l], labels_o, perms)
        d = devs[l]
        h = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
        q, k, v = L.linear_gemv_input([d["q"], d["k"], d["v"]], L.X_RMSNORM, s, eps=1e-6, x_out=h)
        s_a = s.clone()
        xo = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
        L.linear_gemv_input([d["o"]], L.X_F32, v, ys=[s], residuals=[s], x_out=xo)
        s_b = s.clone()
        h2 = torch.empty((1, hidden), dtype=torch.bfloat16, device="cuda")
        g, u = L.linear_gemv_input([d["gate"], d["up"]], L.X_RMSNORM, s, eps=1e-6, x_out=h2)
        xd = torch.empty((1, ffn), dtype=torch.bfloat16, device="cuda")
        L.linear_gemv_input([d["down"]], L.X_SILU_MUL, g, b=u, ys=[s], residuals=[s], x_out=xd)
        torch.cuda.synchronize()
        hx, xox, h2x, xdx = (_bf16_vals(_bf16_bits(t)) for t in (h, xo, h2, xd))
        for nm, y, x in (("q", q, hx), ("k", k, hx), ("v", v, hx), ("gate", g, h2x),
                         ("up", u, h2x)):
            Lo, gat = merged[nm]
            want = O.linear(Lo, x, gather=gat if gat is not None else np.arange(x.shape[1]))
            check_tolerance(y.cpu().numpy(), want, x, x.shape[1])
        Lo, gat = merged["o"]
        assert gat is None  # the plan makes v emit in o's order
        check_tolerance((s_b - s_a).cpu().numpy(), O.linear(Lo, xox, gather=np.arange(hidden)),
                        xox, hidden)
        Lo, gat = merged["down"]
        assert gat is None  # and gate/up in down's
        check_tolerance((s - s_b).cpu().numpy(), O.linear(Lo, xdx, gather=np.arange(ffn)),
                        xdx, ffn)
        s_ref, _ = O.decode_layer(s_ref, merged)
    got = s.cpu().numpy().astype(np.float64)
    assert np.linalg.norm(got - s_ref) / np.linalg.norm(s_ref) <= 1e-2
