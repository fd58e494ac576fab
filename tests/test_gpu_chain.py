"""GPU parity of the chained persistent GEMV (polyq_linear_gemv_chain):
decoder layers as dependent phases against the oracle and against the
per-call path, independent phases against the oracle at every batch size,
and a phase with more activation records than CTAs.  All calls go through the
C ABI."""
import numpy as np
import pytest

from oracle import polyq_oracle as O
from paper_2607_14618_gb300 import synth
from tests.gpu_util import check_tolerance, rel_l2

torch = pytest.importorskip("torch")
pytestmark = pytest.mark.gpu


def _x_dev(xb):
    return torch.from_numpy(np.ascontiguousarray(xb).view(np.int16)).cuda().view(torch.bfloat16)


def _bf16(t):
    return t.float().cpu().numpy().astype(np.float64)


def _decoder_layers(polyq_lib, hidden, ffn, n_layers, config):
    """Packed layers with the v->o and gate/up->down merges, library and
    oracle side."""
    names = [n for n, _, _ in O.llama_layer_linears(hidden, ffn)]
    dev_layers, ora_layers = [], []
    for layer in range(n_layers):
        hosts, refs = {}, {}
        for i, (name, N, K) in enumerate(O.llama_layer_linears(hidden, ffn)):
            W, a = synth.layer_weights(N, K, synth.seed_for(config, 10 * layer + i))
            hosts[name] = polyq_lib.HostLayer.pack(W, a, 3.0)
            refs[name] = O.pack_layer(W, a, 3.0)
        merged = O.merge_decoder_layer(refs)
        hosts["v"].permute_rows(hosts["o"].export()["perm"])
        for n in ("gate", "up"):
            hosts[n].permute_rows(hosts["down"].export()["perm"])
        dev_layers.append({n: polyq_lib.DeviceLayer(hosts[n], "cuda",
                                                    identity_gather=n in ("o", "down"))
                           for n in names})
        ora_layers.append(merged)
    return dev_layers, ora_layers


def _layer_phases(polyq_lib, dev, s, bufs):
    """The four phases of one decoder layer on the residual stream s."""
    q, k, v, g, u, h, xo, h2, xd = bufs
    return [
        dict(layers=[dev["q"], dev["k"], dev["v"]], kind=polyq_lib.X_RMSNORM, a=s, eps=1e-6,
             ys=[q, k, v], x_out=h),
        dict(layers=[dev["o"]], kind=polyq_lib.X_F32, a=v, ys=[s], residuals=[s], x_out=xo),
        dict(layers=[dev["gate"], dev["up"]], kind=polyq_lib.X_RMSNORM, a=s, eps=1e-6,
             ys=[g, u], x_out=h2),
        dict(layers=[dev["down"]], kind=polyq_lib.X_SILU_MUL, a=g, b=u, ys=[s], residuals=[s],
             x_out=xd),
    ]


def _bufs(hidden, ffn, batch=1):
    f = lambda n: torch.zeros((batch, n), dtype=torch.float32, device="cuda")
    b = lambda n: torch.zeros((batch, n), dtype=torch.bfloat16, device="cuda")
    return (f(hidden), f(hidden), f(hidden), f(ffn), f(ffn), b(hidden), b(hidden), b(hidden),
            b(ffn))


def test_chained_decoder_layers_match_oracle_and_per_call(polyq_lib):
    hidden, ffn, n_layers = 256, 640, 3
    dev_layers, ora_layers = _decoder_layers(polyq_lib, hidden, ffn, n_layers, 7)
    s0 = np.random.default_rng(7).standard_normal((1, hidden)).astype(np.float32)
    s = torch.from_numpy(s0).cuda()
    bufs = [_bufs(hidden, ffn) for _ in range(n_layers)]
    phases = []
    for dev, b in zip(dev_layers, bufs):
        phases += _layer_phases(polyq_lib, dev, s, b)
    chain = polyq_lib.GemvChain(phases, batch=1)
    chain.run()
    torch.cuda.synchronize()
    assert int(chain.workspace[:4].view(torch.int32).item()) == 0

    # every linear against the oracle fed the GPU's actual inputs
    s_ref = s0.astype(np.float64)
    for merged, b in zip(ora_layers, bufs):
        q, k, v, g, u, h, xo, h2, xd = b
        hx, xox, h2x, xdx = _bf16(h), _bf16(xo), _bf16(h2), _bf16(xd)
        for name, y, x in (("q", q, hx), ("k", k, hx), ("v", v, hx), ("gate", g, h2x),
                           ("up", u, h2x)):
            L, gat = merged[name]
            check_tolerance(y.cpu().numpy(), O.linear(L, x, gather=gat), x, x.shape[1])
        # the glue: x_out holds bf16 of the transform of the GPU's own values
        assert rel_l2(xox, O.bf16_rn(v.cpu().numpy().astype(np.float64))) == 0.0
        xd_ref = O.bf16_rn(O.silu(g.cpu().numpy().astype(np.float64))
                           * u.cpu().numpy().astype(np.float64))
        assert np.mean(xdx == xd_ref) > 0.99
        s_ref, _ = O.decode_layer(s_ref, merged)
    got = s.cpu().numpy().astype(np.float64)
    assert rel_l2(got, s_ref) <= 1e-2

    # the same layers through the per-call entry point
    s2 = torch.from_numpy(s0).cuda()
    for dev in dev_layers:
        q, k, v = polyq_lib.linear_gemv_input([dev["q"], dev["k"], dev["v"]],
                                              polyq_lib.X_RMSNORM, s2, eps=1e-6)
        polyq_lib.linear_gemv_input([dev["o"]], polyq_lib.X_F32, v, ys=[s2], residuals=[s2])
        g, u = polyq_lib.linear_gemv_input([dev["gate"], dev["up"]], polyq_lib.X_RMSNORM, s2,
                                           eps=1e-6)
        polyq_lib.linear_gemv_input([dev["down"]], polyq_lib.X_SILU_MUL, g, b=u, ys=[s2],
                                    residuals=[s2])
    torch.cuda.synchronize()
    assert rel_l2(got, s2.cpu().numpy()) <= 1e-3

    # a second launch on the same workspace starts from the barrier counters
    # the first one left (zero) and gives the same stream
    s.copy_(torch.from_numpy(s0).cuda())
    chain.run()
    torch.cuda.synchronize()
    assert int(chain.workspace[:4].view(torch.int32).item()) == 0
    assert rel_l2(s.cpu().numpy(), got) <= 1e-4


@pytest.mark.parametrize("batch", [1, 2, 3, 4])
def test_independent_phases_match_oracle(polyq_lib, batch):
    # q+k+v, o, gate+up, down on their own bf16 inputs, as one chain
    hidden, ffn = 512, 1280
    lin = O.llama_layer_linears(hidden, ffn)
    hosts, refs, xs = {}, {}, {}
    for i, (name, N, K) in enumerate(lin):
        W, a = synth.layer_weights(N, K, 3000 + i)
        bits = synth.random_codes_layer_bits(K, 3000 + i) if name in ("k", "down") else None
        hosts[name] = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
        refs[name] = O.pack_layer(W, a, 3.0, bits=bits)
        xs[name] = synth.activations(a, batch, 3100 + i)
    dev = {n: polyq_lib.DeviceLayer(hosts[n], "cuda") for n in hosts}
    xd = {n: _x_dev(xs[n][0]) for n in xs}
    ys = {n: torch.full((batch, N), float("nan"), device="cuda") for n, N, _ in lin}
    res = torch.randn(batch, hidden, device="cuda")
    groups = [("q", "k", "v"), ("o",), ("gate", "up"), ("down",)]
    phases = []
    for grp in groups:
        ph = dict(layers=[dev[n] for n in grp], kind=polyq_lib.X_BF16, a=xd[grp[0]],
                  xs=[xd[n] for n in grp], ys=[ys[n] for n in grp])
        if grp == ("o",):
            ph["residuals"] = [res]
        phases.append(ph)
    chain = polyq_lib.GemvChain(phases, batch=batch)
    for _ in range(2):
        for y in ys.values():
            y.fill_(float("nan"))
        chain.run()
        torch.cuda.synchronize()
        for name, N, K in lin:
            ref = O.linear(refs[name], xs[name][1])
            if name == "o":
                ref = ref + res.cpu().numpy().astype(np.float64)
            check_tolerance(ys[name].cpu().numpy(), ref, xs[name][1], K)


def test_phase_with_more_records_than_ctas(polyq_lib):
    # Four layers of 48 rows (one partial tile each) over K = 65536 channels
    # of all five widths at batch 4: 2048 records, so every CTA builds
    # several, and each CTA's items are consecutive steps of one tile.
    K, N, batch = 65536, 48, 4
    bits = synth.random_codes_layer_bits(K, 91)
    dev, refs = [], []
    for i in range(4):
        W, a = synth.layer_weights(N, K, 90 + i)
        dev.append(polyq_lib.DeviceLayer(
            polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits), "cuda"))
        refs.append(O.pack_layer(W, a, 3.0, bits=bits))
    xb, x = synth.activations(synth.layer_weights(1, K, 95)[1], batch, 95)
    ys = [torch.empty((batch, N), device="cuda") for _ in range(4)]
    chain = polyq_lib.GemvChain([dict(layers=dev, kind=polyq_lib.X_BF16, a=_x_dev(xb), ys=ys)],
                                batch=batch)
    chain.run()
    torch.cuda.synchronize()
    for y, ref in zip(ys, refs):
        check_tolerance(y.cpu().numpy(), O.linear(ref, x), x, K)


def test_record_wait_gives_up_with_a_status(polyq_lib):
    # Failure detection without a fault: the launch count in the workspace is
    # raised so that the producers' target for the records of phase 0 is one
    # nothing will reach.  Their bounded wait gives up after about a second,
    # the launch returns with status 4, and after zeroing the workspace the
    # same chain runs correctly again.
    K, N = 512, 256
    W, a = synth.layer_weights(N, K, 97)
    dev = polyq_lib.DeviceLayer(polyq_lib.HostLayer.pack(W, a, 3.0), "cuda")
    ref = O.pack_layer(W, a, 3.0)
    xb, x = synth.activations(a, 1, 97)
    y = torch.zeros((1, N), device="cuda")
    chain = polyq_lib.GemvChain([dict(layers=[dev], kind=polyq_lib.X_BF16, a=_x_dev(xb),
                                      ys=[y])], batch=1)
    assert polyq_lib.workspace_status(chain.workspace) == 0
    chain.workspace[72:76].view(torch.int32).fill_(1 << 20)  # launches completed
    chain.run()
    with pytest.raises(polyq_lib.PolyqError) as ei:
        polyq_lib.workspace_status(chain.workspace)
    assert ei.value.code == polyq_lib.POLYQ_ETIMEOUT
    assert int(chain.workspace[:4].view(torch.int32).item()) == 4
    # the context still works: clear the workspace and run again
    chain.workspace.zero_()
    chain.run()
    torch.cuda.synchronize()
    assert polyq_lib.workspace_status(chain.workspace) == 0
    check_tolerance(y.cpu().numpy(), O.linear(ref, x), x, K)


@pytest.mark.parametrize("batch", [1, 4])
@pytest.mark.parametrize("scale_exp", [-40, 12, 40])
def test_chained_phases_at_any_activation_scale(polyq_lib, batch, scale_exp):
    """The chained launch builds its records with the same per-chunk exponent
    as the per-call pre-pass: two dependent-free phases of all five widths,
    with inputs scaled by 2^scale_exp, against the oracle."""
    phases, refs, xs = [], [], []
    for i, (N, K) in enumerate(((200, 3001), (96, 1100))):
        W, a = synth.layer_weights(N, K, 90 + i)
        bits = synth.random_codes_layer_bits(K, 90 + i)
        host = polyq_lib.HostLayer.pack(W, a, 3.0, forced_bits=bits)
        dev = polyq_lib.DeviceLayer(host, "cuda")
        refs.append(O.pack_layer(W, a, 3.0, bits=bits))
        _, x = synth.activations(a, batch, 90 + i)
        x = x * 2.0 ** scale_exp
        xb = synth.bf16_bits(x.astype(np.float32))
        assert np.array_equal(synth.bf16_to_f64(xb), x)
        xs.append(x)
        y = torch.zeros((batch, N), dtype=torch.float32, device="cuda")
        phases.append(dict(layers=[dev], kind=polyq_lib.X_BF16, a=_x_dev(xb), ys=[y]))
    chain = polyq_lib.GemvChain(phases, batch=batch)
    chain.run()
    torch.cuda.synchronize()
    assert polyq_lib.workspace_status(chain.workspace) == 0
    for ph, ref, x in zip(phases, refs, xs):
        check_tolerance(ph["ys"][0].cpu().numpy(), O.linear(ref, x), x, x.shape[1])
