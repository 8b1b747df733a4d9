"""Decoding attention on the packed cache: CUDA path (C ABI) vs the oracle.

Eq. (app_decode_logit) with appends at multiplicity 1.  Inputs are seeded
draws (synth.make_decode_cache) or the oracle's own compressed cache; no
oracle input comes from the CUDA path.

Tolerance (fp32 arithmetic on exact bf16 / fp32 inputs): a logit error dx
moves a softmax-weighted mean of values by at most 2 |dx| max|v|, and the
weighted sums accumulate at most n_seq rounding errors of relative size
2^-24 each, n_seq being the longest sum one thread forms (at most the head's
length / 8, plus the merge of pieces).  The logit error is bounded by the
fp32 dot product, d 2^-24 sum_i |q_i k_i| / sqrt(d), plus the base-2
exponential's own error (2^-21 relative, i.e. 2^-21 in the exponent scale).
So per output row:  |err| <= max|v| (2 dx_max + 2^-24 (n / 8 + 64)) + 1e-7.
"""
import math

import numpy as np
import pytest
import torch

from paper_2608_07001_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def _oracle(c, l0=0, nl=None, n_app=None):
    import oracle as O
    L, G = c["L"], c["G"]
    nl = L - l0 if nl is None else nl
    off = c["offsets"].cpu().numpy()
    lo, hi = int(off[l0 * G]), int(off[(l0 + nl) * G])
    sub_off = off[l0 * G:(l0 + nl) * G + 1] - lo
    n_app = c["n_app"] if n_app is None else n_app
    Ka = c["K_app"][l0:l0 + nl] if c["K_app"] is not None else None
    Va = c["V_app"][l0:l0 + nl] if c["V_app"] is not None else None
    return O.decode_attention(c["q"][l0:l0 + nl], c["K"][lo:hi], c["V"][lo:hi], c["log_m"][lo:hi],
                              sub_off, Ka, Va, n_app, L=nl, G=G, l0=0)


def _tolerance(c, l0, nl, n_app):
    """Per (l, h) bound of the module docstring, from the inputs."""
    G, d = c["G"], c["q"].shape[-1]
    Hq = c["q"].shape[1]
    gq = Hq // G
    off = c["offsets"].cpu().numpy()
    q = c["q"].double().cpu()
    tol = np.zeros((nl, Hq))
    for i in range(nl):
        for g in range(G):
            lg = (l0 + i) * G + g
            ks = [c["K"][off[lg]:off[lg + 1]].double().cpu()]
            vs = [c["V"][off[lg]:off[lg + 1]].double().cpu()]
            if n_app:
                ks.append(c["K_app"][l0 + i, g, :n_app].double().cpu())
                vs.append(c["V_app"][l0 + i, g, :n_app].double().cpu())
            kk, vv = torch.cat(ks), torch.cat(vs)
            n = kk.shape[0]
            if n == 0:
                continue
            vmax = float(vv.abs().max())
            for hh in range(gq):
                h = g * gq + hh
                dot_abs = float((kk.abs() @ q[l0 + i, h].abs()).max())
                dx = d * 2.0 ** -24 * dot_abs / math.sqrt(d) + 2.0 ** -21 * (1 + dot_abs / math.sqrt(d))
                tol[i, h] = vmax * (2 * dx + 2.0 ** -24 * (n / 8 + 64)) + 1e-7
    return tol


def _check(c, out, l0=0, nl=None, n_app=None):
    nl = c["L"] - l0 if nl is None else nl
    n_app = c["n_app"] if n_app is None else n_app
    ref = _oracle(c, l0, nl, n_app)
    tol = _tolerance(c, l0, nl, n_app)
    got = out.double().cpu().numpy()
    err = np.abs(got - ref).max(axis=-1)
    bad = np.argwhere(err > tol)
    assert bad.size == 0, (f"{len(bad)} rows over tolerance; worst err {err.max():.3e}, "
                           f"tol there {tol.flat[err.argmax()]:.3e}")
    return float(err.max()), float(tol.min())


def _as_dict(dc: synth.DecodeCache, L, G):
    return dict(q=dc.q, K=dc.K, V=dc.V, log_m=dc.log_m, offsets=dc.offsets, K_app=dc.K_app,
                V_app=dc.V_app, n_app=dc.n_app, L=L, G=G)


def _decoder(c, Hq, app_cap):
    from paper_2608_07001_gb300.gracekv import Decoder
    dev = torch.device("cuda")
    dc = Decoder(c["K"].to(dev), c["V"].to(dev), c["log_m"].to(dev), c["offsets"].to(dev),
                 L=c["L"], G=c["G"], Hq=Hq, app_cap=app_cap)
    return dc


def _run(c, Hq, l0=0, nl=None, app_cap=None):
    app_cap = max(c["n_app"], 1) if app_cap is None else app_cap
    dc = _decoder(c, Hq, app_cap)
    if c["n_app"]:
        dc.K_app[:, :, :c["n_app"]] = c["K_app"][:, :, :c["n_app"]].cuda()
        dc.V_app[:, :, :c["n_app"]] = c["V_app"][:, :, :c["n_app"]].cuda()
        dc.n_app = c["n_app"]
    nl = c["L"] - l0 if nl is None else nl
    out = dc.attention(c["q"][l0:l0 + nl].cuda().contiguous(), l0=l0)
    torch.cuda.synchronize()
    dc.status()
    return out, dc


@pytest.mark.parametrize("wname,ratio,n_app", [("small", 32, 0), ("small", 8, 5), ("llama32k", 32, 17)])
def test_decode_matches_oracle(wname, ratio, n_app):
    # small: d 64, 4 query heads per KV head; llama32k: d 128, gq 4, bf16;
    # the llama32k case uses 4 of its 32 layers (the oracle's budget)
    w = synth.WORKLOADS[wname]
    if wname == "llama32k":
        w = synth.Workload(**{**w.__dict__, "L": 4})
    dc = synth.make_decode_cache(w, ratio, n_app=n_app, app_cap=n_app + 3)
    c = _as_dict(dc, w.L, w.G)
    out, _ = _run(c, w.Hq, app_cap=n_app + 3)
    err, _ = _check(c, out)
    print(wname, ratio, n_app, "max err", err)


@pytest.mark.parametrize("gq,d,dtype", [(1, 128, "f32"), (2, 64, "bf16"), (8, 128, "bf16"),
                                        (8, 64, "f32"), (4, 64, "f32"), (1, 64, "bf16")])
def test_decode_head_group_sizes(gq, d, dtype):
    w = synth.Workload("g", 3, 2, 2 * gq, d, 4096, 8, dtype, "lognormal", 0, 1.0, 1e4, (8,), 11 + gq)
    dc = synth.make_decode_cache(w, 4, n_app=3, app_cap=4)
    c = _as_dict(dc, w.L, w.G)
    out, _ = _run(c, w.Hq, app_cap=4)
    _check(c, out)


def test_decode_ragged_edge_cases():
    # empty heads (no packed entry, no append: zero output), single entries,
    # heads much longer than a CTA's chunk, a total smaller than the grid
    w = synth.Workload("e", 2, 4, 8, 128, 1024, 8, "bf16", "lognormal", 0, 1.0, 1e4, (8,), 21)
    for counts in ([0, 1, 5000, 0, 3, 0, 20000, 1], [1, 0, 0, 0, 0, 0, 0, 2], [0] * 8,
                   [33, 7, 1, 2, 900, 0, 0, 5]):
        dc = synth.make_decode_cache(w, 1, counts=np.asarray(counts))
        c = _as_dict(dc, w.L, w.G)
        out, _ = _run(c, w.Hq)
        _check(c, out)
        for lg, n in enumerate(counts):
            if n == 0:
                l, g = divmod(lg, 4)
                assert torch.all(out[l, 2 * g:2 * g + 2] == 0)


def test_decode_layer_slices_and_repeats_are_identical():
    # calls on a layer range [l0, l0 + n) meet the oracle on that slice, and
    # repeated calls on one workspace agree bit for bit (the per-head counters
    # are left at zero)
    w = synth.WORKLOADS["small"]
    dc = synth.make_decode_cache(w, 16, n_app=2, app_cap=2)
    c = _as_dict(dc, w.L, w.G)
    out, dec = _run(c, w.Hq, app_cap=2)
    q = c["q"].cuda()
    for _ in range(3):
        again = dec.attention(q)
        torch.cuda.synchronize()
        assert torch.equal(again, out)
    for l0, nl in ((0, 1), (5, 3), (15, 1)):
        part = dec.attention(q[l0:l0 + nl].contiguous(), l0=l0)
        torch.cuda.synchronize()
        _check(c, part, l0, nl)
    assert not torch.any(dec.workspace[256:256 + 4 * w.L * w.G])


def test_decode_more_heads_than_one_launch_holds():
    # 160 layers x 8 KV heads = 1280 heads: the call runs as consecutive
    # launches over layer groups
    w = synth.Workload("m", 160, 8, 16, 64, 320, 8, "bf16", "lognormal", 0, 1.0, 1e4, (8,), 41)
    dc = synth.make_decode_cache(w, 8, n_app=1, app_cap=1)
    c = _as_dict(dc, w.L, w.G)
    out, dec = _run(c, w.Hq, app_cap=1)
    _check(c, out)
    part = dec.attention(c["q"][100:].cuda().contiguous(), l0=100)
    torch.cuda.synchronize()
    _check(c, part, 100, 60)


def test_decode_append_through_the_api():
    # tokens appended with gracekv_decode_append join with log m = 0
    w = synth.Workload("a", 4, 2, 8, 128, 2048, 8, "bf16", "lognormal", 0, 1.0, 1e4, (8,), 31)
    dc = synth.make_decode_cache(w, 8, n_app=6, app_cap=8)
    c = _as_dict(dc, w.L, w.G)
    dec = _decoder(c, w.Hq, 8)
    for t in range(6):
        # first the lower two layers, then the upper two (per-layer appends)
        dec.append(c["K_app"][:2, :, t].cuda().contiguous(), c["V_app"][:2, :, t].cuda().contiguous(), l0=0)
        dec.append(c["K_app"][2:, :, t].cuda().contiguous(), c["V_app"][2:, :, t].cuda().contiguous(), l0=2)
    assert dec.n_app == 6
    out = dec.attention(c["q"].cuda())
    torch.cuda.synchronize()
    _check(c, out)
    from paper_2608_07001_gb300.gracekv import GraceKVError
    dec.n_app = 8
    with pytest.raises(GraceKVError):
        dec.append(c["K_app"][:, :, 0].cuda().contiguous(), c["V_app"][:, :, 0].cuda().contiguous())


def test_decode_on_the_oracle_compressed_cache():
    # the packed cache the oracle's own compression writes (prototypes with
    # their log m_eff, singletons, recent window), fp32, 2 KV heads
    import oracle as O
    w = synth.WORKLOADS["pr1"]
    x = synth.make_inputs(w)
    res = O.run(x.K, x.V, x.Q, 256, w.rope_base)
    cache = res["cache"]
    g = torch.Generator().manual_seed(5)
    q = torch.randn(1, 2, 128, generator=g, dtype=torch.float64) * 2
    c = dict(q=q.float(), K=torch.as_tensor(cache["K"]).float(), V=torch.as_tensor(cache["V"]).float(),
             log_m=torch.as_tensor(cache["log_m"]).float(), offsets=torch.as_tensor(cache["offsets"]),
             K_app=None, V_app=None, n_app=0, L=1, G=2)
    assert float(c["log_m"].max()) > 1.0
    out, _ = _run(c, 2)
    _check(c, out)


def test_decode_full_size_sampled_layers():
    # Llama-3-8B shape at 128K context, 32x: 1M packed entries over 32 x 8
    # heads in one launch; the oracle checks 3 sampled layers
    w = synth.WORKLOADS["llama128k"]
    dc = synth.make_decode_cache(w, 32, n_app=9, app_cap=16, device="cuda")
    c = _as_dict(dc, w.L, w.G)
    out, _ = _run(c, w.Hq, app_cap=16)
    cpu = {k: (v.cpu() if torch.is_tensor(v) else v) for k, v in c.items()}
    for l0 in (0, 17, 31):
        _check(cpu, out[l0:l0 + 1], l0, 1)
