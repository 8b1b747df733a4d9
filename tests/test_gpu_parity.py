"""CUDA path vs CPU oracle on seeded inputs (through the C ABI)."""
import json
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


def _run(inp_K, inp_V, inp_Q, B, base, **kw):
    from tests import parity as P
    g = P.run_gpu(inp_K, inp_V, inp_Q, B, base, **kw)
    o = P.run_oracle(inp_K, inp_V, inp_Q, B, base, **kw)
    return P, g, o


def test_pr1_parity():
    # PR1: 1 layer x 2 KV heads x d 128, T = 1024, fp32, 8x (B_total = 256)
    w = synth.WORKLOADS["pr1"]
    x = synth.make_inputs(w)
    B = (1 * 2 * 1024) // 8
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base)
    rep = P.compare(g, o, torch.float32)
    print("pr1", json.dumps(rep))
    assert g["E"] == 256 and g["recent"] == 32


def test_ragged_bf16_gqa_parity():
    # small-model shapes (d 64, 4 query heads per KV head, 64 probes, bf16) on a
    # 2-layer slice with a ragged T = 1000; several slots, tiles and tails.
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[0, 1], heads=[0, 1], T=1000)
    L, G, T, d = x.K.shape
    B = (L * G * T) // 8
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base)
    rep = P.compare(g, o, torch.bfloat16)
    print("ragged_bf16", json.dumps(rep))


@pytest.mark.parametrize("x_ratio", [2, 16])
def test_budget_sweep_bf16(x_ratio):
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[3], heads=[2, 5], T=1536, W=32)
    L, G, T, d = x.K.shape
    B = (L * G * T) // x_ratio
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base)
    rep = P.compare(g, o, torch.bfloat16)
    print(f"x={x_ratio}", json.dumps(rep))


@pytest.mark.parametrize("ablation", ["wo_cs", "wo_ga", "both"])
def test_ablations_match_the_oracle(ablation):
    # the paper's "w/o CS" (uniform slots of target 64, midpoint-only cuts, no
    # curvature reward) and "w/o GA" (fixed per-(l, g) capacity; trees built
    # completely) variants, on a 2-layer x 2-head bf16 slice and on PR1 fp32
    kw = {}
    if ablation in ("wo_cs", "both"):
        kw.update(seg_mode=1, k_cand=0, lambda_kappa=0.0)
    if ablation in ("wo_ga", "both"):
        kw.update(quota_alloc=1)
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[0, 1], heads=[0, 1], T=1000)
    L, G, T, d = x.K.shape
    B = (L * G * T) // 8
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base, **kw)
    rep = P.compare(g, o, torch.bfloat16)
    print(ablation, json.dumps(rep))
    if "seg_mode" in kw:
        np.testing.assert_array_equal(g["slots"], o["seg"]["slot_starts"])
    if "quota_alloc" in kw:
        # every (l, g) stays within its capacity
        LG, J = L * G, g["J"]
        Bf = o["B_free"]
        ex = g["export"]
        first = ex["unit_first"]
        for lg in range(LG):
            q = Bf // LG + (1 if lg < Bf % LG else 0)
            u0, u1 = lg * J, (lg + 1) * J
            used = int((ex["add_sel"][u0:u1] == 1).sum())
            sl = slice(int(first[u0]), int(first[u1]))
            used += int(((ex["split_sel"][sl] == 1) * ex["cost"][sl]).sum())
            assert used <= q, (lg, used, q)
    wp = synth.WORKLOADS["pr1"]
    xp = synth.make_inputs(wp)
    P, g, o = _run(xp.K, xp.V, xp.Q, 256, wp.rope_base, **kw)
    P.compare(g, o, torch.float32)


@pytest.mark.parametrize("wname,alpha", [("small", 0.6), ("pr1", 0.6), ("small", 0.05), ("pr1", 0.1)])
def test_singleton_floor_matches_the_oracle(wname, alpha):
    # Stage I singleton floor at the paper's alpha = 0.6: the accepted floor
    # positions, then the trees (forced extraction), the selection (floor ops
    # first) and the cache against the oracle
    if wname == "small":
        w = synth.WORKLOADS["small"]
        x = synth.make_inputs(w, layers=[0, 1], heads=[0, 1], T=1000)
        dt = torch.bfloat16
    else:
        w = synth.WORKLOADS["pr1"]
        x = synth.make_inputs(w)
        dt = torch.float32
    L, G, T, d = x.K.shape
    B = (L * G * T) // 8
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base, alpha_floor=alpha)
    fl = g["comp"].ctx.gracekv_export_floor()
    ofl = o["floor"]
    assert ofl["accepted"].sum() > 0
    diff = np.argwhere(fl["accepted"] != ofl["accepted"])
    print(wname, "floor", int(ofl["accepted"].sum()), "B_floor", ofl["B_floor"], fl["B_floor"],
          "differing positions", len(diff))
    assert len(diff) == 0, diff[:10]
    assert fl["B_floor"] == ofl["B_floor"]
    np.testing.assert_allclose(fl["f"], ofl["f"], rtol=2e-5, atol=1e-9)
    rep = P.compare(g, o, dt)
    print(wname, json.dumps(rep))


def _floor_skip_case(seed=11):
    # Token values by construction: keys lie along e_0 with logit c_t (plus
    # small noise), every query is sqrt(d) e_0, no RoPE; so R_t is about
    # exp(c_t) / sum exp(c) over the context.  Head 0's candidates in f order:
    # 100 (uncovered slot [64, 128): 3 entries), 300 (uncovered slot [256,
    # 320): 3), 101 (next to 100: 1).  Head 1's: 0, 1, 2 at the start of slot
    # [0, 64): 2 + 1 + 1.  Joint cost 7 + 4 = 11 = cap = floor(0.115 B_free),
    # B_free = 100, so no reduction; shares floor(11 * 3 / 6) = 5 each.
    L, G, Hq, T, d, W = 1, 2, 2, 544, 64, 4
    rng = np.random.default_rng(seed)
    K = 0.05 * rng.normal(size=(L, G, T, d))
    V = rng.normal(size=(L, G, T, d))
    c = np.zeros((G, T))
    c[0, [100, 300, 101]] = np.log([400.0, 300.0, 200.0])
    c[1, [0, 1, 2]] = np.log([400.0, 300.0, 200.0])
    K[0, :, :, 0] += c
    Q = np.zeros((L, Hq, W, d))
    Q[..., 0] = np.sqrt(d)
    f32 = lambda a: torch.as_tensor(a, dtype=torch.float32)
    return f32(K), f32(V), f32(Q), np.arange(0, 513, 64)


def test_floor_skips_an_unaffordable_candidate_on_the_device():
    # App. A.5 Stage I: a candidate is accepted only when its complete path
    # still fits; head 0 skips 300 (3 + 3 > 5) and then accepts 101 (3 + 1)
    K, V, Q, slots = _floor_skip_case()
    kw = dict(slot_starts=slots, alpha_floor=0.115, floor_c=0.0, floor_half=0)
    P, g, o = _run(K, V, Q, 164, 0.0, **kw)
    ofl = o["floor"]
    assert o["B_free"] == 100
    assert set(np.nonzero(ofl["accepted"][0])[0]) == {100, 101}
    assert set(np.nonzero(ofl["accepted"][1])[0]) == {0, 1, 2}
    assert ofl["B_floor"] == 8
    fl = g["comp"].ctx.gracekv_export_floor()
    np.testing.assert_array_equal(fl["accepted"], ofl["accepted"])
    assert fl["B_floor"] == ofl["B_floor"]
    rep = P.compare(g, o, torch.float32)
    print("floor skip", json.dumps(rep))


@pytest.mark.parametrize("L,G,gq,d,D,U", [(3, 2, 4, 128, 1024, 32), (2, 8, 4, 128, 4096, 64),
                                          (4, 4, 1, 64, 520, 5)])
def test_head_sensitivity_matches_the_oracle(L, G, gq, d, D, U):
    # omega of App. A.4 (Eq. app_head_sensitivity) on the tensor cores vs the
    # oracle; the per-(l, g) output of the one call feeds the pass's omega
    import oracle as O
    from paper_2608_07001_gb300 import gracekv as gk
    g = torch.Generator().manual_seed(L * 100 + D)
    Hq = G * gq
    W = (torch.randn(L, D, Hq * d, generator=g) / d ** 0.5)
    W[:, :, :gq * d] *= 3.0                       # one group stands out
    W = W.to(torch.bfloat16)
    o = torch.randn(L, Hq, U, d, generator=g).to(torch.bfloat16)
    om = gk.gracekv_head_sensitivity(W.cuda(), o.cuda(), G).cpu().double().numpy()
    ref = O.head_sensitivity(W, o, G)
    # fp32 sums of exact products: a few ulp of the sums per term, well below 1e-4
    np.testing.assert_allclose(om, ref, rtol=1e-4, atol=1e-6)


@pytest.mark.parametrize("m_seed", [64, 8])
def test_multihop_relevance_matches_the_oracle(m_seed):
    # App. A.4: seeds from the global seed score, two hops of causal seed
    # attention at the graph layers, R = 0.7 s-hat + 0.3 d-hat; then the trees,
    # selection and cache of the pass against the oracle
    import oracle as O
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[0, 1, 2, 3], heads=[0, 1], T=1000)
    L, G, T, d = x.K.shape
    p = O.make_params(L, G, x.Q.shape[1], T, d, x.Q.shape[2], w.rope_base, recent=32)
    gl = O.graph_layers(p)
    Qg = synth.make_graph_queries(w, [int(l) for l in gl], T=T, heads=range(x.Q.shape[1]))
    B = (L * G * T) // 8
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base, Qg=Qg, lambda_graph=0.3, m_seed=m_seed)
    ex = g["export"]
    mh = o["multihop"]
    rt = np.asarray(ex["rtok"]).reshape(o["rtok"].shape)
    err = np.abs(rt - o["rtok"]).max() / np.abs(o["rtok"]).max()
    print("multihop seeds", [int(v) for v in mh["seeds"][0][:8]], "rtok rel err", err)
    assert err < 1e-4
    rep = P.compare(g, o, torch.bfloat16)
    print("multihop", json.dumps(rep))


@pytest.mark.parametrize("T,cs", [(6000, 0), (4500, 7)])
def test_multihop_over_several_selection_parts(T, cs):
    # N_c > 2048: the seed selection merges several sorted 2048-token parts,
    # the last one ragged; a sink prefix (cs > 0) lies inside every seed's
    # causal range but outside C.  The mixed token values against the
    # oracle's token values and multi-hop relevance (App. A.4)
    import oracle as O
    from tests import parity as P
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[0, 1, 2, 3], heads=[0, 1], T=T)
    L, G, T, d = x.K.shape
    Hq, W = x.Q.shape[1], x.Q.shape[2]
    p = O.make_params(L, G, Hq, T, d, W, w.rope_base, cs, lambda_graph=0.3)
    B = (L * G * (T - cs)) // 8
    r_eff, _ = O.budget(p, B)
    p.recent = r_eff
    Nc = T - cs - r_eff
    assert Nc > 2 * 2048 and Nc % 2048 != 0
    gl = O.graph_layers(p)
    Qg = synth.make_graph_queries(w, [int(l) for l in gl], T=T, heads=range(Hq))
    g = P.run_gpu(x.K, x.V, x.Q, B, w.rope_base, ctx_start=cs, Qg=Qg, lambda_graph=0.3)
    rt = np.asarray(g["export"]["rtok"]).reshape(L, G, Nc)
    K64, Q64 = x.K.double().numpy(), x.Q.double().numpy()
    m, Z, _ = O.row_stats(p, Q64, K64)
    shat = O.token_values(p, Q64, K64, m, Z)
    dh, sd, _ = O.multihop(p, shat, Qg, K64)
    ref = 0.7 * shat + 0.3 * dh[None, None, :]
    err = np.abs(rt - ref).max() / np.abs(ref).max()
    print("multihop parts", -(-Nc // 2048), "seeds", int((sd[0] >= 0).sum()), int((sd[1] >= 0).sum()),
          "rel err", err)
    assert err < 1e-4


def test_floor_reads_the_multihop_mixed_values():
    # both NEXT stages at the paper's values (alpha 0.6, lambda 0.3): the floor
    # (App. A.5 Stage I) takes R after the multi-hop mix (Eq.
    # app_bottom_up_value); accepted positions, trees, selection and cache
    import oracle as O
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[0, 1, 2, 3], heads=[0, 1], T=1000)
    L, G, T, d = x.K.shape
    p = O.make_params(L, G, x.Q.shape[1], T, d, x.Q.shape[2], w.rope_base, recent=32)
    gl = O.graph_layers(p)
    Qg = synth.make_graph_queries(w, [int(l) for l in gl], T=T, heads=range(x.Q.shape[1]))
    B = (L * G * T) // 8
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base, Qg=Qg, lambda_graph=0.3, alpha_floor=0.6)
    fl = g["comp"].ctx.gracekv_export_floor()
    ofl = o["floor"]
    assert ofl["accepted"].sum() > 0
    assert np.array_equal(fl["accepted"], ofl["accepted"])
    assert fl["B_floor"] == ofl["B_floor"]
    np.testing.assert_allclose(fl["f"], ofl["f"], rtol=2e-5, atol=1e-9)
    rep = P.compare(g, o, torch.bfloat16)
    print("floor+multihop", int(ofl["accepted"].sum()), json.dumps(rep))


def test_fullkv_identity_is_bit_exact():
    # x = 1: every tree expands to its leaves; the cache is the input (App. C.6)
    w = synth.WORKLOADS["pr1"]
    x = synth.make_inputs(w, T=640)
    L, G, T, d = x.K.shape
    from tests import parity as P
    g = P.run_gpu(x.K, x.V, x.Q, L * G * T, w.rope_base)
    c = g["cache"]
    assert g["E"] == L * G * T
    for lg in range(L * G):
        lo, hi = c["offsets"][lg], c["offsets"][lg + 1]
        assert np.array_equal(c["pos"][lo:hi].numpy(), np.arange(T))
        assert torch.equal(c["K"][lo:hi], x.K[lg // G, lg % G])
        assert torch.equal(c["V"][lo:hi], x.V[lg // G, lg % G])
        assert torch.all(c["log_m"][lo:hi] == 0)


def test_context_prefix_suffix_parity():
    w = synth.WORKLOADS["pr1"]
    x = synth.make_inputs(w, T=700)
    L, G, T, d = x.K.shape
    cs, ce = 37, 650
    B = (L * G * (ce - cs)) // 6
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base, ctx_start=cs, ctx_end=ce)
    rep = P.compare(g, o, torch.float32)
    print("ctx", json.dumps(rep))
    c = g["cache"]
    for lg in range(L * G):
        lo, hi = c["offsets"][lg], c["offsets"][lg + 1]
        assert np.array_equal(c["pos"][lo:lo + cs].numpy(), np.arange(cs))
        assert np.array_equal(c["pos"][hi - (T - ce + g["recent"]):hi].numpy(),
                              np.arange(ce - g["recent"], T))


def test_supplied_slots_hidden_surprisal_omega():
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[0], heads=[0, 1, 2], T=900, W=16)
    L, G, T, d = x.K.shape
    rng = np.random.default_rng(5)
    N = T - 32
    lens = []
    while sum(lens) < N:                      # includes single-token slots
        lens.append(int(rng.integers(1, 129)))
    lens[-1] -= sum(lens) - N
    lens = [n for n in lens if n > 0]
    starts = np.concatenate([[0], np.cumsum(lens)])
    hidden = rng.normal(size=(1, T, 48)).astype(np.float32)
    surprisal = np.abs(rng.normal(size=T)).astype(np.float32)
    surprisal[0] = 0
    omega = rng.uniform(0.5, 1.5, size=L * G).astype(np.float32)
    B = (L * G * T) // 5
    P, g, o = _run(x.K, x.V, x.Q, B, w.rope_base, slot_starts=starts, hidden=hidden,
                   surprisal=surprisal, omega=omega)
    rep = P.compare(g, o, torch.bfloat16)
    print("supplied", json.dumps(rep))


def test_errors_are_reported_not_trapped():
    from paper_2608_07001_gb300 import gracekv as gk
    w = synth.WORKLOADS["pr1"]
    x = synth.make_inputs(w, T=300)
    L, G, T, d = x.K.shape
    p = gk.make_params(L, G, 2, T, d, 32, dtype=torch.float32, budget=100, rope_base=w.rope_base)
    ctx = gk.Context(p)
    K, V, Q = x.K.cuda(), x.V.cuda(), x.Q.cuda()
    with pytest.raises(gk.GraceKVError) as e:          # out of order
        ctx.gracekv_allocate()
    assert e.value.status == gk.GKV_ESTATE
    slots = torch.empty(T, dtype=torch.int32, device="cuda")
    # a view starting one element past a 16-byte boundary is rejected on the host
    buf = torch.empty(V.numel() + 8, dtype=V.dtype, device="cuda")
    Vm = buf[1:1 + V.numel()].view(V.shape)
    Vm.copy_(V)
    with pytest.raises(gk.GraceKVError) as e:
        ctx.gracekv_segment(Vm, slots)
    assert e.value.status == gk.GKV_EINVAL
    ctx.gracekv_segment(V, slots)
    long = torch.tensor([0, 200, T - 32], dtype=torch.int32, device="cuda")   # a slot of 200 tokens builds
    ctx.gracekv_build_trees(K, V, Q, None, long, 2)
    assert ctx.gracekv_allocate() > 0
    ctx = gk.Context(p)
    ctx.gracekv_segment(V, slots)
    bad = torch.tensor([0, 50, 40, T - 32], dtype=torch.int32, device="cuda")
    with pytest.raises(gk.GraceKVError) as e:
        ctx.gracekv_build_trees(K, V, Q, None, bad, 3)
    assert e.value.status == gk.GKV_EINVAL
    # a supplied slot longer than 16384 tokens is refused before any tree work
    xl = synth.make_inputs(w, T=16500)
    pl = gk.make_params(L, G, 2, 16500, d, 32, dtype=torch.float32, budget=2000, rope_base=w.rope_base)
    ctxl = gk.Context(pl)
    Kl, Vl, Ql = xl.K.cuda(), xl.V.cuda(), xl.Q.cuda()
    ctxl.gracekv_segment(Vl, torch.empty(16500, dtype=torch.int32, device="cuda"))
    over = torch.tensor([0, 16400, 16500 - 32], dtype=torch.int32, device="cuda")
    with pytest.raises(gk.GraceKVError) as e:
        ctxl.gracekv_build_trees(Kl, Vl, Ql, None, over, 2)
    assert e.value.status == gk.GKV_EUNSUPPORTED
    del ctxl, Kl, Vl, Ql
    Vn = V.clone()
    Vn[0, 0, 17, 3] = float("nan")
    ctx2 = gk.Context(p)
    with pytest.raises(gk.GraceKVError) as e:
        ctx2.gracekv_segment(Vn, slots)
    assert e.value.status == gk.GKV_ENONFINITE
    Kn = K.clone()
    Kn[0, 1, 5, 0] = float("inf")
    ctx3 = gk.Context(p)
    ctx3.gracekv_segment(V, slots)
    ctx3.gracekv_build_trees(Kn, V, Q)
    with pytest.raises(gk.GraceKVError) as e:
        ctx3.gracekv_allocate()
    assert e.value.status == gk.GKV_ENONFINITE


def test_multihop_errors_are_reported():
    # the graph queries' contract (App. A.4 inputs): statuses, not faults
    from paper_2608_07001_gb300 import gracekv as gk
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[0, 1, 2, 3], heads=[0, 1], T=300)
    L, G, T, d = x.K.shape
    Hq, W = x.Q.shape[1], x.Q.shape[2]
    K, V, Q = x.K.cuda(), x.V.cuda(), x.Q.cuda()
    gl = gk.graph_layers(L)
    Qg = synth.make_graph_queries(w, gl, T=T, heads=range(Hq), device="cuda")
    mk = lambda lam: gk.make_params(L, G, Hq, T, d, W, dtype=torch.bfloat16, budget=L * G * T // 8,
                                    rope_base=w.rope_base, lambda_graph=lam)
    ctx0 = gk.Context(mk(0.0))
    with pytest.raises(gk.GraceKVError) as e:           # no multi-hop stage to feed
        ctx0.gracekv_set_graph_queries(Qg)
    assert e.value.status == gk.GKV_ESTATE
    ctx = gk.Context(mk(0.3))
    slots = torch.empty(T, dtype=torch.int32, device="cuda")
    ctx.gracekv_segment(V, slots)
    with pytest.raises(gk.GraceKVError) as e:           # build without the queries
        ctx.gracekv_build_trees(K, V, Q)
    assert e.value.status == gk.GKV_EINVAL
    buf = torch.empty(Qg.numel() + 8, dtype=Qg.dtype, device="cuda")
    with pytest.raises(gk.GraceKVError) as e:           # one element past a 16-byte boundary
        ctx.gracekv_set_graph_queries(buf[1:1 + Qg.numel()].view(Qg.shape))
    assert e.value.status == gk.GKV_EINVAL
    with pytest.raises(gk.GraceKVError) as e:           # one graph layer instead of two
        ctx.gracekv_set_graph_queries(Qg[:1])
    assert e.value.status == gk.GKV_EINVAL
    hc = gk.Cache.empty_host(L * G * T, d, L * G, K.dtype)
    with pytest.raises(gk.GraceKVError) as e:           # the host-buffer pass takes no queries
        ctx.gracekv_compress_host(x.K.contiguous(), x.V.contiguous(), x.Q.contiguous(), hc)
    assert e.value.status == gk.GKV_EUNSUPPORTED
    # the context still works: the same build with the queries set
    ctx.gracekv_set_graph_queries(Qg)
    ctx.gracekv_build_trees(K, V, Q)
    assert ctx.gracekv_allocate() > 0


def test_score_ahead_matches_inline():
    # The score passes issued ahead on a second stream (gracekv_score, as the
    # Compressor does) give the same bits as the passes the tree build runs
    # itself, and so the same trees and selection.
    from paper_2608_07001_gb300 import gracekv as gk
    w = synth.WORKLOADS["small"]
    x = synth.make_inputs(w, layers=[0, 1], heads=[0, 1], T=1000)
    L, G, T, d = x.K.shape
    p = gk.make_params(L, G, x.Q.shape[1], T, d, x.Q.shape[2], dtype=x.K.dtype, budget=(L * G * T) // 8,
                       rope_base=w.rope_base)
    K, V, Q = (t.cuda() for t in (x.K, x.V, x.Q))
    comp = gk.Compressor(p)
    comp(K, V, Q)
    a = comp.ctx.gracekv_export()
    ctx = gk.Context(p)
    slots = torch.empty(ctx.n_c + 2, dtype=torch.int32, device="cuda")
    ctx.gracekv_segment(V, slots)
    ctx.gracekv_build_trees(K, V, Q)
    ctx.gracekv_allocate()
    b = ctx.gracekv_export()
    for k in ["row_m", "row_Z", "row_ZC", "rtok", "unit_Uadd", "add_sel", "a", "b", "D", "U", "split_sel"]:
        assert np.array_equal(np.asarray(a[k]), np.asarray(b[k])), k


@pytest.mark.parametrize("wname,kw,alpha", [("small", dict(layers=[0, 1, 2, 3], heads=[0, 1], T=1000), 0.0),
                                            ("pr1", dict(T=700), 0.0),
                                            ("small", dict(layers=[0, 1, 2, 3], heads=[0, 1], T=1000), 0.6)])
def test_compress_host_matches_device(wname, kw, alpha):
    # The host-buffer pipeline (layer-group copies overlapped with the score
    # passes and the first tree launch; with a singleton floor the tree build
    # waits for every group) gives the device path's cache bits.
    from paper_2608_07001_gb300 import gracekv as gk
    w = synth.WORKLOADS[wname]
    x = synth.make_inputs(w, **kw)
    L, G, T, d = x.K.shape
    p = gk.make_params(L, G, x.Q.shape[1], T, d, x.Q.shape[2], dtype=x.K.dtype, budget=(L * G * T) // 8,
                       rope_base=w.rope_base, alpha_floor=alpha)
    comp = gk.Compressor(p)
    dev = comp(x.K.cuda(), x.V.cuda(), x.Q.cuda())
    E = comp.n_entries
    hc = gk.Cache.empty_host(dev.K.shape[0], d, L * G, x.K.dtype)
    ctx = gk.Context(p)
    Kh, Vh, Qh = (t.contiguous().pin_memory() for t in (x.K, x.V, x.Q))
    for _ in range(2):   # a second call reuses the context's device buffers
        n = ctx.gracekv_compress_host(Kh, Vh, Qh, hc)
        assert n == E
        for name in ["K", "V", "pos", "log_m", "src_lo", "src_hi"]:
            a, b = getattr(hc, name)[:n], getattr(dev, name)[:n].cpu()
            assert torch.equal(a.view(torch.int32) if a.dtype == torch.float32 else a,
                               b.view(torch.int32) if b.dtype == torch.float32 else b), name
        assert torch.equal(hc.offsets, dev.offsets.cpu())
