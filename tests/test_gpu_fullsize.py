"""Full-size parity: Llama-shaped cache at 32x, 32 layers x 8 KV heads x
131072 tokens x d 128 (bf16) with 64 observation queries per query head --
the workload and launch configuration bench.py times.

The plain oracle cannot run the whole pass at this size (its fp64 tree build
alone would take days), so the GPU result of one compression is checked on
outputs the oracle computes one by one, and by properties that hold at any size:

  curvature      kappa at 256 sampled interior positions: the oracle on a
                 33-row slice around each position (the slice holds every
                 window, so the value equals the full-sequence one)
  segmentation   every slot start equals the oracle's segmentation of the
                 whole context (its three segmentation layers, the paper's
                 prefix form of the dispersion), and curvature matches at all
                 positions; also the partition is locally optimal: moving any
                 of 160 sampled boundaries by up to 8 tokens does not raise the
                 DP objective beyond the near-tie margin
  row stats      all 256 rows of one KV-head group over all 131072 keys
  token values   every compressible token of that group
  trees          24 sampled units of that group: topology (near-tie aware),
                 D, U and the Add gain, from oracle curvature / statistics
  allocation     exact threshold structure of the selection over every built
                 op, tree consistency of the selected splits, entry count
  gather         the group's entries partition its covered slots; 256 sampled
                 entries equal the oracle's prototype of the same interval
  floor          a compression with the singleton floor at alpha 0.6 (App.
                 A.5 Stage I): B_floor within floor(alpha B_free); the accepted
                 set is the paper's acceptance walk replayed on the host from
                 the device's own token values and scores (gate, eta prefix,
                 proportional reduction, shares, skips); each accepted token
                 passes the gate gamma / N_c and is its own entry (m = 1) in the
                 final cache, with the input's K/V bits in the (l, g) that
                 holds the most of them
  multi-hop      a second compression with lambda = 0.3 (App. A.4): the
                 implied d-hat is the same for every (l, g), non-negative, sums
                 to 1 and is exactly zero at the first hop's seeds, chosen on
                 the host in fp64 from the direct token values (64 merged
                 selection parts, the last one ragged)
"""
from __future__ import annotations

import math

import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_07001_gb300 import synth
from tests import parity as P

pytestmark = pytest.mark.gpu

RATIO = 32.0
L_S, G_S = 13, 5          # the sampled KV-head group (layer, KV head)
SEED = 2026


def _seg_layers(L):
    return sorted({min(int(math.floor(r * L)), L - 1) for r in (0.33, 0.5, 0.67)})


@pytest.fixture(scope="module")
def run():
    import __graft_entry__ as g
    from paper_2608_07001_gb300 import gracekv as gk
    g.build()
    assert torch.cuda.is_available()
    w = synth.WORKLOADS["llama128k"]
    x = synth.make_inputs(w, device="cuda")
    L, G, T, d = x.K.shape
    Hq, W = x.Q.shape[1], x.Q.shape[2]
    B = gk.gracekv_budget_for_ratio(L, G, T, RATIO)
    p = gk.make_params(L, G, Hq, T, d, W, dtype=x.K.dtype, budget=B, rope_base=w.rope_base)
    comp = gk.Compressor(p)
    cache = comp(x.K, x.V, x.Q)
    torch.cuda.synchronize()
    ex = comp.ctx.gracekv_export()
    gq = Hq // G
    lg = L_S * G + G_S
    r = comp.ctx.recent
    Nc = comp.ctx.n_c
    off = cache.offsets.cpu().numpy()
    e0, e1 = int(off[lg]), int(off[lg + 1])
    out = dict(
        w=w, L=L, G=G, Hq=Hq, T=T, d=d, W=W, B=B, r=r, Nc=Nc, gq=gq, lg=lg,
        kappa=comp.kappa.cpu().double().numpy(),
        slots=comp.slots[:comp.n_slots + 1].cpu().numpy().astype(np.int64),
        J=comp.n_slots, E=comp.n_entries, b_free=comp.ctx.b_free, ex=ex, offsets=off,
        # the sampled group, on the host
        K1=x.K[L_S, G_S].double().cpu().numpy()[None, None],
        V1=x.V[L_S, G_S].double().cpu().numpy()[None, None],
        Q1=x.Q[L_S, G_S * gq:(G_S + 1) * gq].double().cpu().numpy()[None],
        Kraw=x.K[L_S, G_S].cpu(), Vraw=x.V[L_S, G_S].cpu(),
        cK=cache.K[e0:e1].cpu(), cV=cache.V[e0:e1].cpu(), cpos=cache.pos[e0:e1].cpu().numpy(),
        clogm=cache.log_m[e0:e1].cpu().numpy(), clo=cache.src_lo[e0:e1].cpu().numpy(),
        chi=cache.src_hi[e0:e1].cpu().numpy(),
        Vseg=x.V[_seg_layers(L)],   # stays on the device; sliced per sample
    )
    # oracle statistics of the sampled group (also used by the tree and gather checks)
    po = O.make_params(1, 1, gq, T, d, W, w.rope_base, recent=r)
    m, Z, ZC = O.row_stats(po, out["Q1"], out["K1"])
    out.update(po=po, om=m, oZ=Z, oZC=ZC, ortok=O.token_values(po, out["Q1"], out["K1"], m, Z))
    del x
    yield out
    comp.ctx.close()
    torch.cuda.empty_cache()


def _oracle_kappa(run, lo, hi):
    """Oracle curvature of positions [lo + 16, hi - 16) from rows [lo, hi)."""
    V = run["Vseg"][:, :, lo:hi].double().cpu().numpy()
    p = O.make_params(3, run["G"], run["Hq"], hi - lo, run["d"], run["W"], run["w"].rope_base,
                      seg_layers=(0, 1, 2))
    kap, _ = O.curvature(p, V)
    return kap[16:hi - lo - 16]


def test_curvature_sampled_positions(run):
    rng = np.random.default_rng(SEED)
    T = run["T"]
    pos = rng.choice(np.arange(16, T - 16), size=256, replace=False)
    err = max(abs(_oracle_kappa(run, i - 16, i + 17)[0] - run["kappa"][i]) for i in pos)
    print("kappa max abs err", err)
    assert err <= P.KAPPA_ATOL


def test_segmentation_valid_and_locally_optimal(run):
    s = run["slots"]
    ln = np.diff(s)
    assert s[0] == 0 and s[-1] == run["Nc"]
    assert np.all(ln[:-1] >= 16) and np.all(ln <= 128) and ln[-1] >= 1
    # boundary score from the oracle's robust z of the GPU curvature (surprisal 0)
    b = O.robust_z(run["kappa"])
    rng = np.random.default_rng(SEED + 1)
    J = len(s) - 1
    worst = -np.inf
    for j in rng.choice(np.arange(2, J - 1), size=160, replace=False):
        s0, s1, s2 = int(s[j - 1]), int(s[j]), int(s[j + 1])
        deltas = [dl for dl in range(-8, 9)
                  if 16 <= s1 + dl - s0 <= 128 and 16 <= s2 - s1 - dl <= 128]
        lo, hi = s0 - 1, s2
        V = run["Vseg"][:, :, lo:hi].double().cpu().numpy()
        p = O.make_params(3, run["G"], run["Hq"], hi - lo, run["d"], run["W"], run["w"].rope_base,
                          seg_layers=(0, 1, 2), recent=0)
        a_rel, i_rel = [], []
        for dl in deltas:
            a_rel += [s0 - lo, s1 + dl - lo]
            i_rel += [s1 + dl - lo, s2 - lo]
        wts = O.dp_weights(p, V, b[lo:hi], a_rel, i_rel).reshape(-1, 2).sum(axis=1)
        obj = dict(zip(deltas, wts))
        best = max(obj.values())
        gap = (best - obj[0]) / max(abs(best), 1e-300)
        worst = max(worst, gap)
        assert gap < P.NEAR_TIE, (j, s0, s1, s2, obj)
    print("largest relative improvement found", worst)


def test_segmentation_bit_exact_over_the_full_context(run):
    # The oracle's segmentation of the whole 131072-token context from the
    # three segmentation layers (the partition depends on nothing else), in
    # the paper's prefix form of the dispersion (App. B.3 Eq.
    # app_prefix_dispersion, pinned equal to the sample-variance definition
    # on CPU).  Every slot start must match; a differing DP decision is
    # allowed only at an endpoint where the oracle's best and second-best
    # predecessor values are within the near-tie margin.
    import time
    t0 = time.time()
    V = run["Vseg"].double().cpu().numpy()
    p = O.make_params(3, run["G"], run["Hq"], run["T"], run["d"], run["W"], run["w"].rope_base,
                      seg_layers=(0, 1, 2), recent=run["r"], disp_mode=1)
    seg = O.segment(p, V)
    del V
    kerr = float(np.abs(seg["kappa"] - run["kappa"]).max())
    og, gs = seg["slot_starts"].astype(np.int64), run["slots"]
    print(f"full-context segmentation: oracle {time.time() - t0:.0f} s, {len(og) - 1} slots, "
          f"kappa max abs err {kerr:.2e} over all {run['T']} positions")
    assert kerr <= P.KAPPA_ATOL
    if np.array_equal(og, gs):
        return
    # the decision that differs: the last endpoint both paths reach, going
    # back from N, whose predecessors differ
    so, sg = set(og.tolist()), set(gs.tolist())
    common = sorted(so & sg)
    for i in reversed(common[1:]):
        po = og[np.searchsorted(og, i) - 1]
        pg = gs[np.searchsorted(gs, i) - 1]
        if po != pg:
            best, second = seg["dp_best"][i], seg["dp_second"][i]
            margin = abs(best - second) / max(abs(best), 1e-300)
            print("slot starts differ at endpoint", i, "oracle margin", margin)
            assert margin < P.NEAR_TIE, (i, po, pg, margin)
            return
    raise AssertionError("slot starts differ")


def _group_rows(run, key):
    L, Hq, W, gq = run["L"], run["Hq"], run["W"], run["gq"]
    return run["ex"][key].reshape(L, Hq, W)[L_S, G_S * gq:(G_S + 1) * gq]


def test_row_stats_of_one_group(run):
    for k, ok in (("row_m", "om"), ("row_Z", "oZ"), ("row_ZC", "oZC")):
        a, b = _group_rows(run, k).astype(np.float64), run[ok][0]
        err = np.abs(a - b) / np.maximum(np.abs(b), 1e-30 if k != "row_m" else 1.0)
        print(k, "max rel err", err.max())
        assert err.max() <= P.ROW_RTOL * (1 if k == "row_m" else 10)


def test_token_values_of_one_group(run):
    Nc, lg = run["Nc"], run["lg"]
    g = run["ex"]["rtok"][lg * Nc:(lg + 1) * Nc].astype(np.float64)
    o = run["ortok"].reshape(-1)
    err = np.abs(g - o) / np.maximum(np.abs(o), 1e-3 * o.max())
    print("rtok max rel err", err.max())
    assert err.max() <= P.RTOK_RTOL


def test_trees_of_sampled_units(run):
    ex, J, lg, T = run["ex"], run["J"], run["lg"], run["T"]
    s = run["slots"]
    uf = ex["unit_first"]
    rng = np.random.default_rng(SEED + 2)
    js = [j for j in rng.permutation(np.arange(1, J - 1)) if s[j] >= 16 and s[j + 1] + 16 <= T][:24]
    worst_D = worst_U = worst_add = 0.0
    near = 0
    for j in js:
        sa, sb = int(s[j]), int(s[j + 1])
        kap = np.zeros(T)
        kap[sa:sb] = _oracle_kappa(run, sa - 16, sb + 16)
        tr = O.build_trees(run["po"], run["K1"], run["V1"], run["Q1"], kap, [sa, sb], run["om"],
                           run["oZ"], run["ortok"])
        nd = tr.nodes
        okey = {(int(nd["a"][v]), int(nd["b"][v])): v for v in range(len(nd["a"]))}
        uid = lg * J + j
        gs, ge = int(uf[uid]), int(uf[uid + 1])
        oa = tr.unit_Uadd[0]
        worst_add = max(worst_add, abs(ex["unit_Uadd"][uid] - oa) / max(abs(oa), 1e-30))
        for k in range(gs, ge):
            key = (int(ex["a"][k]), int(ex["b"][k]))
            assert key in okey, (j, key)
            v = okey[key]
            gn = int(ex["nchild"][k])
            if gn == -1:
                continue    # pending: never reached by the allocation
            on = int(nd["nchild"][v])
            gch = [(int(ex["a"][gs + ex["child0"][k] + q]), int(ex["b"][gs + ex["child0"][k] + q]))
                   for q in range(gn)]
            och = [(int(nd["a"][nd["child0"][v] + q]), int(nd["b"][nd["child0"][v] + q]))
                   for q in range(on)]
            if gch != och:
                margin = min(nd["m_cut"][v], nd["m_form"][v], nd["m_topk"][v], nd["m_ext"][v])
                assert margin < P.NEAR_TIE, (j, key, gch, och, margin)
                near += 1
                break
            oD = nd["D"][v]
            worst_D = max(worst_D, abs(ex["D"][k] - oD) / abs(oD) if oD else abs(ex["D"][k]))
            if gn > 0:
                scale = max(nd["R"][v] * max(abs(oD), 1e-300), 1e-300) / max(nd["cost"][v], 1)
                worst_U = max(worst_U, abs(ex["U"][k] - nd["U"][v]) / scale)
    print(f"units {len(js)} near-tie {near} D {worst_D:.3e} U {worst_U:.3e} Uadd {worst_add:.3e}")
    assert len(js) == 24
    assert worst_D <= P.D_RTOL and worst_U <= P.U_RTOL and worst_add <= P.U_RTOL


def test_allocation_threshold_structure(run):
    ex = run["ex"]
    J, L, G = run["J"], run["L"], run["G"]
    nu = L * G * J
    uf = ex["unit_first"]
    nch = ex["nchild"]
    isop = nch >= 2
    keys = np.concatenate([ex["unit_Uadd"], ex["kappa"][isop]]).astype(np.float64)
    cost = np.concatenate([np.ones(nu, np.int64), ex["cost"][isop].astype(np.int64)])
    sel = np.concatenate([ex["add_sel"] == 1, ex["split_sel"][isop] == 1])
    assert np.all(ex["split_sel"][~isop] != 1)
    used = int(cost[sel].sum())
    Bf = run["b_free"]
    assert used in (Bf, Bf - 1) or sel.all()
    assert run["E"] == run["L"] * run["G"] * (run["T"] - run["Nc"]) + used
    # tau with cost{key > tau} <= B_free < cost{key >= tau}
    order = np.argsort(-keys, kind="stable")
    cum = np.cumsum(cost[order])
    if cum[-1] <= Bf:
        assert sel.all()
        return
    tau = keys[order][np.searchsorted(cum, Bf, side="right")]
    assert sel[keys > tau].all(), "an op above the threshold was not selected"
    below = sel & (keys < tau)
    assert below.sum() <= 1 and (cost[below] == 1).all(), "more than the endgame op below tau"
    assert cost[sel & (keys == tau)].sum() <= Bf - cost[keys > tau].sum()
    # tree consistency: a selected split's node is exposed (its creator op was selected)
    parent = np.full(len(nch), -1, np.int64)
    unit_of = np.repeat(np.arange(nu), np.diff(uf))
    v = np.nonzero(isop)[0]
    for q in range(3):
        has = nch[v] > q
        parent[uf[unit_of[v[has]]] + ex["child0"][v[has]] + q] = v[has]
    sv = np.nonzero(ex["split_sel"] == 1)[0]
    roots = parent[sv] < 0
    assert np.all(sv[roots] == uf[unit_of[sv[roots]]])
    assert np.all(ex["add_sel"][unit_of[sv[roots]]] == 1)
    assert np.all(ex["split_sel"][parent[sv[~roots]]] == 1)
    print("tau", tau, "used", used, "of", Bf)


def test_gather_of_one_group(run):
    lo, hi = run["clo"], run["chi"]
    T, r, J, lg = run["T"], run["r"], run["J"], run["lg"]
    s = run["slots"]
    # recent window at the end as single tokens, the rest partitions the covered slots
    nrec = T - run["Nc"]
    assert np.array_equal(lo[-nrec:], np.arange(T - nrec, T)) and np.array_equal(hi[-nrec:], lo[-nrec:] + 1)
    lo, hi = lo[:-nrec], hi[:-nrec]
    assert np.all(hi > lo) and np.all(lo[1:] >= hi[:-1])
    covered = np.nonzero(run["ex"]["add_sel"][lg * J:(lg + 1) * J] == 1)[0]
    tok = np.zeros(T, np.int64)
    for a, b in zip(lo, hi):
        tok[a:b] += 1
    want = np.zeros(T, np.int64)
    for j in covered:
        want[s[j]:s[j + 1]] = 1
    assert np.array_equal(tok, want)
    # sampled entries against the oracle's prototype of the same interval
    rng = np.random.default_rng(SEED + 3)
    idx = rng.choice(len(lo), size=min(256, len(lo)), replace=False)
    worst_k = worst_v = worst_m = 0.0
    for e in idx:
        a, b = int(lo[e]), int(hi[e])
        if b - a == 1:
            assert torch.equal(run["cK"][e], run["Kraw"][a]) and torch.equal(run["cV"][e], run["Vraw"][a])
            assert run["cpos"][e] == a and run["clogm"][e] == 0.0
            continue
        o = O.eval_interval(run["po"], run["K1"], run["V1"], run["Q1"], run["om"], run["oZ"],
                            run["ortok"], 0, 0, a, b)
        assert run["cpos"][e] == o["pos"]
        gk_, gv_ = run["cK"][e].double().numpy(), run["cV"][e].double().numpy()
        worst_k = max(worst_k, np.linalg.norm(gk_ - o["ktil"]) / np.linalg.norm(o["ktil"]))
        worst_v = max(worst_v, np.linalg.norm(gv_ - o["vtil"]) / np.linalg.norm(o["vtil"]))
        worst_m = max(worst_m, abs(run["clogm"][e] - o["logm"]))
    print(f"prototypes K {worst_k:.3e} V {worst_v:.3e} log m {worst_m:.3e}")
    assert worst_k <= P.PROTO_RTOL[torch.bfloat16] and worst_v <= P.PROTO_RTOL[torch.bfloat16]
    assert worst_m <= P.LOGM_ATOL


def test_multihop_full_size_properties(run):
    from paper_2608_07001_gb300 import gracekv as gk
    w = run["w"]
    L, G, T, d, Hq, W, Nc = (run[k] for k in ("L", "G", "T", "d", "Hq", "W", "Nc"))
    lam = 0.3
    x = synth.make_inputs(w, device="cuda")
    Qg = synth.make_graph_queries(w, gk.graph_layers(L), device="cuda")
    p = gk.make_params(L, G, Hq, T, d, W, dtype=x.K.dtype, budget=run["B"], rope_base=w.rope_base,
                       lambda_graph=lam)
    comp = gk.Compressor(p)
    comp(x.K, x.V, x.Q, Qg=Qg)
    torch.cuda.synchronize()
    R = comp.ctx.gracekv_export()["rtok"].reshape(L * G, Nc)
    comp.ctx.close()
    del x, Qg
    torch.cuda.empty_cache()
    shat = run["ex"]["rtok"].reshape(L * G, Nc)       # the direct values, same inputs
    one_m = np.float32(np.float32(1.0) - np.float32(lam))
    prod = one_m * shat                               # fp32, as the device rounds it
    dh = (R.astype(np.float64) - prod.astype(np.float64)) / lam
    mean = dh.mean(0)
    # the same d-hat in every row, up to the rounding of the mix's last add
    tol = 4 * 2.0 ** -24 * (np.abs(R) + np.abs(prod)).max(0).astype(np.float64) / lam
    assert np.all(np.abs(dh - mean[None]) <= tol[None] + 1e-15)
    assert mean.min() >= -tol.max() and abs(mean.sum() - 1.0) < 1e-4
    # the first hop's seeds: S descending (ties lower t) while fewer than 64
    # and the mass is below 0.9 (Eq. app_global_seed_score); there d-hat is 0
    # and R is exactly the rounded (1 - lambda) s-hat
    S = shat.astype(np.float64).mean(0)
    S = S / (S.sum() + 1e-6)
    order = np.lexsort((np.arange(Nc), -S))
    cum, seeds, before = 0.0, [], []
    while len(seeds) < 64 and cum < 0.9:
        seeds.append(int(order[len(seeds)]))
        before.append(cum)
        cum += S[seeds[-1]]
    # skip seeds whose rank or membership fp32 sums could change
    gap = np.abs(np.diff(S[order[:len(seeds) + 1]])) / S[order[0]]
    sure = [t for k, t in enumerate(seeds) if gap[k] > 1e-4 and (k == 0 or gap[k - 1] > 1e-4)]
    if len(seeds) < 64 or 0.9 - before[-1] < 1e-4:
        sure = [t for t in sure if t != seeds[-1] or 0.9 - before[-1] >= 1e-4]
    print("multihop full size: seeds", len(seeds), "checked", len(sure), "d-hat max", mean.max())
    assert len(sure) >= len(seeds) // 2
    for t in sure:
        assert np.all(R[:, t] == prod[:, t]), t


def floor_replay(R, f, slots, cap, gamma=1.2, eta=0.95):
    """App. A.5 Stage I (the paragraph after Eq. app_floor_cap) replayed on the
    host from the device's own token values R and floor scores f (fp32,
    [L G][N_c]): per (l, g) the gated tokens (f >= gamma / N_c in fp32) in
    order f descending, ties lower t, up to the longest prefix whose value sum
    stays <= eta (sums in 2^-40 fixed point, so exact and order-free); the
    proportional reduction when the joint cost C0 exceeds cap; the per-head
    share floor(cap n' / sum n'); then the walk that accepts each kept
    candidate whose path fits what is left of the share and skips the
    others.  Returns the accepted mask, B_floor and the number of skips."""
    import bisect
    LG, Nc = R.shape
    gate = np.float32(gamma / Nc)
    eta_fx = int(eta * 2.0 ** 40)
    fx = np.floor(R.astype(np.float64) * 2.0 ** 40).astype(np.int64)
    slots = np.asarray(slots, np.int64)
    slot_of = np.searchsorted(slots, np.arange(Nc), side="right") - 1
    cands, C0 = [], 0
    for lg in range(LG):
        order = np.lexsort((np.arange(Nc), -f[lg].astype(np.float64)))
        gated = order[f[lg][order] >= gate]
        n = int(np.searchsorted(np.cumsum(fx[lg][gated]), eta_fx, side="right"))
        c = gated[:n]
        cands.append(c)
        if n:
            S = np.zeros(Nc, bool)
            S[c] = True
            start = np.zeros(Nc, bool)
            start[slots[:-1]] = True
            prev_in = np.concatenate([[True], S[:-1]]) | start
            runs = ~S & prev_in
            has = np.bincount(slot_of[c], minlength=len(slots) - 1) > 0
            C0 += n + int(runs[has[slot_of]].sum())
    keep = [len(c) if C0 <= cap or not len(c) else max(1, len(c) * cap // C0) for c in cands]
    nkeep = sum(keep)
    acc = np.zeros((LG, Nc), bool)
    B_floor = skips = 0
    for lg in range(LG):
        if not keep[lg]:
            continue
        share, used, by_slot = cap * keep[lg] // nkeep, 0, {}
        for t in cands[lg][:keep[lg]]:
            t = int(t)
            j = int(slot_of[t])
            sa, sb = int(slots[j]), int(slots[j + 1])
            lst = by_slot.setdefault(j, [])
            i = bisect.bisect_left(lst, t)
            lo = lst[i - 1] + 1 if i > 0 else sa
            hi = lst[i] - 1 if i < len(lst) else sb - 1
            cost = (0 if lst else 1) + (lo < t) + (t < hi)
            if used + cost <= share:
                used += cost
                lst.insert(i, t)
                acc[lg, t] = True
            else:
                skips += 1
        B_floor += used
    return acc, B_floor, skips


def test_singleton_floor_full_size_properties(run):
    from paper_2608_07001_gb300 import gracekv as gk
    w = run["w"]
    L, G, T, d, Hq, W, Nc = (run[k] for k in ("L", "G", "T", "d", "Hq", "W", "Nc"))
    alpha = 0.6
    x = synth.make_inputs(w, device="cuda")
    p = gk.make_params(L, G, Hq, T, d, W, dtype=x.K.dtype, budget=run["B"], rope_base=w.rope_base,
                       alpha_floor=alpha)
    comp = gk.Compressor(p)
    cache = comp(x.K, x.V, x.Q)
    torch.cuda.synchronize()
    fl = comp.ctx.gracekv_export_floor()
    R = comp.ctx.gracekv_export()["rtok"].reshape(L * G, Nc)
    slots = comp.slots[:comp.n_slots + 1].cpu().numpy()
    E = comp.n_entries
    off = cache.offsets.cpu().numpy()
    pos, lo, hi = (getattr(cache, k)[:E].cpu().numpy() for k in ("pos", "src_lo", "src_hi"))
    logm = cache.log_m[:E].cpu().numpy()
    acc, f = fl["accepted"].astype(bool), fl["f"]
    lg_b = int(acc.sum(1).argmax())                       # the (l, g) with the most floor tokens
    Ks, Vs = x.K[lg_b // G, lg_b % G].cpu(), x.V[lg_b // G, lg_b % G].cpu()
    cK, cV = cache.K[:E].cpu(), cache.V[:E].cpu()
    comp.ctx.close()
    del x, cache
    torch.cuda.empty_cache()
    cap = int(math.floor(alpha * run["b_free"]))
    assert 0 < fl["B_floor"] <= cap and E <= run["B"]
    # the accepted set is the paper's walk on the device's own scores
    want, want_B, skips = floor_replay(R, f, slots, cap)
    print("floor full size: replayed acceptance, skipped candidates", skips)
    np.testing.assert_array_equal(acc, want)
    assert fl["B_floor"] == want_B
    gate = np.float32(1.2 / Nc)
    n_acc = 0
    for lg in range(L * G):
        a_idx = np.nonzero(acc[lg])[0]
        if len(a_idx) == 0:
            continue
        n_acc += len(a_idx)
        fmin = f[lg, a_idx].min()
        assert fmin >= gate * np.float32(1 - 1e-6), lg
        e0, e1 = int(off[lg]), int(off[lg + 1])
        single = (hi[e0:e1] - lo[e0:e1]) == 1
        where = {int(t): e0 + k for k, t in enumerate(pos[e0:e1]) if single[k]}
        for t in a_idx:
            e = where.get(int(t))                         # context starts at 0 here
            assert e is not None and logm[e] == 0.0, (lg, int(t))
            if lg == lg_b:
                assert torch.equal(cK[e], Ks[t]) and torch.equal(cV[e], Vs[t])
    print("floor full size: accepted", n_acc, "B_floor", fl["B_floor"], "cap", cap,
          "bit-checked (l, g)", lg_b, int(acc[lg_b].sum()))
    assert n_acc > 0
