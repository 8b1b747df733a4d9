"""Pins of the oracle's ablation variants (App. B.4 last paragraph, App. C.1).

"w/o CS": uniform slots of target length 64 instead of the curvature DP, no
curvature split candidates and no curvature reward (midpoint only).
"w/o GA": fixed per-(l, g) capacity instead of one shared budget.
"""
import numpy as np
import pytest

import oracle as O


def rand_inputs(seed, L=2, G=2, gq=1, T=300, d=8, W=4):
    rng = np.random.default_rng(seed)
    K = rng.normal(size=(L, G, T, d))
    V = rng.normal(size=(L, G, T, d))
    # a few loud tokens so that allocation has something to choose
    K[:, :, rng.integers(0, T, 12)] *= 3.0
    Q = rng.normal(size=(L, G * gq, W, d))
    return K, V, Q


@pytest.mark.parametrize("N,expect", [(100, [0, 50, 100]), (95, [0, 95]), (96, [0, 48, 96]),
                                      (10, [0, 10]), (256, [0, 64, 128, 192, 256]),
                                      (161, [0, 53, 107, 161])])
def test_uniform_slots_closed_form(oracle_lib, N, expect):
    # J = round-half-up(N / 64) slots, starts c_s + floor(j N / J)
    cs = 7
    p = O.make_params(1, 1, 1, cs + N + 32, 8, 2, 0.0, ctx_start=cs, recent=32)
    got = O.uniform_slots(p)
    np.testing.assert_array_equal(got, np.asarray(expect) + cs)
    L_ = np.diff(got)
    assert L_.max() - L_.min() <= 1


def test_wo_cs_splits_only_at_the_midpoint(oracle_lib):
    K, V, Q = rand_inputs(1)
    res = O.run(K, V, Q, 120, 1e4, recent=16, seg_mode=1, k_cand=0, lambda_kappa=0.0)
    nd = res["trees"].nodes
    starts = res["seg"]["slot_starts"]
    assert np.all(res["seg"]["kappa"] == 0)
    np.testing.assert_array_equal(starts, O.uniform_slots(res["params"]))
    n_bin = 0
    for v in range(len(nd["a"])):
        if nd["nchild"][v] == 2 and nd["form"][v] == 0:        # binary split
            a, b, c0 = nd["a"][v], nd["b"][v], nd["child0"][v]
            assert nd["b"][c0] == a + (b - a) // 2 == nd["a"][c0 + 1]
            n_bin += 1
    assert n_bin > 10
    # with the paper's candidates some binary cut leaves the midpoint
    full = O.run(K, V, Q, 120, 1e4, recent=16, seg_mode=1)
    ndf = full["trees"].nodes
    off = [ndf["b"][ndf["child0"][v]] - (ndf["a"][v] + (ndf["b"][v] - ndf["a"][v]) // 2)
           for v in range(len(ndf["a"])) if ndf["nchild"][v] == 2 and ndf["form"][v] == 0]
    assert any(o != 0 for o in off)


def _sub_forest(tr: O.Trees, lg: int, J: int) -> O.Trees:
    nd = tr.nodes
    idx = np.nonzero(nd["lg"] == lg)[0]
    n0, n1 = int(idx[0]), int(idx[-1]) + 1
    assert n1 - n0 == len(idx)                     # a pair's nodes are contiguous
    sub = {f: nd[f][n0:n1].copy() for f in nd}
    for f in ("child0", "parent"):
        sub[f] = np.where(sub[f] >= 0, sub[f] - n0, sub[f]).astype(np.int32)
    uadd = tr.unit_Uadd[lg * J:(lg + 1) * J].copy()
    uroot = tr.unit_root[lg * J:(lg + 1) * J] - n0
    return O.Trees(sub, uadd, uroot.astype(np.int64), J), n0, n1


@pytest.mark.parametrize("B", [97, 200, 400])
def test_quota_allocation_is_per_pair_greedy(oracle_lib, B):
    # with fixed capacities the shared heap decomposes: each (l, g) receives
    # exactly the selection the one-budget greedy makes on its own trees with
    # budget floor(B_free / LG) (+1 for the first B_free mod LG pairs)
    K, V, Q = rand_inputs(2, L=2, G=2)
    res = O.run(K, V, Q, B, 1e4, recent=16, quota_alloc=1)
    p, tr = res["params"], res["trees"]
    LG, J = p.L * p.G, tr.n_slots
    Bf = res["B_free"]
    assert Bf > LG
    used_total = 0
    for lg in range(LG):
        q = Bf // LG + (1 if lg < Bf % LG else 0)
        sub, n0, n1 = _sub_forest(tr, lg, J)
        p1 = O.make_params(1, 1, 1, p.T, p.d, p.W, 1e4, recent=p.recent)
        a1, s1, u1 = O.allocate(p1, q, sub)
        np.testing.assert_array_equal(res["add_sel"][lg * J:(lg + 1) * J], a1)
        np.testing.assert_array_equal(res["split_sel"][n0:n1], s1)
        assert u1 <= q
        used_total += u1
    assert used_total == res["used"]
    # the shared budget moves capacity between pairs: another selection
    shared = O.run(K, V, Q, B, 1e4, recent=16)
    assert shared["used"] >= res["used"]
    assert np.any(shared["add_sel"] != res["add_sel"]) or np.any(shared["split_sel"] != res["split_sel"])


def test_quota_with_one_pair_is_the_shared_budget(oracle_lib):
    K, V, Q = rand_inputs(3, L=1, G=1)
    a = O.run(K, V, Q, 30, 1e4, recent=16, quota_alloc=1)
    b = O.run(K, V, Q, 30, 1e4, recent=16)
    np.testing.assert_array_equal(a["add_sel"], b["add_sel"])
    np.testing.assert_array_equal(a["split_sel"], b["split_sel"])
