"""Pins of the oracle's singleton floor (App. A.5 Stage I, App. C.4).

f = width-7 max-pool of (1 - c) R + c mean_{l,g} R (Eq. app_floor_score); the
gate f >= gamma / N_c (Eq. app_floor_gate); candidates up to value mass eta;
path charging and the cap B_floor <= floor(alpha B_base) (Eq. app_floor_cap);
forced extraction inside the prototype trees; the floor's ops execute before
the auction.
"""
import numpy as np
import pytest
from scipy.ndimage import maximum_filter1d

import oracle as O


def inputs(seed, L=2, G=2, T=400, d=8, W=4, spikes=12):
    rng = np.random.default_rng(seed)
    K = rng.normal(size=(L, G, T, d))
    V = rng.normal(size=(L, G, T, d))
    K[:, :, rng.integers(0, T, spikes)] *= 3.0
    Q = rng.normal(size=(L, G, W, d))
    return K, V, Q


def test_floor_score_is_a_clipped_max_pool_of_the_consensus_mix(oracle_lib):
    rng = np.random.default_rng(0)
    L, G, Nc = 2, 3, 50
    R = rng.random((L * G, Nc))
    R /= R.sum(1, keepdims=True)
    p = O.make_params(L, G, G, Nc + 8, 8, 2, 0.0, recent=8, alpha_floor=0.6)
    f, acc, bf, nc = O.floor(p, R, [0, 25, 50], 10 ** 6)
    mix = 0.5 * R + 0.5 * R.mean(0, keepdims=True)
    ref = maximum_filter1d(mix, size=7, axis=1, mode="constant", cval=-np.inf)
    np.testing.assert_allclose(f, ref, rtol=0, atol=1e-15)
    # identical heads: the consensus is the head itself
    R2 = np.tile(R[:1], (L * G, 1))
    f2, *_ = O.floor(p, R2, [0, 25, 50], 10 ** 6)
    np.testing.assert_allclose(f2, maximum_filter1d(R2, 7, axis=1, mode="constant", cval=-np.inf), atol=1e-15)


def test_flat_heads_buy_no_singletons(oracle_lib):
    # f = 1 / N_c everywhere is below the gate 1.2 / N_c
    L, G, Nc = 1, 2, 64
    R = np.full((L * G, Nc), 1.0 / Nc)
    p = O.make_params(L, G, G, Nc + 8, 8, 2, 0.0, recent=8, alpha_floor=0.6)
    f, acc, bf, nc = O.floor(p, R, [0, 32, 64], 10 ** 6)
    assert nc == 0 and bf == 0 and acc.sum() == 0


def test_candidates_stop_before_the_value_mass_eta(oracle_lib):
    # one head: values 0.5, 0.25, 0.125, 0.1, then a tail below the gate
    # 1.2 / N_c; eta 0.95 admits the first three (0.875) but not the fourth
    # (0.975)
    Nc = 40
    R = np.full(Nc, 0.025 / 36)
    R[[5, 20, 33, 37]] = [0.5, 0.25, 0.125, 0.1]
    p = O.make_params(1, 1, 1, Nc + 8, 8, 2, 0.0, recent=8, alpha_floor=1.0, floor_c=0.0,
                      floor_half=0)
    f, acc, bf, nc = O.floor(p, R[None], [0, 10, 30, 40], 10 ** 6)
    assert nc == 3
    assert set(np.nonzero(acc[0])[0]) == {5, 20, 33}
    # each isolated in its own slot: Add + extraction with two non-empty sides = 3 entries
    assert bf == 9


def _frontier_cost(acc_row, starts):
    tot = 0
    for a, b in zip(starts[:-1], starts[1:]):
        s = acc_row[a:b].astype(bool)
        if not s.any():
            continue
        runs = int(np.sum(~s & np.concatenate([[True], s[:-1]])))
        tot += int(s.sum()) + runs
    return tot


@pytest.mark.parametrize("alpha,B", [(0.6, 150), (0.6, 400), (0.05, 400), (0.3, 1200)])
def test_floor_accounting_trees_and_cache(oracle_lib, alpha, B):
    K, V, Q = inputs(1)
    res = O.run(K, V, Q, B, 1e4, recent=16, alpha_floor=alpha)
    p, fl, tr = res["params"], res["floor"], res["trees"]
    starts = res["seg"]["slot_starts"] - p.ctx_start
    acc = fl["accepted"]
    assert acc.sum() > 0
    # B_floor = the frontier entries the floor leaves (closed form) <= its cap
    assert fl["B_floor"] == sum(_frontier_cost(acc[lg], starts) for lg in range(p.L * p.G))
    assert fl["B_floor"] <= int(np.floor(alpha * res["B_free"]))
    nd = tr.nodes
    J = tr.n_slots
    # every accepted position is a leaf {t}; every floor op extracts the accepted
    # position of largest f inside its node; every floor op is selected
    for lg in range(p.L * p.G):
        m = nd["lg"] == lg
        leaves = {(int(a), int(b)) for a, b in zip(nd["a"][m], nd["b"][m]) if b - a == 1}
        for t in np.nonzero(acc[lg])[0]:
            assert (t + p.ctx_start, t + p.ctx_start + 1) in leaves
    for v in np.nonzero(nd["floor_op"])[0]:
        a, b, lg = int(nd["a"][v]), int(nd["b"][v]), int(nd["lg"][v])
        inside = [t for t in range(a, b) if acc[lg, t - p.ctx_start]]
        best = max(inside, key=lambda t: (fl["f"][lg, t - p.ctx_start], -t))
        ch = [(int(nd["a"][nd["child0"][v] + k]), int(nd["b"][nd["child0"][v] + k]))
              for k in range(nd["nchild"][v])]
        assert (best, best + 1) in ch and nd["form"][v] == 1
        assert res["split_sel"][v] == 1
    assert np.all(res["add_sel"][fl["unit_floor"] == 1] == 1)
    assert res["used"] <= res["B_free"]
    # exact singleton anchors: original K/V, their position, log m = 0
    cache = res["cache"]
    off = cache["offsets"]
    for lg in range(p.L * p.G):
        l, g = divmod(lg, p.G)
        lo, hi = off[lg], off[lg + 1]
        byt = {int(cache["src_lo"][e]): e for e in range(lo, hi) if cache["src_hi"][e] - cache["src_lo"][e] == 1}
        for t in np.nonzero(acc[lg])[0]:
            e = byt[t + p.ctx_start]
            assert cache["pos"][e] == t + p.ctx_start and cache["log_m"][e] == 0.0
            np.testing.assert_array_equal(cache["K"][e], K[l, g, t + p.ctx_start])


def test_floor_ops_first_equals_infinite_keys(oracle_lib):
    # executing the floor ops before the heap (the paper's order) selects the
    # same ops as one heap in which the floor's Adds and extractions carry an
    # infinite key: the formulation the device's threshold allocation uses
    K, V, Q = inputs(2)
    res = O.run(K, V, Q, 400, 1e4, recent=16, alpha_floor=0.6)
    tr = res["trees"]
    nodes = {k: v.copy() for k, v in tr.nodes.items()}
    nodes["U"] = np.where(nodes["floor_op"] == 1, np.inf, nodes["U"])
    uadd = np.where(res["floor"]["unit_floor"] == 1, np.inf, tr.unit_Uadd)
    tr2 = O.Trees(nodes, uadd, tr.unit_root, tr.n_slots)
    a2, s2, u2 = O.allocate(res["params"], res["B_free"], tr2)
    np.testing.assert_array_equal(a2, res["add_sel"])
    np.testing.assert_array_equal(s2, res["split_sel"])
    assert u2 == res["used"]


def test_alpha_zero_and_fullkv_are_unchanged(oracle_lib):
    K, V, Q = inputs(3, L=1, G=2)
    a = O.run(K, V, Q, 300, 1e4, recent=16)
    b = O.run(K, V, Q, 300, 1e4, recent=16, alpha_floor=0.0)
    np.testing.assert_array_equal(a["split_sel"], b["split_sel"])
    # x = 1: everything fits, the cache is the FullKV cache with or without a floor
    T = K.shape[2]
    c = O.run(K, V, Q, 2 * T, 1e4, recent=16, alpha_floor=0.6)
    np.testing.assert_array_equal(c["cache"]["K"], K.reshape(-1, K.shape[-1]))
    assert np.all(c["cache"]["log_m"] == 0)


@pytest.mark.parametrize("alpha,acc0,acc1,b_floor", [
    (0.6, {5, 15, 25}, {10}, 10),    # cap 12: n' = 3, 1; shares 9, 3
    (0.5, {5, 15, 25}, set(), 7),    # cap 10: n' = 3, 1; shares 7, 2 < head 1's cost 3
    (0.35, {5}, set(), 3),           # cap 7: n' = 2, 1; shares 4, 2; {5, 15} costs 5 > 4
])
def test_proportional_reduction_and_per_head_shares(oracle_lib, alpha, acc0, acc1, b_floor):
    # Worked by hand (Eq. app_floor_cap and its per-head safeguard).  f = R
    # (no consensus, no pooling).  Head 0: six spikes of 0.15, three interior,
    # non-adjacent ones per slot: joint cost 3 + 4 = 7 per slot.  Head 1: two
    # spikes of 0.45, one per slot: 1 + 2 = 3 per slot.  C0 = 14 + 6 = 20 over
    # the cap floor(alpha 20): each head keeps max(1, floor(n cap / C0)) of
    # its candidates (ties: lower t), may spend floor(cap n' / sum n'), and
    # accepts, in order, each candidate whose path still fits.
    Nc = 80
    R = np.zeros((2, Nc))
    R[0] = 0.1 / 74
    R[0, [5, 15, 25, 45, 55, 65]] = 0.15
    R[1] = 0.1 / 78
    R[1, [10, 50]] = 0.45
    p = O.make_params(1, 2, 2, Nc + 8, 8, 2, 0.0, recent=8, alpha_floor=alpha, floor_c=0.0,
                      floor_half=0)
    f, acc, bf, nc = O.floor(p, R, [0, 40, 80], 20)
    assert nc == 8
    assert set(np.nonzero(acc[0])[0]) == acc0 and set(np.nonzero(acc[1])[0]) == acc1
    assert bf == b_floor <= int(alpha * 20)


@pytest.mark.parametrize("R0,share,acc0,used0", [
    # share 5; head 0 in f order: 10 (slot [0, 40) uncovered: Add + two sides = 3),
    # 50 (slot [40, 80) uncovered: 3; 3 + 3 = 6 > share 5, skipped),
    # 11 (its interval is now [11, 39]: one new side, 1; 3 + 1 = 4 <= 5)
    ({10: 0.4, 50: 0.3, 11: 0.2}, 5, {10, 11}, 4),
    # share 6: 10 (3), 12 (interval [11, 39]: two sides, 2; total 5), 50 (3;
    # 5 + 3 = 8 > 6: skipped),
    # 11 (interval [11, 11] is already {11}: free, 0)
    ({10: 0.3, 12: 0.25, 50: 0.2, 11: 0.15}, 6, {10, 11, 12}, 5),
])
def test_an_unaffordable_candidate_is_skipped_and_later_ones_still_accepted(oracle_lib, R0, share, acc0,
                                                                             used0):
    # Worked by hand (App. A.5 Stage I, the paragraph after Eq. app_floor_cap:
    # a candidate is accepted only when its complete path remains feasible,
    # and the floor is not disabled for a whole head when the budget is
    # tight).  f = R (no consensus, no pooling), slots [0, 40) and [40, 80).
    # Head 1: candidates 0, 1, 2 at the start of slot [0, 40): joint cost
    # 3 + one run = 4.  No proportional reduction (C0 <= cap), n' = 3 and
    # len(R0), cap = C0, and each head's share is floor(cap n' / sum n').
    Nc = 80
    R = np.zeros((2, Nc))
    R[0] = (1.0 - sum(R0.values())) / (Nc - len(R0)) / 4      # below the gate 1.2 / N_c
    for t, v in R0.items():
        R[0, t] = v
    R[1] = 0.01 / (Nc - 3) / 4
    R[1, [0, 1, 2]] = [0.4, 0.3, 0.2]
    starts = [0, 40, 80]
    c0 = _frontier_cost(np.isin(np.arange(Nc), list(R0)).astype(np.uint8), starts)
    cap = c0 + 4
    assert cap * len(R0) // (len(R0) + 3) == share   # the share the cases are worked against
    p = O.make_params(1, 2, 2, Nc + 8, 8, 2, 0.0, recent=8, alpha_floor=1.0, floor_c=0.0,
                      floor_half=0)
    f, acc, bf, nc = O.floor(p, R, starts, cap)
    assert nc == len(R0) + 3
    assert set(np.nonzero(acc[0])[0]) == acc0
    assert set(np.nonzero(acc[1])[0]) == {0, 1, 2}
    assert bf == used0 + 4
    # the accepted set's closed-form frontier count is what was charged
    assert _frontier_cost(acc[0], starts) == used0
