"""Pins of the oracle's greedy allocation (App. A.5 Stage II, App. C.3).

The oracle's heap is compared with (1) a naive greedy that rescans every
exposed op each step, (2) an exhaustive optimum over all joint frontiers
(App. C.2 frontier counting N(v) = 1 + prod N(child)), and (3) the
bottleneck-key threshold algorithm the CUDA allocator implements, written
here in plain Python so that its equivalence with the heap is checked on CPU.
"""
import itertools

import numpy as np
import pytest

import oracle as O


def random_forest(rng, n_units, max_n, uvals=None, ext_p=0.35, lg_of_unit=None):
    keys = ["lg", "slot", "a", "b", "parent", "child0", "nchild", "form", "cost", "floor_op"]
    fkeys = ["D", "Ddrop", "R", "U", "kappa", "kscale", "m_cut", "m_form", "m_topk", "m_ext"]
    nd = {k: [] for k in keys + fkeys}
    roots, uadd = [], []

    def draw():
        if uvals is not None:
            return float(rng.choice(uvals))
        return float(rng.exponential())

    def add(lg, j, a, b, parent):
        i = len(nd["a"])
        for k, v in zip(keys, [lg, j, a, b, parent, -1, 0, -1, 0, 0]):
            nd[k].append(v)
        for k in fkeys:
            nd[k].append(0.0)
        return i

    pos = 0
    for u in range(n_units):
        n = int(rng.integers(1, max_n + 1))
        lg = 0 if lg_of_unit is None else lg_of_unit[u]
        root = add(lg, u, pos, pos + n, -1)
        roots.append(root)
        uadd.append(draw())
        q = [root]
        while q:
            v = q.pop(0)
            a, b = nd["a"][v], nd["b"][v]
            if b - a < 2:
                continue
            if b - a >= 2 and rng.random() < ext_p:
                p = int(rng.integers(a, b))
                ch = [(x, y) for x, y in ((a, p), (p, p + 1), (p + 1, b)) if y > x]
            else:
                xi = int(rng.integers(a + 1, b))
                ch = [(a, xi), (xi, b)]
            nd["child0"][v] = len(nd["a"])
            nd["nchild"][v] = len(ch)
            nd["cost"][v] = len(ch) - 1
            nd["U"][v] = draw()
            for (x, y) in ch:
                q.append(add(lg, u, x, y, v))
        pos += n
    arr = {k: np.asarray(nd[k], dtype=np.int32) for k in keys}
    arr.update({k: np.asarray(nd[k], dtype=np.float64) for k in fkeys})
    return O.Trees(arr, np.asarray(uadd), np.asarray(roots, dtype=np.int64), n_units)


def heap_alloc(tr, B):
    p = O.make_params(1, 1, 1, 8, 2, 1, 0.0)
    p.L, p.G = 1, 1
    add, split, used = O.allocate(p, B, tr)
    return add, split, used


def op_key(tr, op):
    nd = tr.nodes
    kind, x = op
    if kind == "add":
        u, v = x, tr.unit_root[x]
        U = tr.unit_Uadd[x]
    else:
        v = x
        u = int(nd["slot"][v])
        U = nd["U"][v]
    return (-U, u, nd["a"][v], -nd["b"][v])


def op_cost(tr, op):
    return 1 if op[0] == "add" else int(tr.nodes["cost"][op[1]])


def children_ops(tr, op):
    nd = tr.nodes
    if op[0] == "add":
        vs = [tr.unit_root[op[1]]]
    else:
        c0, nc = nd["child0"][op[1]], nd["nchild"][op[1]]
        vs = list(range(c0, c0 + nc))
    return [("split", int(v)) for v in vs if nd["b"][v] - nd["a"][v] >= 2]


def naive_greedy(tr, B):
    exposed = [("add", u) for u in range(len(tr.unit_Uadd))]
    R = B
    done = set()
    while R > 0 and exposed:
        best = min(exposed, key=lambda o: op_key(tr, o))
        exposed.remove(best)
        c = op_cost(tr, best)
        if c > R:
            continue
        R -= c
        done.add(best)
        exposed.extend(children_ops(tr, best))
    return done, B - R


def sel_set(tr, add, split):
    s = {("add", u) for u in np.nonzero(add)[0]}
    s |= {("split", int(v)) for v in np.nonzero(split)[0]}
    return s


def kappa_threshold_alloc(tr, B):
    """The CUDA allocator's algorithm, in plain Python.

    kappa(op) = min(U(op), kappa(creator)); tau is the cost-weighted
    threshold with cost{kappa > tau} <= B < cost{kappa >= tau}; every op with
    kappa > tau is selected; ops with kappa == tau are replayed unit by unit
    (ascending unit) with a per-unit queue (U desc, a asc, b desc); an op that
    does not fit is discarded with its subtree; if one unit of budget is left,
    the best exposed cost-1 op (U desc, unit asc, a asc, b desc) takes it.
    """
    nd = tr.nodes
    kap, creator = {}, {}
    ops = []
    for u in range(len(tr.unit_Uadd)):
        o = ("add", u)
        kap[o] = tr.unit_Uadd[u]
        creator[o] = None
        ops.append(o)
        stack = [o]
        while stack:
            x = stack.pop()
            for c in children_ops(tr, x):
                kap[c] = min(nd["U"][c[1]], kap[x])
                creator[c] = x
                ops.append(c)
                stack.append(c)
    total = sum(op_cost(tr, o) for o in ops)
    if total <= B:
        return set(ops), total
    vals = sorted({kap[o] for o in ops}, reverse=True)
    tau = None
    for v in vals:
        if sum(op_cost(tr, o) for o in ops if kap[o] >= v) > B:
            tau = v
            break
    sel = {o for o in ops if kap[o] > tau}
    R = B - sum(op_cost(tr, o) for o in sel)
    unit_of = lambda o: o[1] if o[0] == "add" else int(nd["slot"][o[1]])
    tie_units = sorted({unit_of(o) for o in ops if kap[o] == tau})
    discarded = set()
    for u in tie_units:
        if R == 0:
            break
        q = [o for o in ops if unit_of(o) == u and kap[o] == tau
             and (creator[o] is None or creator[o] in sel)]
        while q and R > 0:
            best = min(q, key=lambda o: op_key(tr, o))
            q.remove(best)
            c = op_cost(tr, best)
            if c > R:
                discarded.add(best)
                continue
            R -= c
            sel.add(best)
            q.extend(x for x in children_ops(tr, best) if kap[x] == tau)
    if R == 1:
        cand = [o for o in ops if o not in sel and o not in discarded and op_cost(tr, o) == 1
                and (creator[o] is None or creator[o] in sel)]
        if cand:
            sel.add(min(cand, key=lambda o: op_key(tr, o)))
            R = 0
    return sel, B - R


@pytest.mark.parametrize("seed", range(60))
def test_heap_equals_naive_greedy(oracle_lib, seed):
    rng = np.random.default_rng(seed)
    uvals = [0.0, 0.5, 1.0, 1.0, 2.0, 3.5] if seed % 2 else None
    tr = random_forest(rng, int(rng.integers(1, 6)), 9, uvals)
    total = len(tr.unit_Uadd) + int(tr.nodes["cost"].sum())
    for B in sorted({0, 1, 2, total // 3, total // 2, total - 1, total, total + 3}):
        if B < 0:
            continue
        add, split, used = heap_alloc(tr, B)
        ref, ref_used = naive_greedy(tr, B)
        assert sel_set(tr, add, split) == ref
        assert used == ref_used


@pytest.mark.parametrize("seed", range(80))
def test_kappa_threshold_equals_heap(oracle_lib, seed):
    rng = np.random.default_rng(1000 + seed)
    uvals = [0.0, 0.0, 1.0, 1.0, 2.0] if seed % 3 == 0 else ([0.0, 1.0, 3.0, 7.0] if seed % 3 == 1 else None)
    tr = random_forest(rng, int(rng.integers(1, 7)), 10, uvals, ext_p=0.5)
    total = len(tr.unit_Uadd) + int(tr.nodes["cost"].sum())
    for B in range(0, total + 2):
        add, split, used = heap_alloc(tr, B)
        sel, u2 = kappa_threshold_alloc(tr, B)
        assert sel_set(tr, add, split) == sel, (B, total)
        assert used == u2


def frontier_states(tr, v):
    """(cost, value) of every valid frontier of v's subtree with v covered."""
    nd = tr.nodes
    out = [(0, 0.0)]
    if nd["nchild"][v]:
        c0, nc = nd["child0"][v], nd["nchild"][v]
        cs = nd["cost"][v]
        gain = nd["U"][v] * cs
        for combo in itertools.product(*[frontier_states(tr, c) for c in range(c0, c0 + nc)]):
            out.append((cs + sum(x[0] for x in combo), gain + sum(x[1] for x in combo)))
    return out


def exhaustive_optimum(tr, B):
    best = {0: 0.0}
    for u, root in enumerate(tr.unit_root):
        opts = [(0, 0.0)] + [(1 + c, tr.unit_Uadd[u] + v) for c, v in frontier_states(tr, root)]
        nb = {}
        for used, val in best.items():
            for c, v in opts:
                if used + c <= B:
                    nb[used + c] = max(nb.get(used + c, -1.0), val + v)
        best = nb
    return max(best.values())


def greedy_value(tr, add, split):
    return float((tr.unit_Uadd * add).sum() + (tr.nodes["U"] * tr.nodes["cost"] * split).sum())


@pytest.mark.parametrize("seed", range(25))
def test_greedy_never_beats_exhaustive_optimum(oracle_lib, seed):
    rng = np.random.default_rng(500 + seed)
    tr = random_forest(rng, int(rng.integers(1, 4)), 6)
    total = len(tr.unit_Uadd) + int(tr.nodes["cost"].sum())
    for B in range(total + 1):
        add, split, _ = heap_alloc(tr, B)
        assert greedy_value(tr, add, split) <= exhaustive_optimum(tr, B) + 1e-12


@pytest.mark.parametrize("seed", range(25))
def test_greedy_is_optimal_for_unit_costs_and_monotone_gains(oracle_lib, seed):
    # with cost 1 everywhere and U non-increasing along every path, the top-B
    # ops form a prerequisite-closed set, so greedy reaches the optimum.
    rng = np.random.default_rng(800 + seed)
    tr = random_forest(rng, int(rng.integers(1, 4)), 6, ext_p=0.0)
    nd = tr.nodes
    for u, root in enumerate(tr.unit_root):
        nd["U"][root] = min(nd["U"][root], tr.unit_Uadd[u])
    for v in range(len(nd["a"])):
        if nd["nchild"][v]:
            for c in range(nd["child0"][v], nd["child0"][v] + nd["nchild"][v]):
                nd["U"][c] = min(nd["U"][c], nd["U"][v])
    total = len(tr.unit_Uadd) + int(nd["cost"].sum())
    for B in range(total + 1):
        add, split, _ = heap_alloc(tr, B)
        assert greedy_value(tr, add, split) == pytest.approx(exhaustive_optimum(tr, B), abs=1e-12)


def test_unaffordable_pop_is_discarded_and_cost_one_takes_last_unit(oracle_lib):
    # one unit [0,3) whose root splits by extraction (cost 2) with a high U, and a
    # second unit with a cheap binary split: with B = 2 the Add of unit 0 is
    # taken, its cost-2 split is discarded and unit 1's Add takes the last unit.
    keys = O._NODE_I32 + O._NODE_F64
    rows = [
        dict(lg=0, slot=0, a=0, b=3, parent=-1, child0=1, nchild=3, form=1, cost=2, U=10.0),
        dict(lg=0, slot=0, a=0, b=1, parent=0, child0=-1, nchild=0, form=-1, cost=0, U=0.0),
        dict(lg=0, slot=0, a=1, b=2, parent=0, child0=-1, nchild=0, form=-1, cost=0, U=0.0),
        dict(lg=0, slot=0, a=2, b=3, parent=0, child0=-1, nchild=0, form=-1, cost=0, U=0.0),
        dict(lg=0, slot=1, a=3, b=5, parent=-1, child0=5, nchild=2, form=0, cost=1, U=0.1),
        dict(lg=0, slot=1, a=3, b=4, parent=4, child0=-1, nchild=0, form=-1, cost=0, U=0.0),
        dict(lg=0, slot=1, a=4, b=5, parent=4, child0=-1, nchild=0, form=-1, cost=0, U=0.0),
    ]
    nodes = {k: np.asarray([r.get(k, 0) for r in rows],
                           dtype=np.int32 if k in O._NODE_I32 else np.float64) for k in keys}
    tr = O.Trees(nodes, np.array([5.0, 1.0]), np.array([0, 4], dtype=np.int64), 2)
    add, split, used = heap_alloc(tr, 2)
    assert list(add) == [1, 1] and split.sum() == 0 and used == 2
    add, split, used = heap_alloc(tr, 3)
    assert list(add) == [1, 0] and split[0] == 1 and used == 3
