"""The oracle's tree build split over worker processes (test infrastructure).

The prototype trees of different slots are independent (App. A.3: one tree
per layer-KV-head-slot unit), so the oracle can build the forest of a long
context slot range by slot range in separate processes and merge the
results; the heap allocation and the gather then run once on the merged
forest.  For one (l, g) the merged forest is exactly what one call over all
slots returns: units in ascending slot order, each unit's nodes contiguous.

Workers are started with the spawn method (never forked from a process that
has used the GPU) and import only numpy and the oracle.  Inputs travel as
.npy files that the workers map read-only.
"""
from __future__ import annotations

import multiprocessing as mp
import os
import tempfile

import numpy as np

import oracle as O


def _chunk(args):
    folder, kw, k0, k1 = args
    ld = lambda n: np.load(os.path.join(folder, n + ".npy"), mmap_mode="r")
    p = O.make_params(**kw)
    slots = np.asarray(ld("slots"))[k0:k1 + 1]
    tr = O.build_trees(p, ld("K"), ld("V"), ld("Q"), ld("kappa"), slots, ld("m"), ld("Z"), ld("rtok"))
    return k0, tr.nodes, tr.unit_Uadd, tr.unit_root


def build_trees_pooled(kw: dict, K, V, Q, kappa, slot_starts, m, Z, rtok, workers: int = 0) -> O.Trees:
    """O.build_trees for one layer and one KV head (L = G = 1), over slot
    chunks in spawned worker processes; kw are O.make_params' arguments."""
    assert kw["L"] == 1 and kw["G"] == 1
    J = len(slot_starts) - 1
    workers = workers or max(1, min(32, os.cpu_count() or 1))
    n_chunks = min(J, 4 * workers)
    bounds = np.linspace(0, J, n_chunks + 1).astype(int)
    with tempfile.TemporaryDirectory() as folder:
        for name, a in (("K", K), ("V", V), ("Q", Q), ("kappa", kappa), ("m", m), ("Z", Z),
                        ("rtok", rtok), ("slots", np.asarray(slot_starts, np.int32))):
            np.save(os.path.join(folder, name + ".npy"), np.ascontiguousarray(a, dtype=a.dtype))
        jobs = [(folder, kw, int(bounds[i]), int(bounds[i + 1])) for i in range(n_chunks)
                if bounds[i + 1] > bounds[i]]
        with mp.get_context("spawn").Pool(workers) as pool:
            parts = sorted(pool.map(_chunk, jobs), key=lambda r: r[0])
    nodes = {k: [] for k in parts[0][1]}
    uadd, uroot = [], []
    base = 0
    for k0, nd, ua, ur in parts:
        n = len(nd["a"])
        for k, v in nd.items():
            v = v.copy()
            if k in ("child0", "parent"):
                v = np.where(v >= 0, v + base, v)
            elif k == "slot":
                v = v + k0
            nodes[k].append(v)
        uadd.append(ua)
        uroot.append(ur + base)
        base += n
    return O.Trees({k: np.concatenate(v) for k, v in nodes.items()}, np.concatenate(uadd),
                   np.concatenate(uroot), J)


def run_pooled(K, V, Q, budgets, rope_base, slot_starts=None, **overrides):
    """The oracle pass of O.run for one layer and one KV head at several
    budgets, with the tree build pooled.  The trees do not depend on the
    budget (only the recent window does, and it is the same for every budget
    here), so segmentation, statistics and trees are computed once; each
    budget gets its own allocation and gather.  Without slot_starts the
    segmentation runs with the dispersion in the paper's prefix form (App.
    B.3 Eq. app_prefix_dispersion, pinned equal to the definition); with them
    the curvature is still computed (the refinement rule reads it)."""
    K64, V64, Q64 = (np.asarray(t.double().numpy() if hasattr(t, "double") else t, np.float64)
                     for t in (K, V, Q))
    L, G, T, d = K64.shape
    Hq, W = Q64.shape[1], Q64.shape[2]
    kw = dict(L=L, G=G, Hq=Hq, T=T, d=d, W=W, rope_base=rope_base, disp_mode=1, **overrides)
    p = O.make_params(**kw)
    r_eff, _ = O.budget(p, budgets[0])
    p.recent = r_eff
    kw["recent"] = r_eff
    if slot_starts is None:
        seg = O.segment(p, V64)
    else:
        kap, _ = O.curvature(p, V64)
        seg = dict(kappa=kap, b=None, slot_starts=np.asarray(slot_starts, np.int32) + p.ctx_start,
                   dp_best=None, dp_second=None)
    m, Z, ZC = O.row_stats(p, Q64, K64)
    rtok = O.token_values(p, Q64, K64, m, Z)
    tr = build_trees_pooled(kw, K64, V64, Q64, seg["kappa"], seg["slot_starts"], m, Z, rtok)
    out = []
    for B in budgets:
        pb = O.make_params(**kw)
        r_b, B_free = O.budget(pb, B)
        assert r_b == r_eff, "the budgets must share the recent window"
        pb.recent = r_eff
        add_sel, split_sel, used = O.allocate(pb, B_free, tr)
        cap = B + L * G * (T - (pb.ctx_end - pb.ctx_start)) + 16
        cache = O.gather(pb, K64, V64, rtok, tr, add_sel, split_sel, cap)
        out.append(dict(params=pb, r_eff=r_eff, B_free=B_free, seg=seg, m=m, Z=Z, ZC=ZC, rtok=rtok,
                        trees=tr, add_sel=add_sel, split_sel=split_sel, used=used, cache=cache, floor=None))
    return out
