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
