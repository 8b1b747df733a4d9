"""Full-context slice parity: one layer and one KV head of the llama128k
workload (131072 tokens, bf16, head dim 128, 4 query heads x 64 observation
queries) compressed 32x, through all four stages, against the oracle.

At this length the oracle's own segmentation (dispersion in the paper's
prefix form), row statistics and token values run directly; its tree build
runs slot range by slot range in spawned worker processes and is merged
(tests/oracle_pool.py), then the oracle's heap allocation and gather run on
the merged forest.  The comparison is the
same as at test sizes (tests/parity.py): bit-exact slots, trees, selection,
positions and intervals, single tokens bit-exact, prototypes within the bf16
tolerance, no near-tie exemption.
"""
import time

import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_07001_gb300 import synth
from tests import parity as P
from tests.oracle_pool import build_trees_pooled

pytestmark = pytest.mark.gpu

L_S, G_S = 13, 5          # the sliced (layer, KV head) of the 32 x 8 workload
RATIO = 32


def oracle_slice(K, V, Q, B, base):
    """The oracle pass of O.run for L = G = 1, with the tree build pooled."""
    L, G, T, d = K.shape
    Hq, W = Q.shape[1], Q.shape[2]
    # the dispersion in the paper's prefix form (App. B.3 Eq.
    # app_prefix_dispersion), pinned equal to the sample-variance definition
    kw = dict(L=L, G=G, Hq=Hq, T=T, d=d, W=W, rope_base=base, disp_mode=1)
    p = O.make_params(**kw)
    r_eff, B_free = O.budget(p, B)
    p.recent = r_eff
    kw["recent"] = r_eff
    K64, V64, Q64 = (t.double().numpy() for t in (K, V, Q))
    seg = O.segment(p, V64)
    m, Z, ZC = O.row_stats(p, Q64, K64)
    rtok = O.token_values(p, Q64, K64, m, Z)
    tr = build_trees_pooled(kw, K64, V64, Q64, seg["kappa"], seg["slot_starts"], m, Z, rtok)
    add_sel, split_sel, used = O.allocate(p, B_free, tr)
    cache = O.gather(p, K64, V64, rtok, tr, add_sel, split_sel, B + 16)
    return dict(params=p, r_eff=r_eff, B_free=B_free, seg=seg, m=m, Z=Z, ZC=ZC, rtok=rtok,
                trees=tr, add_sel=add_sel, split_sel=split_sel, used=used, cache=cache, floor=None)


def test_full_context_slice_matches_the_oracle():
    import __graft_entry__ as g
    g.build()
    w = synth.WORKLOADS["llama128k"]
    x = synth.make_inputs(w, layers=[L_S], heads=[G_S])
    L, G, T, d = x.K.shape
    assert (L, G, T, d) == (1, 1, 131072, 128) and x.K.dtype == torch.bfloat16
    B = (L * G * T) // RATIO
    t0 = time.time()
    o = oracle_slice(x.K, x.V, x.Q, B, w.rope_base)
    t1 = time.time()
    gr = P.run_gpu(x.K, x.V, x.Q, B, w.rope_base)
    rep = P.compare(gr, o, torch.bfloat16)
    print(f"full-context slice: oracle {t1 - t0:.0f} s, {len(o['seg']['slot_starts']) - 1} slots, "
          f"{len(o['trees'].nodes['a'])} oracle nodes, {gr['E']} entries", rep)
    assert gr["E"] == B
