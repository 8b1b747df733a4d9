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

from paper_2608_07001_gb300 import synth
from tests import parity as P
from tests.oracle_pool import run_pooled

pytestmark = pytest.mark.gpu

L_S, G_S = 13, 5          # the sliced (layer, KV head) of the 32 x 8 workload
RATIO = 32


def test_full_context_slice_matches_the_oracle():
    import __graft_entry__ as g
    g.build()
    w = synth.WORKLOADS["llama128k"]
    x = synth.make_inputs(w, layers=[L_S], heads=[G_S])
    L, G, T, d = x.K.shape
    assert (L, G, T, d) == (1, 1, 131072, 128) and x.K.dtype == torch.bfloat16
    B = (L * G * T) // RATIO
    t0 = time.time()
    o = run_pooled(x.K, x.V, x.Q, [B], w.rope_base)[0]
    t1 = time.time()
    gr = P.run_gpu(x.K, x.V, x.Q, B, w.rope_base)
    rep = P.compare(gr, o, torch.bfloat16)
    print(f"full-context slice: oracle {t1 - t0:.0f} s, {len(o['seg']['slot_starts']) - 1} slots, "
          f"{len(o['trees'].nodes['a'])} oracle nodes, {gr['E']} entries", rep)
    assert gr["E"] == B
