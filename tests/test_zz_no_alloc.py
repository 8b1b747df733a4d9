"""The allocation-free row-statistics entry point against the context path.

Callers that cannot call cudaMalloc (an engine that owns the device's memory
pool, or a latency-critical loop that cannot take an allocation's device
synchronisation) use gracekv_row_stats_noalloc, whose scratch is a fixed
array inside the library.  Its outputs must match the row statistics the
normal path (gracekv_build_trees) computes, on two calls in a row that share
that array.  This file is collected last on purpose.
"""
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


def reference_rows(x, B, base):
    from paper_2608_07001_gb300 import gracekv as gk
    L, G, T, d = x.K.shape
    p = gk.make_params(L, G, x.Q.shape[1], T, d, x.Q.shape[2], dtype=x.K.dtype, budget=B,
                       rope_base=base)
    ctx = gk.Context(p)
    K, V, Q = x.K.cuda(), x.V.cuda(), x.Q.cuda()
    slots = torch.empty(T + 2, dtype=torch.int32, device="cuda")
    ctx.gracekv_segment(V, slots)
    ctx.gracekv_build_trees(K, V, Q)
    ex = ctx.gracekv_export()
    c_lo, c_hi = 0, T - ctx.recent
    return K, Q, (ex["row_m"], ex["row_Z"], ex["row_ZC"]), c_lo, c_hi


@pytest.mark.parametrize("name,kw", [("pr1", dict(T=1000)),
                                     ("small", dict(layers=[0, 1], heads=[0, 3], T=1500))])
def test_noalloc_row_stats_match_the_context_path_twice(name, kw):
    from paper_2608_07001_gb300 import gracekv as gk
    w = synth.WORKLOADS[name]
    x = synth.make_inputs(w, **kw)
    L, G, T, d = x.K.shape
    K, Q, ref, c_lo, c_hi = reference_rows(x, (L * G * T) // 8, w.rope_base)
    shape = (L, x.Q.shape[1], x.Q.shape[2])
    for call in range(2):
        outs = [torch.full(shape, float("nan"), device="cuda") for _ in range(3)]
        gk.gracekv_row_stats_noalloc(K, Q, c_lo, c_hi, *outs)
        torch.cuda.synchronize()
        for o, r, tol in zip(outs, ref, (2e-6, 2e-5, 2e-5)):
            o = o.cpu().numpy().reshape(-1)
            err = np.abs(o - r) / np.maximum(np.abs(r), 1.0 if tol == 2e-6 else 1e-30)
            assert np.isfinite(o).all()
            assert err.max() <= tol, (call, err.max())


def test_noalloc_rejects_too_many_rows():
    from paper_2608_07001_gb300 import gracekv as gk
    K = torch.zeros(1, 1, 64, 64, device="cuda")
    Q = torch.zeros(1, 1, 400000, 64, device="cuda")
    o = [torch.empty(400000, device="cuda") for _ in range(3)]
    with pytest.raises(gk.GraceKVError) as e:
        gk.gracekv_row_stats_noalloc(K, Q, 0, 32, *o)
    assert e.value.status == gk.GKV_ECAPACITY
