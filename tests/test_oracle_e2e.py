"""End-to-end pins of the oracle pipeline (App. A.5 packing, App. C.6)."""
import numpy as np
import pytest

import oracle as O


def inputs(seed, L=1, G=2, gq=2, T=150, d=8, W=4):
    rng = np.random.default_rng(seed)
    K = rng.normal(size=(L, G, T, d)) * 1.3
    V = rng.normal(size=(L, G, T, d))
    Q = rng.normal(size=(L, G * gq, W, d))
    return K, V, Q


SMALL = dict(n_min=8, n_max=32, n0=16, recent=8, windows=(2, 4, 8))


@pytest.mark.parametrize("ctx", [(0, None), (5, 140)])
def test_full_budget_recovers_fullkv_exactly(oracle_lib, ctx):
    # App. C.6 "FullKV recovery": x = 1 -> every tree expands to its leaves and
    # the cache equals the input entry by entry, positions 0..T-1, log m = 0.
    K, V, Q = inputs(0)
    L, G, T, d = K.shape
    cs, ce = ctx
    ce = T if ce is None else ce
    res = O.run(K, V, Q, L * G * (ce - cs), 1e4, ctx_start=cs, ctx_end=ce, **SMALL)
    c = res["cache"]
    assert res["used"] == res["B_free"]
    for lg in range(L * G):
        lo, hi = c["offsets"][lg], c["offsets"][lg + 1]
        assert hi - lo == T
        assert np.array_equal(c["pos"][lo:hi], np.arange(T))
        assert np.all(c["log_m"][lo:hi] == 0.0)
        assert np.array_equal(c["K"][lo:hi], K[lg // G, lg % G])
        assert np.array_equal(c["V"][lo:hi], V[lg // G, lg % G])


@pytest.mark.parametrize("x", [2, 4, 8])
def test_frontiers_partition_covered_slots_and_fill_budget(oracle_lib, x):
    K, V, Q = inputs(1)
    L, G, T, d = K.shape
    B = (L * G * T) // x
    res = O.run(K, V, Q, B, 1e4, **SMALL)
    c, p = res["cache"], res["params"]
    ss = res["seg"]["slot_starts"]
    r = res["r_eff"]
    E = len(c["pos"])
    assert E == L * G * r + res["used"] and E <= B
    # reading: the budget is used in full unless the endgame finds no cost-1 op
    assert res["used"] in (res["B_free"], res["B_free"] - 1)
    for lg in range(L * G):
        lo, hi = c["offsets"][lg], c["offsets"][lg + 1]
        a, b = c["src_lo"][lo:hi], c["src_hi"][lo:hi]
        assert np.all(a[1:] >= b[:-1])                 # non-overlapping, ascending
        assert np.all(c["pos"][lo:hi] >= a) and np.all(c["pos"][lo:hi] < b)
        # every covered slot is exactly partitioned by its frontier
        for j in range(len(ss) - 1):
            inside = (a >= ss[j]) & (b <= ss[j + 1])
            if inside.any():
                cov = np.concatenate([np.arange(s, e) for s, e in zip(a[inside], b[inside])])
                assert np.array_equal(cov, np.arange(ss[j], ss[j + 1]))
        # recent window kept verbatim at the end
        assert np.array_equal(c["pos"][hi - r:hi], np.arange(T - r, T))
        single = (b - a) == 1
        assert np.all(c["log_m"][lo:hi][single] == 0.0)
        assert np.array_equal(c["K"][lo:hi][single], K[lg // G, lg % G][a[single]])


def test_omega_scales_gains(oracle_lib):
    K, V, Q = inputs(2)
    L, G, T, d = K.shape
    base = O.run(K, V, Q, (L * G * T) // 4, 1e4, **SMALL)
    om = O.run(K, V, Q, (L * G * T) // 4, 1e4, omega=np.full(L * G, 2.0), **SMALL)
    np.testing.assert_allclose(om["trees"].nodes["U"], 2 * base["trees"].nodes["U"], rtol=1e-15)
    assert np.array_equal(om["split_sel"], base["split_sel"])
