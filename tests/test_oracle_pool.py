"""The pooled oracle tree build equals one call over all slots (CPU)."""
import numpy as np

import oracle as O
from tests.oracle_pool import build_trees_pooled


def test_pooled_forest_equals_one_call(oracle_lib):
    rng = np.random.default_rng(4)
    T, d, W, gq = 700, 16, 4, 2
    K = rng.normal(size=(1, 1, T, d))
    V = rng.normal(size=(1, 1, T, d))
    Q = rng.normal(size=(1, gq, W, d))
    kw = dict(L=1, G=1, Hq=gq, T=T, d=d, W=W, rope_base=1e4, recent=32)
    p = O.make_params(**kw)
    m, Z, _ = O.row_stats(p, Q, K)
    R = O.token_values(p, Q, K, m, Z)
    kappa = np.round(rng.random(T), 2)
    cuts = np.sort(rng.choice(np.arange(1, T - 32), 9, replace=False))
    slots = np.concatenate([[0], cuts, [T - 32]]).astype(np.int32)
    one = O.build_trees(p, K, V, Q, kappa, slots, m, Z, R)
    pooled = build_trees_pooled(kw, K, V, Q, kappa, slots, m, Z, R, workers=3)
    assert pooled.n_slots == one.n_slots
    np.testing.assert_array_equal(pooled.unit_root, one.unit_root)
    np.testing.assert_array_equal(pooled.unit_Uadd, one.unit_Uadd)
    assert set(pooled.nodes) == set(one.nodes)
    for k in one.nodes:
        np.testing.assert_array_equal(pooled.nodes[k], one.nodes[k], err_msg=k)
    a1 = O.allocate(p, 200, one)
    a2 = O.allocate(p, 200, pooled)
    for x, y in zip(a1, a2):
        np.testing.assert_array_equal(x, y)
