"""Pins of the oracle's row statistics, token values, prototypes and trees."""
import math

import numpy as np
import pytest
from scipy.special import logsumexp, softmax

import oracle as O


def rand_inputs(seed, L=1, G=2, gq=1, T=96, d=8, W=4, scale=1.0):
    rng = np.random.default_rng(seed)
    K = rng.normal(size=(L, G, T, d)) * scale
    V = rng.normal(size=(L, G, T, d))
    Q = rng.normal(size=(L, G * gq, W, d))
    return K, V, Q


# --- row statistics / token values: App. A.4 ---------------------------------------

def test_row_stats_match_logsumexp(oracle_lib):
    K, V, Q = rand_inputs(0, G=2, gq=2, T=80, W=3)
    p = O.make_params(1, 2, 4, 80, 8, 3, 0.0, ctx_start=5, ctx_end=70, recent=6)
    m, Z, ZC = O.row_stats(p, Q, K)
    for h in range(4):
        for u in range(3):
            x = K[0, h // 2] @ Q[0, h, u] / math.sqrt(8)
            assert m[0, h, u] == pytest.approx(x.max(), abs=1e-13)
            assert Z[0, h, u] == pytest.approx(math.exp(logsumexp(x) - x.max()), rel=1e-13)
            assert ZC[0, h, u] == pytest.approx(math.exp(logsumexp(x[5:64]) - x.max()), rel=1e-13)


def test_token_values_single_probe_is_renormalised_softmax(oracle_lib):
    # one probe, one query head per KV head: shat = softmax over [0,T) restricted
    # to C and renormalised (plus eps), Eq. (app_direct_relevance)
    K, V, Q = rand_inputs(1, G=2, gq=1, T=64, W=1)
    p = O.make_params(1, 2, 2, 64, 8, 1, 0.0, recent=8)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    for g in range(2):
        s = softmax(K[0, g] @ Q[0, g, 0] / math.sqrt(8))
        np.testing.assert_allclose(r[0, g], s[:56] / (s[:56].sum() + 1e-6), rtol=1e-12)


def test_token_values_gqa_sum_and_normalisation(oracle_lib):
    K, V, Q = rand_inputs(2, G=2, gq=2, T=50, W=3)
    p = O.make_params(1, 2, 4, 50, 8, 3, 0.0, recent=4)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    for g in range(2):
        s = sum(softmax(K[0, g] @ Q[0, h, u] / math.sqrt(8))
                for h in (2 * g, 2 * g + 1) for u in range(3))[:46]
        np.testing.assert_allclose(r[0, g], s / (s.sum() + 1e-6), rtol=1e-12)
        tot = s.sum()
        assert r[0, g].sum() == pytest.approx(tot / (tot + 1e-6), rel=1e-13)


# --- prototypes: App. A.3 Eqs. (app_rope_prototype) .. (app_effective_multiplicity) ----

def rope_complex(x, t, base):
    """RoPE on half-split pairs as a complex rotation z_i -> z_i exp(i t theta_i)."""
    d = x.shape[-1]
    h = d // 2
    th = base ** (-2.0 * np.arange(h) / d)
    z = (x[..., :h] + 1j * x[..., h:]) * np.exp(1j * np.asarray(t)[..., None] * th)
    return np.concatenate([z.real, z.imag], -1)


@pytest.mark.parametrize("a,b,pos", [(0, 4, 2), (1, 5, 2), (2, 6, 4), (0, 3, 1), (7, 8, 7),
                                     (10, 21, 15), (11, 21, 16)])
def test_representative_position_half_even(oracle_lib, a, b, pos):
    K, V, Q = rand_inputs(3, G=1, T=32)
    p = O.make_params(1, 1, 1, 32, 8, 4, 1e4, recent=4)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    assert O.eval_interval(p, K, V, Q, m, Z, r, 0, 0, a, b)["pos"] == pos


def test_root_prototype_closed_form_complex(oracle_lib):
    base = 500000.0
    T, d = 64, 16
    K, V, Q = rand_inputs(4, G=1, T=T, d=d, scale=2.0)
    p = O.make_params(1, 1, 1, T, d, 4, base, recent=8)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    a, b = 11, 47
    res = O.eval_interval(p, K, V, Q, m, Z, r, 0, 0, a, b)
    t = np.arange(a, b)
    kc = rope_complex(K[0, 0, a:b], -t, base)
    mu = kc.mean(0)
    pos = int(np.round((a + b - 1) / 2))          # numpy rounds half to even
    np.testing.assert_allclose(res["ktil"], rope_complex(mu, pos, base), rtol=0, atol=1e-12)
    coh = np.linalg.norm(mu) / (np.linalg.norm(kc, axis=1).mean() + 1e-6)
    assert res["logm"] == pytest.approx(math.log(min(max((b - a) * coh ** 2, 1.0), b - a)), abs=1e-12)
    w = r[0, 0, a:b] + 0.1 * r[0, 0, a:b].mean()
    np.testing.assert_allclose(res["vtil"], (w[:, None] * V[0, 0, a:b]).sum(0) / (w.sum() + 1e-6),
                               atol=1e-12)


def test_coherent_rotated_keys_have_full_multiplicity(oracle_lib):
    # k_t = RoPE(c, t): the inverse rotation maps every key to c, so
    # ktil = RoPE(c, p), coh = |c| / (|c| + eps), m_eff ~= n.
    base, T, d = 1e4, 40, 8
    c = np.random.default_rng(5).normal(size=d)
    K = rope_complex(np.tile(c, (T, 1)), np.arange(T), base).reshape(1, 1, T, d)
    V = np.random.default_rng(6).normal(size=(1, 1, T, d))
    Q = np.random.default_rng(7).normal(size=(1, 1, 2, d))
    p = O.make_params(1, 1, 1, T, d, 2, base, recent=4)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    res = O.eval_interval(p, K, V, Q, m, Z, r, 0, 0, 3, 19)
    assert res["pos"] == 10                      # mean 10.5, half to even
    np.testing.assert_allclose(res["ktil"], rope_complex(c, 10, base), atol=1e-12)
    n = 16
    coh = np.linalg.norm(c) / (np.linalg.norm(c) + 1e-6)
    assert res["logm"] == pytest.approx(math.log(n * coh ** 2), abs=1e-12)


def test_identical_entries_without_rope_have_no_distortion(oracle_lib):
    # App. A.3 text after Eq. (app_decode_logit): identical, coherent keys and
    # identical values recover the partition mass; D vanishes up to eps terms.
    T, d = 48, 8
    rng = np.random.default_rng(8)
    K = rng.normal(size=(1, 1, T, d))
    V = rng.normal(size=(1, 1, T, d))
    K[0, 0, 10:30] = K[0, 0, 10]
    V[0, 0, 10:30] = V[0, 0, 10]
    Q = rng.normal(size=(1, 1, 4, d))
    p = O.make_params(1, 1, 1, T, d, 4, 0.0, recent=4)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    res = O.eval_interval(p, K, V, Q, m, Z, r, 0, 0, 10, 30)
    assert res["D"] < 1e-9
    assert res["logm"] == pytest.approx(math.log(20), abs=1e-5)
    assert res["Ddrop"] > 0


def test_singleton_interval_is_the_token(oracle_lib):
    K, V, Q = rand_inputs(9, G=1, T=32)
    p = O.make_params(1, 1, 1, 32, 8, 4, 1e4, recent=4)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    res = O.eval_interval(p, K, V, Q, m, Z, r, 0, 0, 13, 14)
    assert res["D"] == 0.0 and res["pos"] == 13 and res["logm"] == 0.0
    assert np.array_equal(res["ktil"], K[0, 0, 13]) and np.array_equal(res["vtil"], V[0, 0, 13])


def test_distortion_drop_is_mean_attention_mass(oracle_lib):
    # Ddrop(I) = Mean_q Z_q(I) / Z_q  (Eq. app_node_and_drop_distortion):
    # probe u of KV head g uses query head H(g)[u mod |H(g)|].
    K, V, Q = rand_inputs(10, G=2, gq=2, T=60, W=3)
    p = O.make_params(1, 2, 4, 60, 8, 3, 0.0, recent=4)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    g, a, b = 1, 7, 33
    res = O.eval_interval(p, K, V, Q, m, Z, r, 0, g, a, b)
    exp = np.mean([softmax(K[0, g] @ Q[0, 2 * g + (u % 2), u] / math.sqrt(8))[a:b].sum()
                   for u in range(3)])
    assert res["Ddrop"] == pytest.approx(exp, rel=1e-12)


# --- trees: App. A.3 refinement, App. A.4 conservation, App. C.6 telescoping ------------

@pytest.fixture(scope="module")
def small_run(oracle_lib):
    rng = np.random.default_rng(11)
    L, G, gq, T, d, W = 1, 2, 2, 160, 8, 4
    K = rng.normal(size=(L, G, T, d)) * 1.5
    V = rng.normal(size=(L, G, T, d))
    Q = rng.normal(size=(L, G * gq, W, d))
    res = O.run(K, V, Q, (L * G * T) // 4, 1e4, n_min=8, n_max=40, n0=20, recent=8,
                windows=(2, 4, 8))
    return K, V, Q, res


def test_tree_structure_and_value_conservation(small_run):
    K, V, Q, res = small_run
    nd = res["trees"].nodes
    leaves = 0
    for v in range(len(nd["a"])):
        a, b = nd["a"][v], nd["b"][v]
        if b - a == 1:
            assert nd["nchild"][v] == 0
            leaves += 1
            continue
        c0, nc = nd["child0"][v], nd["nchild"][v]
        assert nc in (2, 3) and nd["cost"][v] == nc - 1
        ch = range(c0, c0 + nc)
        assert nd["a"][c0] == a and nd["b"][c0 + nc - 1] == b
        assert all(nd["b"][c] == nd["a"][c + 1] for c in range(c0, c0 + nc - 1))
        assert all(nd["parent"][c] == v for c in ch)
        # Eq. (app_value_conservation)
        assert sum(nd["R"][c] for c in ch) == pytest.approx(nd["R"][v], rel=1e-12)
        assert nd["U"][v] >= 0.0
        if nc == 3:
            assert nd["b"][c0 + 1] - nd["a"][c0 + 1] == 1   # extraction isolates one token
    assert leaves == res["params"].L * res["params"].G * (res["seg"]["slot_starts"][-1]
                                                          - res["seg"]["slot_starts"][0])


def test_telescoping_cost_identity(small_run):
    # App. C.6: 1 + sum over expanded nodes (|child| - 1) = n per tree.
    K, V, Q, res = small_run
    nd, tr = res["trees"].nodes, res["trees"]
    for u, root in enumerate(tr.unit_root):
        n = nd["b"][root] - nd["a"][root]
        stack, cost = [root], 1
        while stack:
            v = stack.pop()
            if nd["nchild"][v]:
                cost += nd["nchild"][v] - 1
                stack.extend(range(nd["child0"][v], nd["child0"][v] + nd["nchild"][v]))
        assert cost == n


def test_node_distortion_consistent_with_interval_evaluation(small_run):
    K, V, Q, res = small_run
    p, nd = res["params"], res["trees"].nodes
    rng = np.random.default_rng(0)
    for v in rng.choice(len(nd["a"]), size=25, replace=False):
        lg = nd["lg"][v]
        e = O.eval_interval(p, K, V, Q, res["m"], res["Z"], res["rtok"], lg // p.G, lg % p.G,
                            int(nd["a"][v]), int(nd["b"][v]))
        assert e["D"] == nd["D"][v]
