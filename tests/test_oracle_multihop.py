"""Pins of the oracle's multi-hop relevance (App. A.4, Eqs.
app_global_seed_score, app_hop_propagation, app_diffused_relevance and
app_bottom_up_value)."""
import math

import numpy as np
import pytest
import torch

import oracle as O


def setup(seed=0, L=4, G=2, gq=2, T=96, d=8, recent=8, cs=0):
    rng = np.random.default_rng(seed)
    K = rng.normal(size=(L, G, T, d))
    p = O.make_params(L, G, G * gq, T, d, 2, 0.0, ctx_start=cs, recent=recent, lambda_graph=0.3)
    gl = O.graph_layers(p)
    Qg = rng.normal(size=(len(gl), G * gq, T, d))
    Nc = T - recent - cs
    shat = rng.random((L * G, Nc)) ** 8
    shat /= shat.sum(1, keepdims=True)
    return p, K, Qg, shat, gl


def test_graph_layers_are_at_half_and_three_quarter_depth(oracle_lib):
    p = O.make_params(32, 8, 32, 64, 8, 2, 0.0, recent=8)
    np.testing.assert_array_equal(O.graph_layers(p), [16, 24])


def test_first_hop_seeds_follow_the_global_seed_score(oracle_lib):
    # S-hat = normalised mean over (l, g); seeds in descending order until the
    # running mass reaches 0.9 (the seed that reaches it included)
    p, K, Qg, shat, gl = setup()
    Nc = shat.shape[1]
    shat[:] = 1e-4
    shat[:, [10, 40, 70]] = [0.5, 0.3, 0.15]      # masses 0.5, 0.8, 0.95 after normalisation
    shat /= shat.sum(1, keepdims=True)
    dh, sd, sw = O.multihop(p, shat, Qg, K)
    S = shat.mean(0) / shat.mean(0).sum()
    order = [10, 40, 70]
    assert list(sd[0][:3]) == order and sd[0][3] == -1
    np.testing.assert_allclose(sw[0][:3], S[order] / S[order].sum(), rtol=1e-12)


def test_uniform_attention_closed_form(oracle_lib):
    # zero queries: every seed attends uniformly to [0, u]; one hop: d_t is
    # sum over graph layers and heads of sum_u w_u / (u + 1) for t <= u,
    # zero at the seeds, then normalised
    p, K, Qg, shat, gl = setup(1)
    p.r_hop = 1
    Qg[:] = 0.0
    dh, sd, sw = O.multihop(p, shat, Qg, K)
    Nc = shat.shape[1]
    seeds = sd[0][sd[0] >= 0]
    w = sw[0][:len(seeds)]
    ref = np.zeros(Nc)
    for u, wu in zip(seeds, w):
        ref[:u + 1] += len(gl) * p.Hq * wu / (u + 1)
    ref[seeds] = 0.0
    np.testing.assert_allclose(dh, ref / (ref.sum() + p.eps), rtol=1e-12, atol=1e-15)


def test_one_seed_row_is_torch_softmax_and_causal(oracle_lib):
    # a single seed, one graph layer, one head: d-hat is the seed's softmax row
    # over [0, u] (torch), zeroed at the seed, restricted to C and normalised
    rng = np.random.default_rng(2)
    L, G, T, d = 2, 1, 40, 8
    K = rng.normal(size=(L, G, T, d))
    p = O.make_params(L, G, 1, T, d, 2, 0.0, recent=4, lambda_graph=0.3, m_seed=1, r_hop=1)
    Qg = rng.normal(size=(1, 1, T, d))
    Nc = T - 4
    shat = np.full((L * G, Nc), 1e-3)
    shat[:, 20] = 1.0
    shat /= shat.sum(1, keepdims=True)
    dh, sd, sw = O.multihop(p, shat, Qg, K, graph_l=[1])
    assert sd[0][0] == 20
    x = torch.as_tensor(K[1, 0, :21] @ Qg[0, 0, 20] / math.sqrt(d))
    pi = torch.softmax(x, 0).numpy()
    ref = np.zeros(Nc)
    ref[:21] = pi
    ref[20] = 0.0
    np.testing.assert_allclose(dh, ref / (ref.sum() + p.eps), rtol=1e-12, atol=1e-15)
    assert np.all(dh[21:] == 0)                     # the seed sees only its past


def test_hops_zero_their_seeds_and_mix_into_the_token_values(oracle_lib):
    p, K, Qg, shat, gl = setup(3)
    dh, sd, sw = O.multihop(p, shat, Qg, K)
    # every hop's score is zeroed at its own and earlier seeds: the first hop's
    # seeds end at zero; the second hop's keep the mass the first hop found
    first = sd[0][sd[0] >= 0]
    assert np.all(dh[first] == 0)
    assert np.all(dh[sd[1][sd[1] >= 0]] > 0)
    assert dh.sum() == pytest.approx(1.0, abs=1e-5)
    assert len(sd[1][sd[1] >= 0]) > 0 and not set(sd[1][sd[1] >= 0]) & set(sd[0][sd[0] >= 0])
    # the whole pass mixes R = (1 - lambda) s-hat + lambda d-hat
    rng = np.random.default_rng(4)
    L, G, T, d = p.L, p.G, p.T, p.d
    V = rng.normal(size=(L, G, T, d))
    Q = rng.normal(size=(L, p.Hq, 2, d))
    res = O.run(K, V, Q, 120, 0.0, recent=8, lambda_graph=0.3, Qg=Qg)
    mh = res["multihop"]
    np.testing.assert_allclose(res["rtok"], 0.7 * mh["shat"] + 0.3 * mh["dhat"][None, None, :], rtol=1e-13)
    res0 = O.run(K, V, Q, 120, 0.0, recent=8)
    np.testing.assert_allclose(mh["shat"], res0["rtok"], rtol=1e-13)


def test_decay_weights_only_the_later_hops(oracle_lib):
    # d = d1 + rho d2: rho = 0 gives the one-hop result, and d-hat at rho = 1/2
    # lies on the segment from d-hat(0) to d-hat(1), strictly past its middle
    # when the second hop carries mass (the weights are (A + eps) / 2 and
    # (A + B + eps) / 2 over A + B / 2 + eps, A and B the hops' sums)
    p, K, Qg, shat, gl = setup(5)
    p.r_hop = 1
    d_one, _, _ = O.multihop(p, shat, Qg, K)
    p.r_hop = 2
    res = {}
    for rho in (0.0, 0.5, 1.0):
        p.rho_hop = rho
        res[rho], _, _ = O.multihop(p, shat, Qg, K)
    np.testing.assert_allclose(res[0.0], d_one, rtol=1e-12, atol=1e-15)
    a, diff = res[0.0], res[1.0] - res[0.0]
    theta = np.dot(res[0.5] - a, diff) / np.dot(diff, diff)
    np.testing.assert_allclose(res[0.5], a + theta * diff, rtol=1e-9, atol=1e-14)
    assert 0.5 < theta < 1.0


def test_second_hop_seeds_follow_the_first_hops_propagation(oracle_lib):
    # hop 2 chooses its seeds by the same rule from hop 1's propagation score
    # normalised over C (the one-hop d-hat up to its eps), and weights them by
    # that score over the seed set
    p, K, Qg, shat, gl = setup(6)
    p.r_hop = 1
    d1, sd1, _ = O.multihop(p, shat, Qg, K)
    p.r_hop = 2
    dh, sd, sw = O.multihop(p, shat, Qg, K)
    np.testing.assert_array_equal(sd[0], sd1[0])
    score = d1 / d1.sum()
    order = np.lexsort((np.arange(len(score)), -score))
    cum, want = 0.0, []
    while len(want) < p.m_seed and cum < p.eta_seed:
        want.append(int(order[len(want)]))
        cum += score[want[-1]]
    n = len(want)
    assert 1 < n < p.m_seed
    assert list(sd[1][:n]) == want and np.all(sd[1][n:] == -1)
    np.testing.assert_allclose(sw[1][:n], score[want] / score[want].sum(), rtol=1e-12)
