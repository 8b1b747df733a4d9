"""Pins of the oracle's layer-KV-head sensitivity (App. A.4, Eqs.
app_head_sensitivity_raw and app_head_sensitivity)."""
import numpy as np
import pytest

import oracle as O


def test_sensitivity_matches_numpy_linear_algebra(oracle_lib):
    # the static norm is numpy's Frobenius norm of the group's column blocks,
    # the input term numpy's matrix-vector products and 2-norms
    rng = np.random.default_rng(0)
    L, G, gq, d, D, U = 3, 2, 2, 8, 20, 5
    Hq = G * gq
    W = rng.normal(size=(L, D, Hq * d))
    o = rng.normal(size=(L, Hq, U, d))
    om = O.head_sensitivity(W, o, G, eps=0.0)
    raw = np.zeros((L, G))
    for l in range(L):
        for g in range(G):
            cols = slice(g * gq * d, (g + 1) * gq * d)
            st = np.linalg.norm(W[l][:, cols], "fro")
            x = o[l, g * gq:(g + 1) * gq].transpose(1, 0, 2).reshape(U, gq * d)   # [U, gq d]
            inp = np.linalg.norm(x @ W[l][:, cols].T, axis=1).mean()
            raw[l, g] = np.sqrt(st * inp)
    np.testing.assert_allclose(om, raw / raw.mean(), rtol=1e-12)


def test_sensitivity_closed_forms_and_invariances(oracle_lib):
    L, G, d, U = 2, 2, 4, 3
    rng = np.random.default_rng(1)
    o = rng.normal(size=(L, G, U, d))
    # W_O^{l,h} = s_{l,h} [I_d; 0]: static = s sqrt(d), input = s mean ||o||
    s = np.array([[1.0, 2.0], [3.0, 0.5]])
    D = 6
    W = np.zeros((L, D, G * d))
    for l in range(L):
        for h in range(G):
            W[l, :d, h * d:(h + 1) * d] = s[l, h] * np.eye(d)
    om = O.head_sensitivity(W, o, G, eps=0.0)
    raw = np.sqrt(s * np.sqrt(d) * s * np.linalg.norm(o, axis=-1).mean(-1))
    np.testing.assert_allclose(om, raw / raw.mean(), rtol=1e-12)
    assert om.mean() == pytest.approx(1.0, abs=1e-12)
    # a global scale of W_O or of o cancels in the normalisation
    np.testing.assert_allclose(O.head_sensitivity(7.0 * W, o, G, eps=0.0), om, rtol=1e-12)
    np.testing.assert_allclose(O.head_sensitivity(W, 0.1 * o, G, eps=0.0), om, rtol=1e-12)
    # heads of one group add inside the norm: opposite outputs cancel
    W2 = np.zeros((1, d, 2 * d))
    W2[0, :, :d] = np.eye(d)
    W2[0, :, d:] = np.eye(d)
    o2 = rng.normal(size=(1, 2, U, d))
    o2[0, 1] = -o2[0, 0]
    assert O.head_sensitivity(W2, o2, 1, eps=1e-6)[0, 0] == pytest.approx(0.0, abs=1e-9)
