"""Pins of the oracle's decoding attention, App. A.3 Eq. (app_decode_logit).

The logit of a packed entry is q . k / sqrt(d) + log m_eff; a token generated
after the compression is appended with multiplicity 1 (App. A.5, packing
paragraph).  The pins tie the oracle to things it does not compute itself:
torch's scaled-dot-product attention when every log m is 0, the identity
"one entry with log m = log n  ==  n identical entries" (the exact limiting
form the paper states after Eq. app_decode_logit), the oracle's own
compression of an interval of identical tokens, and invariances of softmax.
"""
import math

import numpy as np
import pytest
import torch

import oracle as O


def ragged(seed, L=2, G=2, gq=2, d=16, counts=None, app_cap=0, n_app=0, logm_scale=0.0):
    rng = np.random.default_rng(seed)
    if counts is None:
        counts = rng.integers(1, 40, size=L * G)
    counts = np.asarray(counts)
    off = np.concatenate([[0], np.cumsum(counts)]).astype(np.int64)
    E = int(off[-1])
    K = rng.normal(size=(E, d))
    V = rng.normal(size=(E, d))
    lm = logm_scale * rng.random(E)
    q = rng.normal(size=(L, G * gq, d)) * 2.0
    Ka = rng.normal(size=(L, G, max(app_cap, 1), d))
    Va = rng.normal(size=(L, G, max(app_cap, 1), d))
    return dict(q=q, K=K, V=V, log_m=lm, offsets=off, K_app=Ka, V_app=Va, n_app=n_app,
                L=L, G=G)


def sdpa(q, K, V, bias=None):
    """torch's attention in fp64 for one query row."""
    t = lambda x: torch.as_tensor(x, dtype=torch.float64)
    mask = None if bias is None else t(bias)[None, None, None, :]
    return torch.nn.functional.scaled_dot_product_attention(
        t(q)[None, None, None, :], t(K)[None, None], t(V)[None, None],
        attn_mask=mask)[0, 0, 0].numpy()


def call(c, l0=0, nl=None):
    nl = c["L"] - l0 if nl is None else nl
    return O.decode_attention(c["q"][l0:l0 + nl], c["K"], c["V"], c["log_m"], c["offsets"],
                              c["K_app"], c["V_app"], c["n_app"], L=c["L"], G=c["G"], l0=l0)


def test_zero_log_m_is_sdpa_per_head(oracle_lib):
    # every (l, h) attends to the entries of its own KV head g = h // gq only
    c = ragged(0, L=2, G=3, gq=2, d=16)
    out = call(c)
    off = c["offsets"]
    for l in range(2):
        for h in range(6):
            lg = l * 3 + h // 2
            ref = sdpa(c["q"][l, h], c["K"][off[lg]:off[lg + 1]], c["V"][off[lg]:off[lg + 1]])
            np.testing.assert_allclose(out[l, h], ref, rtol=0, atol=1e-12)


def test_log_m_is_an_additive_logit_bias(oracle_lib):
    # Eq. app_decode_logit adds log m to the scaled logit: the same as
    # torch's attention with an additive float mask equal to log m
    c = ragged(1, L=1, G=2, gq=4, d=8, logm_scale=5.0)
    out = call(c)
    off = c["offsets"]
    for h in range(8):
        lg = h // 4
        s = slice(off[lg], off[lg + 1])
        ref = sdpa(c["q"][0, h], c["K"][s], c["V"][s], bias=c["log_m"][s])
        np.testing.assert_allclose(out[0, h], ref, rtol=0, atol=1e-12)


def test_multiplicity_equals_duplicated_entries(oracle_lib):
    # one entry with log m = log n equals n identical copies with log m = 0
    rng = np.random.default_rng(2)
    d, n_e = 8, 12
    K = rng.normal(size=(n_e, d))
    V = rng.normal(size=(n_e, d))
    mult = rng.integers(1, 6, size=n_e)
    q = rng.normal(size=(1, 1, d)) * 3
    a = O.decode_attention(q, K, V, np.log(mult), [0, n_e], L=1, G=1)
    Kd, Vd = np.repeat(K, mult, axis=0), np.repeat(V, mult, axis=0)
    b = O.decode_attention(q, Kd, Vd, np.zeros(len(Kd)), [0, len(Kd)], L=1, G=1)
    np.testing.assert_allclose(a, b, rtol=0, atol=1e-12)
    # a sign or base mistake in the bias would move the output
    c = O.decode_attention(q, K, V, -np.log(mult), [0, n_e], L=1, G=1)
    assert np.abs(c - b).max() > 1e-3


def test_compressed_identical_interval_recovers_full_attention(oracle_lib):
    # App. A.3 (text after Eq. app_decode_logit): identical, coherent keys and
    # identical values -> the prototype with its log m_eff recovers the
    # interval's attention mass exactly (up to the eps of the coherence)
    T, d, a, b = 48, 8, 10, 30
    rng = np.random.default_rng(8)
    K = rng.normal(size=(1, 1, T, d))
    V = rng.normal(size=(1, 1, T, d))
    K[0, 0, a:b] = K[0, 0, a]
    V[0, 0, a:b] = V[0, 0, a]
    Q = rng.normal(size=(1, 1, 4, d))
    p = O.make_params(1, 1, 1, T, d, 4, 0.0, recent=4)
    m, Z, _ = O.row_stats(p, Q, K)
    r = O.token_values(p, Q, K, m, Z)
    pr = O.eval_interval(p, K, V, Q, m, Z, r, 0, 0, a, b)
    Kc = np.concatenate([K[0, 0, :a], pr["ktil"][None], K[0, 0, b:]])
    Vc = np.concatenate([V[0, 0, :a], pr["vtil"][None], V[0, 0, b:]])
    lm = np.zeros(len(Kc))
    lm[a] = pr["logm"]
    q = rng.normal(size=(1, 1, d)) * 2
    comp = O.decode_attention(q, Kc, Vc, lm, [0, len(Kc)], L=1, G=1)
    full = sdpa(q[0, 0], K[0, 0], V[0, 0])
    np.testing.assert_allclose(comp[0, 0], full, rtol=0, atol=1e-6)


def test_appended_rows_have_multiplicity_one(oracle_lib):
    # appends behave exactly like packed entries with log m = 0 placed after
    # the packed entries of their (l, g)
    c = ragged(3, L=2, G=2, gq=2, d=8, app_cap=5, n_app=3, logm_scale=3.0)
    out = call(c)
    off = c["offsets"]
    Ks, Vs, lms, offs = [], [], [], [0]
    for lg in range(4):
        l, g = divmod(lg, 2)
        Ks += [c["K"][off[lg]:off[lg + 1]], c["K_app"][l, g, :3]]
        Vs += [c["V"][off[lg]:off[lg + 1]], c["V_app"][l, g, :3]]
        lms += [c["log_m"][off[lg]:off[lg + 1]], np.zeros(3)]
        offs.append(offs[-1] + off[lg + 1] - off[lg] + 3)
    ref = O.decode_attention(c["q"], np.concatenate(Ks), np.concatenate(Vs),
                             np.concatenate(lms), offs, L=2, G=2)
    np.testing.assert_allclose(out, ref, rtol=0, atol=1e-13)
    # rows past n_app are not read
    c2 = dict(c)
    c2["K_app"] = c["K_app"].copy()
    c2["K_app"][:, :, 3:] = 1e6
    np.testing.assert_array_equal(call(c2), out)


def test_softmax_invariances_and_special_cases(oracle_lib):
    c = ragged(4, L=1, G=2, gq=1, d=8, counts=[5, 1], logm_scale=2.0)
    out = call(c)
    # a single entry returns its value whatever its logit
    np.testing.assert_allclose(out[0, 1], c["V"][5], rtol=0, atol=1e-15)
    # a constant added to every log m of an (l, g) changes nothing
    c2 = dict(c)
    c2["log_m"] = c["log_m"] + np.array([7.0] * 5 + [-3.0])
    np.testing.assert_allclose(call(c2), out, rtol=0, atol=1e-13)
    # the output is a convex combination of the values
    lo, hi = c["V"][:5].min(0), c["V"][:5].max(0)
    assert np.all(out[0, 0] >= lo - 1e-12) and np.all(out[0, 0] <= hi + 1e-12)


def test_empty_head_gives_zero_and_layer_slices_agree(oracle_lib):
    c = ragged(5, L=3, G=2, gq=2, d=8, counts=[3, 0, 4, 2, 0, 6])
    out = call(c)
    assert np.all(out[0, 2:4] == 0) and np.all(out[2, 0:2] == 0)
    np.testing.assert_array_equal(call(c, l0=1, nl=2), out[1:])
    # with an append the empty heads attend to the appended row alone
    c2 = ragged(5, L=3, G=2, gq=2, d=8, counts=[3, 0, 4, 2, 0, 6], app_cap=2, n_app=1)
    out2 = call(c2)
    np.testing.assert_allclose(out2[0, 2], c2["V_app"][0, 1, 0], rtol=0, atol=1e-15)


def test_extreme_logits_stay_finite(oracle_lib):
    c = ragged(6, L=1, G=1, gq=2, d=8, counts=[30])
    c["q"] = c["q"] * 400.0
    c["log_m"] = np.linspace(0, 50, 30)
    out = call(c)
    assert np.all(np.isfinite(out))
    # the largest logit dominates completely
    x = c["K"] @ c["q"][0, 0] / math.sqrt(8) + c["log_m"]
    e = int(np.argmax(x))
    srt = np.sort(x)
    if srt[-1] - srt[-2] > 50:
        np.testing.assert_allclose(out[0, 0], c["V"][e], atol=1e-12)
