"""Pins of the oracle's budget, curvature, robust-z and DP segmentation.

Each pin compares the oracle with something other than its own code: a
closed form, a library routine, or brute-force enumeration.
"""
import itertools
import math

import numpy as np
import pytest

import oracle as O


def params(L=1, G=1, Hq=1, T=64, d=2, W=1, **kw):
    return O.make_params(L, G, Hq, T, d, W, 0.0, **kw)


# --- budget: App. A.1 Eq. (app_total_budget), (app_free_budget) -----------------

def test_budget_pr1_closed_form(oracle_lib):
    # PR1: 1 layer x 2 KV heads x 1024 tokens at 8x -> B_total = 256,
    # recent window 32 per (l, g) -> B_free = 256 - 2*32 = 192.
    p = O.make_params(1, 2, 2, 1024, 128, 32, 1e4)
    assert O.budget(p, (1 * 2 * 1024) // 8) == (32, 192)


def test_budget_shrinks_recent_window(oracle_lib):
    p = O.make_params(1, 4, 4, 1024, 8, 4, 0.0)
    # 4 * 32 = 128 > 100 -> r = floor(100 / 4) = 25, B_free = 0
    assert O.budget(p, 100) == (25, 0)
    with pytest.raises(ValueError):   # floor(12/4) = 3 < 4
        O.budget(p, 12)


# --- curvature: App. B.2 ----------------------------------------------------------

def circle_kappa(w, omega):
    """Closed form of kappa^(l,w) on a unit circle h_t = (cos wt, sin wt).

    With r = sin(w om/2) / (w sin(om/2)), the window means are
    mu_- = r (cos((w-1) om/2), -sin((w-1) om/2)) and
    mu_+ = r (cos((w+1) om/2), sin((w+1) om/2)) in the frame where h_i = (1, 0)
    (Dirichlet-kernel sums), so delta_- = h_i - mu_- and delta_+ = mu_+ - h_i.
    """
    r = math.sin(w * omega / 2) / (w * math.sin(omega / 2))
    dm = np.array([1 - r * math.cos((w - 1) * omega / 2), r * math.sin((w - 1) * omega / 2)])
    dp = np.array([r * math.cos((w + 1) * omega / 2) - 1, r * math.sin((w + 1) * omega / 2)])
    return 1.0 - dm @ dp / (np.linalg.norm(dm) * np.linalg.norm(dp))


@pytest.mark.parametrize("omega", [0.05, 0.3, 1.1])
def test_curvature_circle_closed_form(oracle_lib, omega):
    T = 64
    t = np.arange(T)
    V = np.stack([np.cos(omega * t), np.sin(omega * t)], -1).reshape(1, 1, T, 2) * 2.5
    p = params(T=T)
    kap, klw = O.curvature(p, V)
    ws = (4, 8, 16)
    for wi, w in enumerate(ws):
        exp = np.zeros(T)
        exp[w:T - w] = circle_kappa(w, omega)
        np.testing.assert_allclose(klw[:, wi], exp, rtol=0, atol=1e-12)
    vals = np.stack([klw[:, wi] for wi in range(3)], -1)
    # Eq. (app_stabilized_curvature): mean minus 0.25 population std
    np.testing.assert_allclose(kap, vals.mean(-1) - 0.25 * vals.std(-1), atol=1e-12)


def test_curvature_constant_trajectory_is_one_inside(oracle_lib):
    # delta_- = delta_+ = 0 -> u = 0 / eps = 0 -> kappa = 1 - <0, 0> = 1.
    T = 40
    V = np.ones((1, 1, T, 3))
    _, klw = O.curvature(params(T=T, d=3), V)
    for wi, w in enumerate((4, 8, 16)):
        exp = np.zeros(T)
        exp[w:T - w] = 1.0
        np.testing.assert_array_equal(klw[:, wi], exp)


def test_curvature_short_sequence_is_zero(oracle_lib):
    # T < 2w+1 -> the scale is zero everywhere (App. B.2).
    T = 9
    V = np.random.default_rng(0).normal(size=(1, 1, T, 4))
    _, klw = O.curvature(params(T=T, d=4), V)
    assert np.all(klw[:, 1] == 0) and np.all(klw[:, 2] == 0)
    assert np.any(klw[:, 0] != 0)


def test_curvature_invariances(oracle_lib):
    rng = np.random.default_rng(1)
    T, G, d = 50, 2, 4
    V = rng.normal(size=(1, G, T, d))
    p = params(G=G, Hq=G, T=T, d=d)
    k0, _ = O.curvature(p, V)
    k1, _ = O.curvature(p, V * 7.0)                       # per-token normalisation
    Qm, _ = np.linalg.qr(rng.normal(size=(G * d, G * d)))
    h = V[0].transpose(1, 0, 2).reshape(T, G * d) @ Qm.T  # rotation of the trajectory
    k2, _ = O.curvature(p, h.reshape(T, G, d).transpose(1, 0, 2)[None])
    np.testing.assert_allclose(k1, k0, atol=1e-12)
    np.testing.assert_allclose(k2, k0, atol=1e-12)


def test_curvature_hidden_states_override(oracle_lib):
    rng = np.random.default_rng(2)
    T = 40
    H = rng.normal(size=(1, T, 6))
    p = params(T=T, d=2)
    k_h, _ = O.curvature(p, np.zeros((1, 1, T, 2)), hidden=H)
    # the same trajectory passed as values of one 6-dim head
    p6 = params(T=T, d=6)
    k_v, _ = O.curvature(p6, H.reshape(1, 1, T, 6))
    np.testing.assert_allclose(k_h, k_v, atol=1e-14)


# --- robust z: App. B.2 Eqs. (app_robust_z), (app_mad) ---------------------------------

@pytest.mark.parametrize("n", [1, 2, 7, 10, 101])
def test_robust_z_matches_sort_median(oracle_lib, n):
    a = np.random.default_rng(n).normal(size=n) ** 3
    s = np.sort(a)
    med = s[(n - 1) // 2]                 # lower median
    mad = np.sort(np.abs(a - med))[(n - 1) // 2]
    np.testing.assert_allclose(O.robust_z(a), (a - med) / (1.4826 * mad + 1e-6), rtol=1e-15)
    if n % 2 == 1:
        np.testing.assert_allclose(med, np.median(a))


def test_robust_z_of_zero_signal_is_zero(oracle_lib):
    # surprisal defaults to 0: median 0, MAD 0 -> z = 0 / 1e-6 = 0 exactly.
    assert np.all(O.robust_z(np.zeros(17)) == 0.0)


# --- DP segmentation: App. B.3 --------------------------------------------------------

def _disp_lib(hb, cs, a, e):
    """Sample variance of adjacent differences via numpy's var (ddof=1)."""
    nS = e - a - 1
    if nS < 2:
        return 0.0
    d = hb[cs + a + 1:cs + e] - hb[cs + a:cs + e - 1]
    return float(np.var(d, axis=0, ddof=1).sum())


def _brute_dp(b, hb, cs, N, n_min, n_max, n0, lam_d=0.25, lam_n=0.10, c_cut=1.0):
    """Enumerate every composition of N; return (best value, best starts)."""
    best, arg = -np.inf, None

    def value(starts):
        v = 0.0
        for j in range(len(starts) - 1):
            a, e = starts[j], starts[j + 1]
            if a > 0:
                v += b[cs + a - 1] - c_cut
            v -= lam_d * _disp_lib(hb, cs, a, e)
            v -= lam_n * ((e - a - n0) / n0) ** 2
        return v

    def rec(pos, acc, relaxed):
        nonlocal best, arg
        if pos == N:
            v = value(acc + [N])
            if v > best + 1e-12:
                best, arg = v, acc + [N]
            return
        lo = 1 if relaxed else n_min
        for ln in range(lo, n_max + 1):
            if pos + ln > N:
                break
            if relaxed and pos + ln != N:
                continue
            rec(pos + ln, acc + [pos], relaxed)

    rec(0, [], False)
    if arg is None:                     # terminal relaxation of the last slot only
        rec(0, [], True) if N <= n_max else None
        if arg is None:
            # general relaxation: standard prefix then a short final slot
            def rec2(pos, acc):
                nonlocal best, arg
                for ln in range(1, n_max + 1):
                    if pos + ln == N:
                        v = value(acc + [pos, N])
                        if v > best + 1e-12:
                            best, arg = v, acc + [pos, N]
                for ln in range(n_min, n_max + 1):
                    if pos + ln < N:
                        rec2(pos + ln, acc + [pos])
            rec2(0, [])
    return best, arg


def _traj(V, cs=0):
    L, G, T, d = V.shape
    h = V[0].transpose(1, 0, 2).reshape(T, G * d)
    return h / np.maximum(np.linalg.norm(h, axis=1, keepdims=True), 1e-6)


@pytest.mark.parametrize("seed,N,n_min,n_max,n0,cs", [
    (0, 18, 2, 6, 4, 0), (1, 21, 2, 6, 4, 3), (2, 16, 3, 5, 4, 0), (3, 7, 4, 6, 5, 0),
    (4, 3, 4, 6, 5, 0), (5, 22, 2, 7, 3, 2)])
def test_dp_matches_exhaustive_enumeration(oracle_lib, seed, N, n_min, n_max, n0, cs):
    rng = np.random.default_rng(seed)
    r = 4
    T = cs + N + r + 2
    V = rng.normal(size=(1, 2, T, 3))
    p = O.make_params(1, 2, 2, T, 3, 1, 0.0, ctx_start=cs, ctx_end=T - 2, recent=r,
                      n_min=n_min, n_max=n_max, n0=n0, windows=(2, 3))
    seg = O.segment(p, V)
    best, arg = _brute_dp(seg["b"], _traj(V), cs, N, n_min, n_max, n0)
    np.testing.assert_allclose(seg["dp_best"][N], best, rtol=1e-12, atol=1e-12)
    assert list(seg["slot_starts"] - cs) == arg


@pytest.mark.parametrize("disp_mode", [0, 1])
def test_dp_weights_match_numpy_and_sum_to_dp_value(oracle_lib, disp_mode):
    # w(a, i) = Gamma(a) - lambda_d Disp([a, i)) - lambda_n ((i-a-n0)/n0)^2, Eq. (app_dp_recurrence):
    # each weight against numpy's sample variance of the differences, and the
    # weights along the DP's own partition add up to its optimum F[N].
    rng = np.random.default_rng(11)
    cs, N, r = 3, 60, 4
    T = cs + N + r + 2
    V = rng.normal(size=(1, 2, T, 5))
    p = O.make_params(1, 2, 2, T, 5, 1, 0.0, ctx_start=cs, ctx_end=T - 2, recent=r,
                      n_min=4, n_max=12, n0=8, windows=(2, 3), disp_mode=disp_mode)
    seg = O.segment(p, V)
    b, hb = seg["b"], _traj(V)
    pairs = [(a, i) for a in range(0, N - 1, 3) for i in range(a + 1, min(N, a + 14) + 1, 2)]
    w = O.dp_weights(p, V, b, [x for x, _ in pairs], [y for _, y in pairs])
    ref = [(b[cs + a - 1] - 1.0 if a > 0 else 0.0) - 0.25 * _disp_lib(hb, cs, a, i)
           - 0.10 * ((i - a - 8) / 8) ** 2 for a, i in pairs]
    np.testing.assert_allclose(w, ref, rtol=1e-10, atol=1e-10)
    ss = seg["slot_starts"] - cs
    w_path = O.dp_weights(p, V, b, ss[:-1], ss[1:])
    np.testing.assert_allclose(w_path.sum(), seg["dp_best"][N], rtol=1e-12, atol=1e-12)


def test_dp_dispersion_forms_agree(oracle_lib):
    # Eq. (app_layer_dispersion) vs the equivalent form Eq. (app_prefix_dispersion)
    rng = np.random.default_rng(9)
    T = 300
    V = rng.normal(size=(1, 2, T, 8)) + np.linspace(0, 3, T)[None, None, :, None]
    kw = dict(recent=8, n_min=8, n_max=24, n0=16)
    s0 = O.segment(O.make_params(1, 2, 2, T, 8, 1, 0.0, disp_mode=0, **kw), V)
    s1 = O.segment(O.make_params(1, 2, 2, T, 8, 1, 0.0, disp_mode=1, **kw), V)
    assert np.array_equal(s0["slot_starts"], s1["slot_starts"])
    np.testing.assert_allclose(s0["dp_best"], s1["dp_best"], rtol=1e-9)


def test_segment_lengths_respect_bounds(oracle_lib):
    rng = np.random.default_rng(3)
    T = 700
    V = rng.normal(size=(1, 2, T, 8))
    p = O.make_params(1, 2, 2, T, 8, 1, 0.0)
    ss = O.segment(p, V)["slot_starts"]
    ln = np.diff(ss)
    assert ss[0] == 0 and ss[-1] == T - 32
    assert np.all(ln[:-1] >= 16) and np.all(ln <= 128) and ln[-1] >= 1
