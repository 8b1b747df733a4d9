"""Independent pins of the oracle's distortion, refinement rule and gains.

Everything here is restated in numpy from the paper's equations, sharing no
code with the oracle:

  D_q = lambda_Z (Z - Zt)^2 / (Z^2 + eps) + lambda_M |M - Zt vt|^2 / (|M|^2 + eps),
  Zt = m_eff exp(q.kt / sqrt d - m), D = Mean_q [Z_q / Ztot_q D_q],
  D_drop = Mean_q Z_q / Ztot_q             (App. A.3 Eqs. app_original_attention_stats,
                                          app_prototype_attention_stats,
                                          app_probe_distortion,
                                          app_node_and_drop_distortion)
  kt = RoPE(mean_t RoPE^-1(k_t, t), p), p = round(mean t), coh, m_eff, beta,
  vt                                       (Eqs. app_rope_prototype,
                                          app_value_prototype,
                                          app_effective_multiplicity)
  X_v = TopK16(kappa) u {mid}, G_bin = D(I) - D(L) - D(R) + lambda_kappa kappa-hat,
  G_ext = D(I) - sum D(children), c_ext = |children| - 1, the larger rho wins
                                         (Eqs. app_tree_split_candidates,
                                          app_binary_split, app_extract_split,
                                          app_split_choice)
  U = max(0, omega R (D - sum D(children))) / c, Add: omega R (D_drop - D)
                                         (App. A.5 Eqs. app_operation_gains,
                                          app_operation_costs, app_unit_utility)

with the readings the oracle states for the places the paper leaves open:
probe u of KV head g uses query head g |H(g)| + (u mod |H(g)|); the shift m
and the partition Ztot are the probe's over [0, T); epsilon = 1e-6; RoPE
pairs (i, i + d/2) with theta_i = base^(-2i/d); p rounds half to even; a
candidate position t in [a, b-2] cuts at xi = t + 1 (ties: lower t), the
midpoint is a + floor(n/2), kappa-hat is the min-max over [a, b-2] (0 when
flat) read at xi - 1, cut ties go to the smallest xi, extraction is at
argmax R (ties: lower t), binary wins a rho tie; gains are clamped at 0; one
token is its own prototype with D = 0.
"""
import numpy as np
import pytest

import oracle as O

LAMBDA_Z, LAMBDA_M, EPS, BASE_FRAC, K_CAND = 0.25, 0.75, 1e-6, 0.1, 16


# ---------------------------------------------------------------- numpy model
def rope(x, t, base):
    """Rotate the pairs (i, i + d/2) of x by t theta_i (complex form)."""
    h = x.shape[-1] // 2
    theta = base ** (-2.0 * np.arange(h) / x.shape[-1])
    z = (x[..., :h] + 1j * x[..., h:]) * np.exp(1j * np.asarray(t, dtype=float)[..., None] * theta)
    return np.concatenate([z.real, z.imag], axis=-1)


class Model:
    """Row statistics, token values and interval evaluation for one problem."""

    def __init__(self, K, V, Q, base, recent, lambda_kappa=0.05, omega=None):
        self.K, self.V, self.Q, self.base = K, V, Q, base
        L, G, T, d = K.shape
        Hq, W = Q.shape[1], Q.shape[2]
        self.L, self.G, self.T, self.d, self.Hq, self.W, self.gq = L, G, T, d, Hq, W, Hq // G
        self.Nc = T - recent
        self.lambda_kappa = lambda_kappa
        self.omega = np.ones((L, G)) if omega is None else omega
        # x[l, h, u, t] = q . k / sqrt d over the visible range [0, T)
        self.x = np.einsum("lhud,lhtd->lhut", Q, np.repeat(K, self.gq, axis=1)) / np.sqrt(d)
        self.m = self.x.max(-1)
        e = np.exp(self.x - self.m[..., None])
        self.Z = e.sum(-1)
        pi = e / self.Z[..., None]                          # Eq. app_attention_probability
        s = pi.reshape(L, G, self.gq * W, T).sum(2)[..., :self.Nc]
        self.R = s / (s.sum(-1, keepdims=True) + EPS)       # Eq. app_direct_relevance

    def proto(self, l, g, a, b):
        K, V, R = self.K[l, g], self.V[l, g], self.R[l, g]
        n = b - a
        if n == 1:
            return K[a], V[a], 1.0
        t = np.arange(a, b)
        kc = rope(K[a:b], -t, self.base)
        mu = kc.mean(0)
        kt = rope(mu, np.round((a + b - 1) / 2.0), self.base)
        coh = np.linalg.norm(mu) / (np.linalg.norm(kc, axis=1).mean() + EPS)
        meff = min(max(n * coh ** 2, 1.0), float(n))
        w = R[a:b] + BASE_FRAC * R[a:b].mean()
        vt = (w[:, None] * V[a:b]).sum(0) / (w.sum() + EPS)
        return kt, vt, meff

    def D(self, l, g, a, b, raw_terms=False):
        """(D, D_drop) of [a, b) for (l, g); with raw_terms the per-probe parts."""
        kt, vt, meff = self.proto(l, g, a, b)
        Dq, w = [], []
        for u in range(self.W):
            h = g * self.gq + (u % self.gq)
            q, mu_ = self.Q[l, h, u], self.m[l, h, u]
            e = np.exp(self.x[l, h, u, a:b] - mu_)
            Zi, Mi = e.sum(), (e[:, None] * self.V[l, g, a:b]).sum(0)
            Zt = meff * np.exp(q @ kt / np.sqrt(self.d) - mu_)
            Dq.append(LAMBDA_Z * (Zi - Zt) ** 2 / (Zi ** 2 + EPS)
                      + LAMBDA_M * np.sum((Mi - Zt * vt) ** 2) / (np.sum(Mi ** 2) + EPS))
            w.append(Zi / self.Z[l, h, u])
        Dq, w = np.array(Dq), np.array(w)
        D = 0.0 if b - a == 1 else float(np.mean(w * Dq))
        return (D, float(w.mean()), Dq, w) if raw_terms else (D, float(w.mean()))

    def split(self, l, g, a, b, kappa):
        """The preselected children of [a, b) and the form (0 binary, 1 extraction)."""
        n = b - a
        DI = self.D(l, g, a, b)[0]
        pos = np.arange(a, b - 1)                                   # t in [a, b-2]
        order = sorted(pos, key=lambda t: (-kappa[t], t))
        cands = sorted({int(t) + 1 for t in order[:K_CAND]} | {a + n // 2})
        kmin, kmax = kappa[a:b - 1].min(), kappa[a:b - 1].max()
        best, bxi = -np.inf, None
        for xi in cands:
            kh = (kappa[xi - 1] - kmin) / (kmax - kmin) if kmax > kmin else 0.0
            gb = DI - self.D(l, g, a, xi)[0] - self.D(l, g, xi, b)[0] + self.lambda_kappa * kh
            if gb > best:
                best, bxi = gb, xi
        R = self.R[l, g]
        p = a + int(np.argmax(R[a:b]))                              # first maximum: lower t
        ext = [(x, y) for x, y in ((a, p), (p, p + 1), (p + 1, b)) if y > x]
        rho_ext = (DI - sum(self.D(l, g, x, y)[0] for x, y in ext)) / (len(ext) - 1)
        if rho_ext > best:
            return ext, 1
        return [(a, bxi), (bxi, b)], 0

    def tree(self, l, g, a, b, kappa):
        """Every node of the unit's tree: (a, b) -> (children, form, U, key)."""
        om = self.omega[l, g]
        D, Dd = self.D(l, g, a, b)
        Rr = self.R[l, g, a:b].sum()
        uadd = max(0.0, om * Rr * (Dd - D))
        out = {}
        todo = [((a, b), uadd)]
        while todo:
            (x, y), creator = todo.pop()
            if y - x == 1:
                continue
            ch, form = self.split(l, g, x, y, kappa)
            gain = om * self.R[l, g, x:y].sum() * (self.D(l, g, x, y)[0]
                                                   - sum(self.D(l, g, s, e)[0] for s, e in ch))
            U = max(0.0, gain) / (len(ch) - 1)
            key = min(U, creator)
            out[(x, y)] = (ch, form, U, key, gain)
            todo += [(c, key) for c in ch]
        return out, uadd


# ---------------------------------------------------------------- problems
def problem(seed, T=72, recent=8, d=8, W=6, G=2, gq=2, spikes=5):
    rng = np.random.default_rng(seed)
    K = rng.normal(size=(1, G, T, d))
    V = rng.normal(size=(1, G, T, d))
    # a few strong keys so that attention concentrates and extraction wins somewhere
    K[:, :, rng.choice(T - recent, spikes, replace=False)] *= 3.0
    Q = rng.normal(size=(1, G * gq, W, d))
    kappa = np.round(rng.random(T), 1)           # ties on purpose
    return K, V, Q, kappa


def oracle_inputs(M, recent, **kw):
    p = O.make_params(M.L, M.G, M.Hq, M.T, M.d, M.W, M.base, recent=recent,
                      lambda_kappa=M.lambda_kappa, **kw)
    return p


# ---------------------------------------------------------------- the pins
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_interval_distortion_matches_the_equations(oracle_lib, seed):
    K, V, Q, _ = problem(seed)
    M = Model(K, V, Q, 1e4, recent=8)
    p = oracle_inputs(M, 8)
    m, Z, _ = O.row_stats(p, Q, K)
    np.testing.assert_allclose(m, M.m, rtol=0, atol=1e-12)
    np.testing.assert_allclose(Z, M.Z, rtol=1e-12)
    R = O.token_values(p, Q, K, m, Z)
    np.testing.assert_allclose(R, M.R, rtol=1e-10, atol=1e-15)
    rng = np.random.default_rng(100 + seed)
    nonzero = 0
    for _ in range(40):
        g = int(rng.integers(0, 2))
        a = int(rng.integers(0, 60))
        b = int(rng.integers(a + 1, min(a + 30, 64) + 1))
        want_D, want_Dd, Dq, w = M.D(0, g, a, b, raw_terms=True)
        got = O.eval_interval(p, K, V, Q, m, Z, R, 0, g, a, b)
        assert got["Ddrop"] == pytest.approx(want_Dd, rel=1e-12)
        assert got["D"] == pytest.approx(want_D, rel=1e-10, abs=1e-300)
        kt, vt, meff = M.proto(0, g, a, b)
        np.testing.assert_allclose(got["ktil"], kt, rtol=1e-10, atol=1e-12)
        np.testing.assert_allclose(got["vtil"], vt, rtol=1e-10, atol=1e-12)
        assert got["logm"] == pytest.approx(np.log(meff), abs=1e-12)
        assert got["pos"] == (a if b - a == 1 else int(np.round((a + b - 1) / 2.0)))
        if b - a > 1:
            nonzero += want_D > 1e-3
            # both terms of D_q matter here, and they differ: swapping lambda_Z
            # and lambda_M would move D by far more than the tolerance
            zt = [LAMBDA_M * x for x in Dq]
            assert abs(np.mean(w * np.array(zt)) - want_D) > 1e-6 * want_D
    assert nonzero >= 20


@pytest.mark.parametrize("seed,lambda_kappa", [(0, 0.05), (1, 0.0), (2, 0.0), (3, 0.05)])
def test_refinement_rule_and_gains_match_a_brute_force_tree(oracle_lib, seed, lambda_kappa):
    recent = 8
    K, V, Q, kappa = problem(seed)
    omega = np.array([[0.7, 1.9]])
    M = Model(K, V, Q, 1e4, recent=recent, lambda_kappa=lambda_kappa, omega=omega)
    p = oracle_inputs(M, recent)
    m, Z, _ = O.row_stats(p, Q, K)
    R = O.token_values(p, Q, K, m, Z)
    slots = np.array([0, 40, 64], np.int32)
    tr = O.build_trees(p, K, V, Q, kappa, slots, m, Z, R, omega=omega)
    nd = tr.nodes
    forms = set()
    for g in range(2):
        for j in range(2):
            a, b = int(slots[j]), int(slots[j + 1])
            want, uadd = M.tree(0, g, a, b, kappa)
            u = g * 2 + j
            assert tr.unit_Uadd[u] == pytest.approx(uadd, rel=1e-9, abs=1e-300)
            r0 = int(tr.unit_root[u])
            r1 = int(tr.unit_root[u + 1]) if u + 1 < len(tr.unit_root) else len(nd["a"])
            got = {}
            for v in range(r0, r1):
                if nd["nchild"][v] <= 0:
                    continue
                c0 = nd["child0"][v]
                ch = [(int(nd["a"][c0 + k]), int(nd["b"][c0 + k])) for k in range(nd["nchild"][v])]
                got[(int(nd["a"][v]), int(nd["b"][v]))] = (ch, int(nd["form"][v]), nd["U"][v],
                                                          nd["kappa"][v], int(nd["cost"][v]))
            assert set(got) == set(want)
            for key, (ch, form, U, kap, gain) in want.items():
                gch, gform, gU, gkap, gcost = got[key]
                assert gch == ch and gform == form, (key, gch, ch)
                assert gcost == len(ch) - 1
                assert gU == pytest.approx(U, rel=1e-9, abs=1e-300), key
                assert gkap == pytest.approx(kap, rel=1e-9, abs=1e-300), key
                forms.add(form)
    assert forms == {0, 1}          # both refinement forms occur


def test_gains_are_clamped_at_zero(oracle_lib):
    # Add: keys k_t = RoPE(c, t) over the slot [0, 32) and one query aimed at
    # RoPE(c, 16), the prototype's position; the prototype then holds the
    # largest logit with m_eff = n, so Zt is about n Z, D_q far exceeds 1 and
    # the raw Add gain omega R (D_drop - D) is negative.  Split: seed 1's
    # problem has a binary split whose children's distortions exceed the
    # parent's.  Both must come out as U = 0 (non-elastic gains, App. C.6).
    d, T, recent = 8, 40, 8
    rng = np.random.default_rng(5)
    c = rng.normal(size=d)
    c *= 2.0 / np.linalg.norm(c)
    K = rope(np.tile(c, (T, 1)), np.arange(T), 2.0)[None, None]
    V = rng.normal(size=(1, 1, T, d))
    Q = np.stack([3.0 * rope(c, 16, 2.0), rng.normal(size=d)])[None, None]
    M = Model(K, V, Q, 2.0, recent=recent)
    D, Dd = M.D(0, 0, 0, 32)
    assert D > Dd > 0
    p = oracle_inputs(M, recent)
    m, Z, _ = O.row_stats(p, Q, K)
    R = O.token_values(p, Q, K, m, Z)
    tr = O.build_trees(p, K, V, Q, np.zeros(T), np.array([0, 32], np.int32), m, Z, R)
    assert tr.unit_Uadd[0] == 0.0
    K, V, Q, kappa = problem(1)
    M = Model(K, V, Q, 1e4, recent=recent)
    p = oracle_inputs(M, recent)
    m, Z, _ = O.row_stats(p, Q, K)
    R = O.token_values(p, Q, K, m, Z)
    tr = O.build_trees(p, K, V, Q, kappa, np.array([0, 40, 64], np.int32), m, Z, R)
    nd = tr.nodes
    negative = 0
    for g in range(2):
        for a, b in ((0, 40), (40, 64)):
            for (x, y), (ch, form, U, key, gain) in M.tree(0, g, a, b, kappa)[0].items():
                if gain < 0:
                    negative += 1
                    v = np.nonzero((nd["lg"] == g) & (nd["a"] == x) & (nd["b"] == y))[0]
                    assert len(v) == 1 and nd["U"][v[0]] == 0.0 and nd["kappa"][v[0]] == 0.0
    assert negative >= 1


def test_extraction_ties_go_to_the_lower_position(oracle_lib):
    # The strongest keys are copied three positions later inside their slot,
    # so two tokens carry bit-identical token values; where such a pair holds
    # a node's largest value and the node extracts, the lower position is the
    # one extracted (reading: argmax R_tok, ties lower t).
    recent = 8
    K, V, Q, kappa = problem(3)
    sp = np.argsort(-np.linalg.norm(K[0, 0, :64], axis=1))[:3]
    for t in sp:
        if t + 3 < 64 and (t < 40) == (t + 3 < 40):
            K[0, :, t + 3] = K[0, :, t]
    M = Model(K, V, Q, 1e4, recent=recent, lambda_kappa=0.0)
    p = oracle_inputs(M, recent)
    m, Z, _ = O.row_stats(p, Q, K)
    R = O.token_values(p, Q, K, m, Z)
    tr = O.build_trees(p, K, V, Q, kappa, np.array([0, 40, 64], np.int32), m, Z, R)
    nd = tr.nodes
    tied = 0
    for g in range(2):
        for a, b in ((0, 40), (40, 64)):
            for (x, y), (ch, form, U, key, gain) in M.tree(0, g, a, b, kappa)[0].items():
                v = np.nonzero((nd["lg"] == g) & (nd["a"] == x) & (nd["b"] == y))[0][0]
                c0 = nd["child0"][v]
                got = [(int(nd["a"][c0 + k]), int(nd["b"][c0 + k])) for k in range(nd["nchild"][v])]
                assert got == ch and nd["form"][v] == form, (x, y)
                Rn = M.R[0, g, x:y]
                if form == 1 and (Rn == Rn.max()).sum() >= 2:
                    tied += 1
                    first = x + int(np.nonzero(Rn == Rn.max())[0][0])
                    assert (first, first + 1) in got
    assert tied >= 2
