"""ctypes wrapper of the plain C oracle (gracekv_oracle.c).

TEST INFRASTRUCTURE ONLY: tests/, __graft_entry__.smoke() and bench.py's
CPU-baseline leg use it to check and time against the CUDA path.  It shares
nothing with the CUDA library; inputs are widened to float64 exactly.
"""
from __future__ import annotations

import ctypes as C
import dataclasses
import os
import subprocess
from typing import Optional

import numpy as np

HERE = os.path.dirname(os.path.abspath(__file__))
SRC = os.path.join(HERE, "gracekv_oracle.c")
LIB = os.path.join(HERE, "liboracle.so")

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with gcc (no fast-math, no FMA contraction)."""
    if force or not os.path.exists(LIB) or os.path.getmtime(LIB) < max(
            os.path.getmtime(SRC), os.path.getmtime(os.path.join(HERE, "gracekv_oracle.h"))):
        tmp = LIB + f".tmp{os.getpid()}"
        subprocess.check_call(["gcc", "-O2", "-ffp-contract=off", "-fno-fast-math", "-std=c11",
                               "-shared", "-fPIC", "-o", tmp, SRC, "-lm"])
        os.replace(tmp, LIB)
    return LIB


class Params(C.Structure):
    _fields_ = [
        ("L", C.c_int32), ("G", C.c_int32), ("Hq", C.c_int32), ("T", C.c_int32),
        ("d", C.c_int32), ("W", C.c_int32),
        ("ctx_start", C.c_int32), ("ctx_end", C.c_int32), ("recent", C.c_int32),
        ("rope_base", C.c_double),
        ("n_min", C.c_int32), ("n_max", C.c_int32), ("n0", C.c_int32),
        ("lambda_stab", C.c_double), ("lambda_s", C.c_double), ("lambda_d", C.c_double),
        ("lambda_n", C.c_double), ("c_cut", C.c_double),
        ("seg_layers", C.c_int32 * 8), ("n_seg_layers", C.c_int32),
        ("windows", C.c_int32 * 4), ("n_windows", C.c_int32),
        ("k_cand", C.c_int32),
        ("lambda_kappa", C.c_double), ("lambda_Z", C.c_double), ("lambda_M", C.c_double),
        ("eps", C.c_double), ("base_frac", C.c_double),
        ("disp_mode", C.c_int32),
        ("alpha_floor", C.c_double), ("floor_c", C.c_double), ("floor_gamma", C.c_double),
        ("floor_eta", C.c_double), ("floor_half", C.c_int32),
        ("lambda_graph", C.c_double), ("eta_seed", C.c_double), ("rho_hop", C.c_double),
        ("m_seed", C.c_int32), ("r_hop", C.c_int32),
        ("seg_mode", C.c_int32), ("quota_alloc", C.c_int32),
    ]


_NODE_I32 = ["lg", "slot", "a", "b", "parent", "child0", "nchild", "form", "cost", "floor_op"]
_NODE_F64 = ["D", "Ddrop", "R", "U", "kappa", "kscale", "m_cut", "m_form", "m_topk", "m_ext"]


class Nodes(C.Structure):
    _fields_ = ([("cap", C.c_int64), ("count", C.c_int64)]
                + [(n, C.POINTER(C.c_int32)) for n in _NODE_I32]
                + [(n, C.POINTER(C.c_double)) for n in _NODE_F64])


def lib():
    global _lib
    if _lib is None:
        build()
        _lib = C.CDLL(LIB)
    return _lib


def _p(a, t):
    return a.ctypes.data_as(C.POINTER(t))


def _f64(x) -> np.ndarray:
    if x is None:
        return None
    if hasattr(x, "detach"):
        x = x.detach().to("cpu").double().numpy()
    return np.ascontiguousarray(np.asarray(x, dtype=np.float64))


PAPER_DEFAULTS = dict(
    recent=32, n_min=16, n_max=128, n0=64, lambda_stab=0.25, lambda_s=0.15,
    lambda_d=0.25, lambda_n=0.10, c_cut=1.0, windows=(4, 8, 16), k_cand=16,
    lambda_kappa=0.05, lambda_Z=0.25, lambda_M=0.75, eps=1e-6, base_frac=0.1,
    seg_layers=(), disp_mode=0, seg_mode=0, quota_alloc=0,
    alpha_floor=0.0, floor_c=0.5, floor_gamma=1.2, floor_eta=0.95, floor_half=3,
    lambda_graph=0.0, eta_seed=0.9, rho_hop=0.5, m_seed=64, r_hop=2)


def make_params(L, G, Hq, T, d, W, rope_base, ctx_start=0, ctx_end=None, **kw) -> Params:
    o = dict(PAPER_DEFAULTS)
    o.update(kw)
    p = Params()
    p.L, p.G, p.Hq, p.T, p.d, p.W = L, G, Hq, T, d, W
    p.ctx_start = ctx_start
    p.ctx_end = T if ctx_end is None else ctx_end
    p.recent = o["recent"]
    p.rope_base = float(rope_base)
    p.n_min, p.n_max, p.n0 = o["n_min"], o["n_max"], o["n0"]
    p.lambda_stab, p.lambda_s = o["lambda_stab"], o["lambda_s"]
    p.lambda_d, p.lambda_n, p.c_cut = o["lambda_d"], o["lambda_n"], o["c_cut"]
    sl = tuple(o["seg_layers"])
    for i, v in enumerate(sl):
        p.seg_layers[i] = v
    p.n_seg_layers = len(sl)
    for i, v in enumerate(o["windows"]):
        p.windows[i] = v
    p.n_windows = len(o["windows"])
    p.k_cand = o["k_cand"]
    p.lambda_kappa, p.lambda_Z, p.lambda_M = o["lambda_kappa"], o["lambda_Z"], o["lambda_M"]
    p.eps, p.base_frac = o["eps"], o["base_frac"]
    p.disp_mode = o["disp_mode"]
    p.seg_mode = o["seg_mode"]
    p.quota_alloc = o["quota_alloc"]
    p.alpha_floor, p.floor_c = o["alpha_floor"], o["floor_c"]
    p.floor_gamma, p.floor_eta, p.floor_half = o["floor_gamma"], o["floor_eta"], o["floor_half"]
    p.lambda_graph, p.eta_seed, p.rho_hop = o["lambda_graph"], o["eta_seed"], o["rho_hop"]
    p.m_seed, p.r_hop = o["m_seed"], o["r_hop"]
    return p


def budget(p: Params, B_total: int):
    r = C.c_int32()
    bf = C.c_int64()
    rc = lib().orc_budget(C.byref(p), C.c_int64(B_total), C.byref(r), C.byref(bf))
    if rc:
        raise ValueError(f"budget rejected (rc={rc})")
    return r.value, bf.value


def curvature(p: Params, V, hidden=None):
    V = _f64(V)
    hid = _f64(hidden)
    Dh = 0 if hid is None else hid.shape[-1]
    kap = np.zeros(p.T)
    nl = p.n_seg_layers or len({min(int(np.floor(r * p.L)), p.L - 1) for r in (0.33, 0.5, 0.67)})
    klw = np.zeros((p.T, nl * p.n_windows))
    rc = lib().orc_curvature(C.byref(p), _p(V, C.c_double),
                             None if hid is None else _p(hid, C.c_double), C.c_int32(Dh),
                             _p(kap, C.c_double), _p(klw, C.c_double))
    assert rc == 0, rc
    return kap, klw


def robust_z(a):
    a = _f64(a)
    z = np.zeros_like(a)
    rc = lib().orc_robust_z(_p(a, C.c_double), C.c_int32(a.size), _p(z, C.c_double))
    assert rc == 0
    return z


def uniform_slots(p: Params):
    """Slot starts of the "w/o CS" ablation (uniform slots of target n0)."""
    N = p.ctx_end - p.recent - p.ctx_start
    starts = np.zeros(N + 2, dtype=np.int32)
    J = C.c_int32()
    rc = lib().orc_uniform_slots(C.byref(p), _p(starts, C.c_int32), C.c_int32(N + 1), C.byref(J))
    assert rc == 0, rc
    return starts[:J.value + 1].copy()


def segment(p: Params, V, hidden=None, surprisal=None):
    V = _f64(V)
    hid = _f64(hidden)
    sur = _f64(surprisal)
    Dh = 0 if hid is None else hid.shape[-1]
    N = p.ctx_end - p.recent - p.ctx_start
    kap = np.zeros(p.T)
    b = np.zeros(p.T)
    cap = N + 2
    starts = np.zeros(cap + 1, dtype=np.int32)
    J = C.c_int32()
    best = np.full(N + 1, -np.inf)
    second = np.full(N + 1, -np.inf)
    rc = lib().orc_segment(C.byref(p), _p(V, C.c_double),
                           None if hid is None else _p(hid, C.c_double), C.c_int32(Dh),
                           None if sur is None else _p(sur, C.c_double),
                           _p(kap, C.c_double), _p(b, C.c_double), _p(starts, C.c_int32),
                           C.c_int32(cap), C.byref(J), _p(best, C.c_double), _p(second, C.c_double))
    assert rc == 0, rc
    return dict(kappa=kap, b=b, slot_starts=starts[:J.value + 1].copy(), dp_best=best,
                dp_second=second)


def dp_weights(p: Params, V, b, a_rel, i_rel, hidden=None):
    """Edge weights w(a, i) of the segmentation DP for the given position pairs."""
    V = _f64(V)
    hid = _f64(hidden)
    bb = _f64(b)
    Dh = 0 if hid is None else hid.shape[-1]
    a_ = np.ascontiguousarray(np.asarray(a_rel, dtype=np.int32))
    i_ = np.ascontiguousarray(np.asarray(i_rel, dtype=np.int32))
    w = np.zeros(len(a_))
    rc = lib().orc_dp_weights(C.byref(p), _p(V, C.c_double),
                              None if hid is None else _p(hid, C.c_double), C.c_int32(Dh),
                              _p(bb, C.c_double), C.c_int32(len(a_)), _p(a_, C.c_int32),
                              _p(i_, C.c_int32), _p(w, C.c_double))
    assert rc == 0, rc
    return w


def row_stats(p: Params, Q, K):
    Q, K = _f64(Q), _f64(K)
    n = p.L * p.Hq * p.W
    m, Z, ZC = np.zeros(n), np.zeros(n), np.zeros(n)
    rc = lib().orc_row_stats(C.byref(p), _p(Q, C.c_double), _p(K, C.c_double),
                             _p(m, C.c_double), _p(Z, C.c_double), _p(ZC, C.c_double))
    assert rc == 0
    sh = (p.L, p.Hq, p.W)
    return m.reshape(sh), Z.reshape(sh), ZC.reshape(sh)


def token_values(p: Params, Q, K, m, Z):
    Q, K = _f64(Q), _f64(K)
    m, Z = _f64(m), _f64(Z)
    Nc = p.ctx_end - p.recent - p.ctx_start
    r = np.zeros(p.L * p.G * Nc)
    rc = lib().orc_token_values(C.byref(p), _p(Q, C.c_double), _p(K, C.c_double),
                                _p(m, C.c_double), _p(Z, C.c_double), _p(r, C.c_double))
    assert rc == 0
    return r.reshape(p.L, p.G, Nc)


def eval_interval(p: Params, K, V, Q, m, Z, rtok, l, g, a, b):
    K, V, Q, m, Z, rtok = map(_f64, (K, V, Q, m, Z, rtok))
    D, Dd, lm = C.c_double(), C.c_double(), C.c_double()
    pos = C.c_int32()
    kt, vt = np.zeros(p.d), np.zeros(p.d)
    rc = lib().orc_eval_interval(C.byref(p), _p(K, C.c_double), _p(V, C.c_double),
                                 _p(Q, C.c_double), _p(m, C.c_double), _p(Z, C.c_double),
                                 _p(rtok, C.c_double), *(C.c_int32(int(v)) for v in (l, g, a, b)),
                                 C.byref(D), C.byref(Dd),
                                 _p(kt, C.c_double), _p(vt, C.c_double), C.byref(pos),
                                 C.byref(lm))
    assert rc == 0
    return dict(D=D.value, Ddrop=Dd.value, ktil=kt, vtil=vt, pos=pos.value, logm=lm.value)


@dataclasses.dataclass
class Trees:
    nodes: dict           # field -> array (length count)
    unit_Uadd: np.ndarray  # [L*G*J]
    unit_root: np.ndarray  # [L*G*J]
    n_slots: int
    _keep: tuple = ()

    def struct(self) -> Nodes:
        ns = Nodes()
        n = len(self.nodes["a"])
        ns.cap = n
        ns.count = n
        for f in _NODE_I32:
            setattr(ns, f, _p(self.nodes[f], C.c_int32))
        for f in _NODE_F64:
            setattr(ns, f, _p(self.nodes[f], C.c_double))
        return ns


def floor(p: Params, rtok, slot_starts, B_base: int):
    """Singleton floor (App. A.5 Stage I, App. C.4): scores f, accepted
    positions [L*G, N_c] (uint8), B_floor, number of initial candidates."""
    rtok = _f64(rtok)
    LG, Nc = p.L * p.G, p.ctx_end - p.recent - p.ctx_start
    ss = np.ascontiguousarray(np.asarray(slot_starts, dtype=np.int32))
    f = np.zeros((LG, Nc))
    acc = np.zeros((LG, Nc), dtype=np.uint8)
    bf, nc = C.c_int64(), C.c_int64()
    rc = lib().orc_floor(C.byref(p), _p(rtok, C.c_double), _p(ss, C.c_int32), C.c_int32(len(ss) - 1),
                         C.c_int64(B_base), _p(f, C.c_double), _p(acc, C.c_uint8), C.byref(bf),
                         C.byref(nc))
    assert rc == 0, rc
    return f, acc, bf.value, nc.value


def unit_floor(p: Params, acc, slot_starts):
    """1 for every slot (unit lg * J + j) holding an accepted floor position."""
    ss = np.asarray(slot_starts) - p.ctx_start
    J = len(ss) - 1
    acc = np.asarray(acc).reshape(p.L * p.G, -1)
    return np.stack([acc[:, ss[j]:ss[j + 1]].any(axis=1) for j in range(J)], axis=1).reshape(-1).astype(np.uint8)


def build_trees(p: Params, K, V, Q, kappa, slot_starts, m, Z, rtok, omega=None,
                floor_acc=None, floor_f=None) -> Trees:
    K, V, Q, kappa, m, Z, rtok, om = map(_f64, (K, V, Q, kappa, m, Z, rtok, omega))
    fa = None if floor_acc is None else np.ascontiguousarray(floor_acc, dtype=np.uint8)
    ff = None if floor_f is None else _f64(floor_f)
    ss = np.ascontiguousarray(np.asarray(slot_starts, dtype=np.int32))
    J = len(ss) - 1
    Nc = p.ctx_end - p.recent - p.ctx_start
    cap = p.L * p.G * 2 * Nc + 8
    arr = {f: np.zeros(cap, dtype=np.int32) for f in _NODE_I32}
    arr.update({f: np.zeros(cap) for f in _NODE_F64})
    ns = Nodes()
    ns.cap = cap
    for f in _NODE_I32:
        setattr(ns, f, _p(arr[f], C.c_int32))
    for f in _NODE_F64:
        setattr(ns, f, _p(arr[f], C.c_double))
    uadd = np.zeros(p.L * p.G * J)
    uroot = np.zeros(p.L * p.G * J, dtype=np.int64)
    rc = lib().orc_build_trees(C.byref(p), _p(K, C.c_double), _p(V, C.c_double),
                               _p(Q, C.c_double), None if om is None else _p(om, C.c_double),
                               _p(kappa, C.c_double), _p(ss, C.c_int32), C.c_int32(J),
                               _p(m, C.c_double), _p(Z, C.c_double), _p(rtok, C.c_double),
                               None if fa is None else _p(fa, C.c_uint8),
                               None if ff is None else _p(ff, C.c_double),
                               C.byref(ns), _p(uadd, C.c_double), _p(uroot, C.c_int64))
    assert rc == 0, rc
    n = ns.count
    return Trees({f: arr[f][:n].copy() for f in arr}, uadd, uroot, J)


def allocate(p: Params, B_free: int, tr: Trees, unit_fl=None):
    ns = tr.struct()
    nu = len(tr.unit_Uadd)
    add_sel = np.zeros(nu, dtype=np.uint8)
    split_sel = np.zeros(len(tr.nodes["a"]), dtype=np.uint8)
    used = C.c_int64()
    uf = None if unit_fl is None else np.ascontiguousarray(unit_fl, dtype=np.uint8)
    rc = lib().orc_allocate(C.byref(p), C.c_int64(B_free), C.c_int32(tr.n_slots), C.byref(ns),
                            _p(tr.unit_Uadd, C.c_double), _p(tr.unit_root, C.c_int64),
                            None if uf is None else _p(uf, C.c_uint8),
                            _p(add_sel, C.c_uint8), _p(split_sel, C.c_uint8), C.byref(used))
    assert rc == 0
    return add_sel, split_sel, used.value


def gather(p: Params, K, V, rtok, tr: Trees, add_sel, split_sel, cap: int):
    K, V, rtok = map(_f64, (K, V, rtok))
    ns = tr.struct()
    Ko = np.zeros((cap, p.d))
    Vo = np.zeros((cap, p.d))
    pos = np.zeros(cap, dtype=np.int32)
    lm = np.zeros(cap)
    lo = np.zeros(cap, dtype=np.int32)
    hi = np.zeros(cap, dtype=np.int32)
    off = np.zeros(p.L * p.G + 1, dtype=np.int64)
    ne = C.c_int64()
    rc = lib().orc_gather(C.byref(p), _p(K, C.c_double), _p(V, C.c_double),
                          _p(rtok, C.c_double), C.c_int32(tr.n_slots), C.byref(ns),
                          _p(tr.unit_root, C.c_int64), _p(add_sel, C.c_uint8),
                          _p(split_sel, C.c_uint8), C.c_int64(cap), _p(Ko, C.c_double),
                          _p(Vo, C.c_double), _p(pos, C.c_int32), _p(lm, C.c_double),
                          _p(lo, C.c_int32), _p(hi, C.c_int32), _p(off, C.c_int64), C.byref(ne))
    assert rc == 0, rc
    E = ne.value
    return dict(K=Ko[:E], V=Vo[:E], pos=pos[:E], log_m=lm[:E], src_lo=lo[:E], src_hi=hi[:E],
                offsets=off)


def graph_layers(p: Params):
    out = np.zeros(4, dtype=np.int32)
    n = lib().orc_graph_layers(C.byref(p), _p(out, C.c_int32))
    return out[:n].copy()


def multihop(p: Params, shat, Qg, K, graph_l=None):
    """d-hat [N_c] and the seeds [r_hop, m_seed] / weights of every hop (App. A.4)."""
    shat, Qg, K = _f64(shat), _f64(Qg), _f64(K)
    gl = graph_layers(p) if graph_l is None else np.asarray(graph_l, dtype=np.int32)
    gl = np.ascontiguousarray(gl, dtype=np.int32)
    Nc = p.ctx_end - p.recent - p.ctx_start
    dh = np.zeros(Nc)
    sd = np.zeros((p.r_hop, p.m_seed), dtype=np.int32)
    sw = np.zeros((p.r_hop, p.m_seed))
    rc = lib().orc_multihop(C.byref(p), _p(shat, C.c_double), _p(Qg, C.c_double), _p(gl, C.c_int32),
                            C.c_int32(len(gl)), _p(K, C.c_double), _p(dh, C.c_double), _p(sd, C.c_int32),
                            _p(sw, C.c_double))
    assert rc == 0, rc
    return dh, sd, sw


def head_sensitivity(W_O, o, G: int, eps: float = 1e-6):
    """omega [L, G] from W_O [L, D, Hq*d] and o [L, Hq, U, d] (Eq. app_head_sensitivity)."""
    W_O, o = _f64(W_O), _f64(o)
    L, Hq, U, d = o.shape
    D = W_O.shape[1]
    om = np.zeros((L, G))
    rc = lib().orc_head_sensitivity(*(C.c_int32(v) for v in (L, G, Hq, d, D, U)),
                                    _p(W_O, C.c_double), _p(o, C.c_double), C.c_double(eps),
                                    _p(om, C.c_double))
    assert rc == 0, rc
    return om


def decode_attention(q, K, V, log_m, offsets, K_app=None, V_app=None, n_app: int = 0,
                     *, L: int, G: int, l0: int = 0):
    """Eq. (app_decode_logit) over the packed cache plus n_app appended rows.

    q [nl, Hq, d]; K, V [E, d]; log_m [E]; offsets [L*G + 1];
    K_app, V_app [L, G, app_cap, d] or None.  Returns out [nl, Hq, d]."""
    q, K, V, log_m = map(_f64, (q, K, V, log_m))
    nl, Hq, d = q.shape
    off = np.ascontiguousarray(np.asarray(offsets, dtype=np.int64))
    if K_app is None:
        K_app = np.zeros((L, G, 1, d))
        V_app = np.zeros((L, G, 1, d))
    K_app, V_app = _f64(K_app), _f64(V_app)
    app_cap = K_app.shape[2]
    if K.size == 0:
        K, V, log_m = np.zeros((1, d)), np.zeros((1, d)), np.zeros(1)
    out = np.zeros((nl, Hq, d))
    rc = lib().orc_decode_attention(*(C.c_int32(v) for v in (L, G, Hq, d, l0, nl)),
                                    _p(q, C.c_double), _p(K, C.c_double), _p(V, C.c_double),
                                    _p(log_m, C.c_double), _p(off, C.c_int64),
                                    _p(K_app, C.c_double), _p(V_app, C.c_double),
                                    C.c_int32(app_cap), C.c_int32(n_app), _p(out, C.c_double))
    assert rc == 0, rc
    return out


def run(K, V, Q, B_total: int, rope_base: float, *, ctx_start=0, ctx_end=None, omega=None,
        surprisal=None, hidden=None, slot_starts=None, Qg=None, **overrides) -> dict:
    """Whole compression pass on the oracle; returns every intermediate."""
    L, G, T, d = K.shape
    Hq, W = Q.shape[1], Q.shape[2]
    p = make_params(L, G, Hq, T, d, W, rope_base, ctx_start, ctx_end, **overrides)
    r_eff, B_free = budget(p, B_total)
    p.recent = r_eff
    K64, V64, Q64 = _f64(K), _f64(V), _f64(Q)
    if slot_starts is None and p.seg_mode == 1:
        seg = dict(kappa=np.zeros(p.T), b=None, slot_starts=uniform_slots(p), dp_best=None,
                   dp_second=None)
    elif slot_starts is None:
        seg = segment(p, V64, hidden, surprisal)
    else:
        kap, _ = curvature(p, V64, hidden)
        seg = dict(kappa=kap, b=None, slot_starts=np.asarray(slot_starts, np.int32) + p.ctx_start,
                   dp_best=None, dp_second=None)
    m, Z, ZC = row_stats(p, Q64, K64)
    rtok = token_values(p, Q64, K64, m, Z)
    mh = None
    if p.lambda_graph > 0:
        # App. A.4 Eq. (app_bottom_up_value): R = (1 - lambda) s-hat + lambda d-hat
        assert Qg is not None, "multi-hop relevance needs the graph layers' queries"
        dh, sd, sw = multihop(p, rtok, Qg, K64)
        mh = dict(dhat=dh, seeds=sd, weights=sw, shat=rtok.copy())
        rtok = (1.0 - p.lambda_graph) * rtok + p.lambda_graph * dh[None, None, :]
    fl = None
    if p.alpha_floor > 0:
        f, acc, B_floor, n_cand = floor(p, rtok, seg["slot_starts"], B_free)
        fl = dict(f=f, accepted=acc, B_floor=B_floor, n_cand=n_cand,
                  unit_floor=unit_floor(p, acc, seg["slot_starts"]))
    tr = build_trees(p, K64, V64, Q64, seg["kappa"], seg["slot_starts"], m, Z, rtok, omega,
                     None if fl is None else fl["accepted"], None if fl is None else fl["f"])
    add_sel, split_sel, used = allocate(p, B_free, tr, None if fl is None else fl["unit_floor"])
    cap = B_total + L * G * (T - (p.ctx_end - p.ctx_start)) + 16
    cache = gather(p, K64, V64, rtok, tr, add_sel, split_sel, cap)
    return dict(params=p, r_eff=r_eff, B_free=B_free, seg=seg, m=m, Z=Z, ZC=ZC, rtok=rtok,
                trees=tr, add_sel=add_sel, split_sel=split_sel, used=used, cache=cache, floor=fl,
                multihop=mh)
