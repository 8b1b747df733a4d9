"""C ABI checks that need no GPU: the library loads, exports every function
include/gracekv.h declares, and validates arguments on the host."""
import ctypes as C
import os
import re

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def gk():
    import __graft_entry__ as g
    from paper_2608_07001_gb300 import build_ext
    build_ext.build()
    from paper_2608_07001_gb300 import gracekv
    gracekv.lib()
    return gracekv


def declared_functions():
    src = open(os.path.join(ROOT, "include", "gracekv.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(gracekv_[a-z_]+)\s*\(", src)))


def test_header_declarations_are_exported(gk):
    names = declared_functions()
    assert len(names) >= 12
    lib = C.CDLL(gk.LIBPATH)
    for n in names:
        assert hasattr(lib, n), n
    assert set(names) == set(gk.EXPORTED)


def test_default_params_are_the_papers(gk):
    p = gk.gracekv_default_params()
    assert (p.recent, p.n_min, p.n_max, p.n0, p.k_cand) == (32, 16, 128, 64, 16)
    assert (p.lambda_stab, p.lambda_s, p.lambda_d, p.lambda_n, p.c_cut) == (0.25, 0.15, 0.25, 0.10, 1.0)
    assert list(p.windows)[:p.n_windows] == [4, 8, 16]
    assert (p.lambda_kappa, p.lambda_Z, p.lambda_M, p.eps, p.base_frac) == (0.05, 0.25, 0.75, 1e-6, 0.1)
    assert p.n_seg_layers == 0 and p.lambda_graph == 0.0 and p.alpha_floor == 0.0


def test_budget_for_ratio(gk):
    assert gk.gracekv_budget_for_ratio(1, 2, 1024, 8) == 256
    assert gk.gracekv_budget_for_ratio(32, 8, 131072, 32) == 1048576
    assert gk.gracekv_budget_for_ratio(16, 8, 8192, 1) == 16 * 8 * 8192
    assert gk.gracekv_budget_for_ratio(1, 1, 10, 3.5) == 2
    assert gk.gracekv_budget_for_ratio(0, 2, 1024, 8) == -1
    assert gk.gracekv_budget_for_ratio(1, 2, 1024, 0.5) == -1


def test_graph_layers_match_the_oracle(gk, oracle_lib):
    # the library's host rule for the multi-hop graph layers against the oracle's
    import oracle as O
    for L in range(1, 65):
        p = O.make_params(L, 1, 1, 64, 8, 2, 0.0, recent=8)
        assert gk.gracekv_graph_layers(L) == [int(v) for v in O.graph_layers(p)]
    assert gk.lib().gracekv_graph_layers(0, None) == -1


def _create(gk, **kw):
    base = dict(L=1, G=2, Hq=2, T=1024, d=128, W=32)
    base.update({k: kw.pop(k) for k in list(kw) if k in base})
    p = gk.make_params(base["L"], base["G"], base["Hq"], base["T"], base["d"], base["W"],
                       dtype=kw.pop("dtype", "f32"), budget=kw.pop("budget", 256), rope_base=1e4, **kw)
    h = C.c_void_p()
    return gk.lib().gracekv_create(C.byref(p), C.byref(h)), h


@pytest.mark.parametrize("kw,status", [
    (dict(Hq=3), 1),                       # Hq not a multiple of G
    (dict(ctx_start=5, ctx_end=3), 1),     # empty context
    (dict(n_min=20, n_max=10), 1),
    (dict(k_cand=17), 1),
    (dict(windows=(4, 32)), 1),             # window scale above 16
    (dict(seg_layers=(3,)), 1),             # layer out of range
    (dict(lambda_graph=0.3), 8),            # multi-hop relevance needs bf16
    (dict(lambda_graph=1.5, dtype="bf16"), 1),
    (dict(lambda_graph=0.3, dtype="bf16", m_seed=65), 1),     # one 64-row seed tile
    (dict(lambda_graph=0.3, dtype="bf16", m_seed=0), 1),
    (dict(lambda_graph=0.3, dtype="bf16", eta_seed=0.0), 1),
    (dict(lambda_graph=0.3, dtype="bf16", r_hop=0), 1),
    (dict(lambda_graph=0.3, dtype="bf16", rho_hop=-0.5), 1),
    (dict(lambda_graph=0.3, dtype="bf16", T=131072 + 64), 8),  # N_c above the seed selection's
    (dict(alpha_floor=1.5), 1),             # floor cap above the budget
    (dict(alpha_floor=0.6, floor_eta=1.5), 1),
    (dict(alpha_floor=0.6, quota_alloc=1), 8),   # floor with fixed per-pair capacity
    (dict(d=96), 8),
    (dict(W=128), 8),
    (dict(budget=7), 2),                    # floor(7 / 2) = 3 < 4 recent tokens
])
def test_create_rejects_on_host(gk, kw, status):
    st, h = _create(gk, **kw)
    assert st == status
    assert not h.value


def test_status_strings(gk):
    for s in range(10):
        assert gk.lib().gracekv_status_string(s)


def test_null_context_is_rejected(gk):
    lib = gk.lib()
    n = C.c_int64()
    assert lib.gracekv_allocate(None, C.byref(n), None) == gk.GKV_EINVAL
    assert lib.gracekv_last_error(None) == b"null context"


def test_stage_names_match_the_header(gk):
    # gracekv_stats fills GRACEKV_N_STAGES timers; the binding names each one
    hdr = open(os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))),
                            "include", "gracekv.h")).read()
    n = int(re.search(r"#define GRACEKV_N_STAGES (\d+)", hdr).group(1))
    assert len(gk.Context.STAGES) == n
    assert gk.Context.STAGES[6:] == ("floor", "multihop")
