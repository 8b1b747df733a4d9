"""The paper's printed hyperparameters (tests/golden/paper_hyperparameters.txt,
each line cited) against the defaults of the oracle and of the library.

A stage marked "switch" is off by default in both (0); its paper value is
what the tests and the bench pass when they switch it on.
"""
import os

import numpy as np
import pytest

import oracle as O

GOLDEN = os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                      "paper_hyperparameters.txt")


def _entries():
    out = []
    for line in open(GOLDEN):
        line = line.split("#", 1)[0] if line.lstrip().startswith("#") else line
        if not line.strip():
            continue
        head, cite = line.split("|", 1)
        tok = head.split()
        assert cite.strip(), tok                      # every value carries its citation
        vals = [float(v) for v in tok[1].split(",")]
        out.append((tok[0], vals, len(tok) > 2 and tok[2] == "switch"))
    return out


ENTRIES = _entries()


@pytest.fixture(scope="module")
def gk():
    from paper_2608_07001_gb300 import build_ext
    build_ext.build()
    from paper_2608_07001_gb300 import gracekv
    return gracekv


def test_every_line_is_read():
    assert len(ENTRIES) == 27
    assert {n for n, _, s in ENTRIES if s} == {"alpha_floor", "lambda_graph"}


@pytest.mark.parametrize("name,vals,switch", ENTRIES, ids=[e[0] for e in ENTRIES])
def test_oracle_defaults_are_the_papers(oracle_lib, name, vals, switch):
    if name == "graph_depths":
        for L in (32, 100, 1000):
            p = O.make_params(L, 1, 1, 64, 8, 2, 0.0, recent=8)
            assert list(O.graph_layers(p)) == [min(int(np.floor(r * L)), L - 1) for r in vals]
        return
    got = O.PAPER_DEFAULTS[name]
    want = 0.0 if switch else (vals if len(vals) > 1 else vals[0])
    assert np.allclose(got, want, rtol=0, atol=0), (name, got, want)


@pytest.mark.parametrize("name,vals,switch", ENTRIES, ids=[e[0] for e in ENTRIES])
def test_library_defaults_are_the_papers(gk, name, vals, switch):
    if name == "graph_depths":
        for L in (32, 100, 1000):
            assert gk.gracekv_graph_layers(L) == [min(int(np.floor(r * L)), L - 1) for r in vals]
        return
    p = gk.gracekv_default_params()
    if name == "windows":
        got = list(p.windows)[:p.n_windows]
    else:
        got = getattr(p, name)
    want = 0.0 if switch else (vals if len(vals) > 1 else vals[0])
    assert np.allclose(got, want, rtol=0, atol=0), (name, got, want)
