"""The segmentation DP's chunked execution against the oracle (through the C ABI).

The device runs the recurrence of App. B.3 Eq. app_dp_recurrence in chunks on
separate CTAs, each started some tokens early from a flat state, and re-runs in
order every chunk whose starting state is not the previous chunk's up to a
constant.  The slots must not depend on that: every warm-up length, including
one so short that most chunks are re-run and the single-chunk sequential run,
gives the oracle's slot starts bit for bit (the oracle is the plain fp64
recurrence from F[0] = 0).  Cases: a structured bf16 trajectory at T = 8192
(16 chunks), an unstructured fp32 one (Gaussian values, no segment structure),
and n_min = 5 / n_max = 40 (steps of 5 endpoints, 160 per chunk, ragged end).
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

import oracle as O
from paper_2608_07001_gb300 import gracekv as gk
from paper_2608_07001_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def _structured():
    w = synth.WORKLOADS["small"]
    inp = synth.make_inputs(w, layers=[5, 8, 10], T=8192)
    return inp.V, dict(Hq=w.Hq, W=w.W, rope=w.rope_base), {}


def _unstructured():
    g = torch.Generator().manual_seed(20260)
    V = torch.randn(1, 2, 6000, 64, generator=g)
    return V, dict(Hq=2, W=8, rope=1e4), {}


def _short_slots():
    w = synth.WORKLOADS["small"]
    inp = synth.make_inputs(w, layers=[3], heads=[0, 1, 2, 3], T=3001)
    return inp.V, dict(Hq=16, W=w.W, rope=w.rope_base), dict(n_min=5, n_max=40, n0=20)


CASES = {"structured": _structured, "unstructured": _unstructured, "short_slots": _short_slots}


def _gpu_slots(V, meta, ov, warmup):
    L, G, T, d = V.shape
    seg = tuple(range(L))
    B = gk.gracekv_budget_for_ratio(L, G, T, 8.0)
    p = gk.make_params(L, G, meta["Hq"], T, d, meta["W"], dtype=V.dtype, budget=B,
                       rope_base=meta["rope"], seg_layers=seg, dp_warmup=warmup, **ov)
    ctx = gk.Context(p)
    buf = torch.empty(ctx.n_c + 2, dtype=torch.int32, device="cuda")
    J = ctx.gracekv_segment(V.cuda().contiguous(), buf)
    torch.cuda.synchronize()
    _, _, work = ctx.gracekv_stats()
    out = buf[:J + 1].cpu().numpy().astype(np.int64)
    recent = ctx.recent
    ctx.close()
    return out, work["dp_chunks"], work["dp_rerun"], recent


@pytest.mark.parametrize("case", list(CASES))
def test_chunked_dp_gives_the_oracle_slots_for_every_warm_up(case):
    V, meta, ov = CASES[case]()
    L, G, T, d = V.shape
    runs = {wu: _gpu_slots(V, meta, ov, wu) for wu in (0, 16, 100, -1)}
    recent = runs[0][3]
    p = O.make_params(L, G, meta["Hq"], T, d, meta["W"], meta["rope"], seg_layers=tuple(range(L)),
                      recent=recent, disp_mode=1, **ov)
    o = O.segment(p, V.double().numpy())
    og = o["slot_starts"].astype(np.int64)
    N = T - recent
    step = min(ov.get("n_min", 16), 16)
    for wu, (gs, chunks, rerun, _) in runs.items():
        print(f"{case}: warm-up {wu}: {chunks} chunks, {rerun} re-run, {len(gs) - 1} slots")
        if not np.array_equal(gs, og):
            # the first endpoint (from N back) whose predecessor differs must be an oracle near-tie
            common = sorted(set(og.tolist()) & set(gs.tolist()))
            for i in reversed(common[1:]):
                po, pg = og[np.searchsorted(og, i) - 1], gs[np.searchsorted(gs, i) - 1]
                if po != pg:
                    m = abs(o["dp_best"][i] - o["dp_second"][i]) / max(abs(o["dp_best"][i]), 1e-300)
                    raise AssertionError(f"warm-up {wu}: slots differ at endpoint {i} (oracle margin {m:.2e})")
            raise AssertionError(f"warm-up {wu}: slots differ")
        if wu < 0:
            assert (chunks, rerun) == (1, 0)
        else:
            assert chunks == -(-N // (32 * step))
            assert 0 <= rerun < chunks
    # a 16-token warm-up is too short for the paths to coalesce: chunks are re-run
    assert runs[16][2] >= 1
