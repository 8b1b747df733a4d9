"""Trees of slots longer than 128 tokens against the oracle.

A supplied partition may hold slots far longer than the segmentation's 128
tokens (the skewed workload draws 1% of its slots from 4097..8192 tokens and
1% of length 1); their trees still recurse to single-token leaves (App. A.3,
"Recursive refinement rule").  The unit kernel keeps at most 128 tokens in
shared memory, so these units are built level by level across CTAs
(build_long.cu).  The comparison is the test-size one (tests/parity.py):
bit-exact trees, selection, positions and intervals, single tokens
bit-exact, prototypes within the dtype's tolerance, no near-tie exemption.

  long_slots   slots of 1, 2, 16, 40, 70, 100, 129, 4097 and 8192 tokens on a
               small-model head (d 64, 4 query heads x 8 probes): bf16 at 8x
               and 2x (tensor-core score path, probe weights from it), fp32 at
               4x (probe weights formed in the scan), the singleton floor at
               alpha 0.6 (forced extraction inside long nodes), and the
               per-(l, g) capacity ablation (trees built completely)
  skew         one layer x one KV head of the skewed workload (d 128, 4 query
               heads x 64 probes, keys aligned with the queries in three
               512-token regions) at 16384 tokens with its drawn slots, at 4x,
               32x and 128x; the oracle's trees are built once, pooled
"""
import numpy as np
import pytest
import torch

from paper_2608_07001_gb300 import synth
from tests import parity as P
from tests.oracle_pool import run_pooled

pytestmark = pytest.mark.gpu

LENS = [40, 1, 129, 70, 4097, 2, 8192, 16, 100]


@pytest.fixture(scope="module", autouse=True)
def built():
    import __graft_entry__ as g
    g.build()
    assert torch.cuda.is_available()


def _long_inputs(dtype):
    w = synth.WORKLOADS["small"]
    N = sum(LENS)
    x = synth.make_inputs(w, layers=[2], heads=[3], T=N + 32, W=8)
    K, V, Q = x.K, x.V, x.Q
    if dtype == "fp32":
        K, V, Q = K.float(), V.float(), Q.float()
    return w, K, V, Q, np.concatenate([[0], np.cumsum(LENS)]).astype(np.int32)


@pytest.mark.parametrize("dtype,ratio,extra", [
    ("bf16", 8, {}), ("bf16", 2, {}), ("fp32", 4, {}),
    ("bf16", 8, {"alpha_floor": 0.6}), ("bf16", 8, {"quota_alloc": 1}),
])
def test_long_slots_match_the_oracle(dtype, ratio, extra):
    w, K, V, Q, slots = _long_inputs(dtype)
    L, G, T, d = K.shape
    B = (L * G * T) // ratio
    g = P.run_gpu(K, V, Q, B, w.rope_base, slot_starts=slots, **extra)
    o = P.run_oracle(K, V, Q, B, w.rope_base, slot_starts=slots, **extra)
    if "alpha_floor" in extra:
        fl = g["comp"].ctx.gracekv_export_floor()
        np.testing.assert_array_equal(fl["accepted"], o["floor"]["accepted"])
        assert fl["B_floor"] == o["floor"]["B_floor"]
    rep = P.compare(g, o, torch.float32 if dtype == "fp32" else torch.bfloat16)
    # the long slots' units did expand beyond their roots
    ex = g["export"]
    uf = ex["unit_first"]
    for j in (4, 6):                                 # the 4097- and 8192-token slots
        assert uf[j + 1] - uf[j] > 1, j
    print(dtype, ratio, extra, rep)


@pytest.fixture(scope="module")
def skew_case():
    w = synth.WORKLOADS["skew"]
    T = 16384
    x = synth.make_inputs(w, layers=[0], heads=[0], T=T)
    ratios = (4, 32, 128)
    budgets = [T // r for r in ratios]
    oracles = run_pooled(x.K, x.V, x.Q, budgets, w.rope_base, slot_starts=x.slots)
    return w, x, dict(zip(ratios, zip(budgets, oracles)))


@pytest.mark.parametrize("ratio", [4, 32, 128])
def test_skew_slice_matches_the_oracle(skew_case, ratio):
    w, x, cases = skew_case
    B, o = cases[ratio]
    lens = np.diff(x.slots)
    assert (lens > 4096).sum() >= 2 and (lens == 1).sum() >= 1
    g = P.run_gpu(x.K, x.V, x.Q, B, w.rope_base, slot_starts=x.slots)
    rep = P.compare(g, o, torch.bfloat16)
    assert g["E"] == len(o["cache"]["pos"])
    print("skew", ratio, rep)
