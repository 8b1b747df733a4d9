"""The Python binding moves no computation to the host.

Every entry point that takes device tensors rejects host tensors before the
library sees them, and a missing library is an ImportError: there is no CPU
path to fall back to.  Runs without a GPU.
"""
import pytest
import torch


@pytest.fixture(scope="module")
def gk():
    from paper_2608_07001_gb300 import build_ext
    build_ext.build()
    from paper_2608_07001_gb300 import gracekv
    gracekv.lib()
    return gracekv


def test_missing_library_is_an_import_error(gk, monkeypatch, tmp_path):
    monkeypatch.setattr(gk, "LIBPATH", str(tmp_path / "absent.so"))
    monkeypatch.setattr(gk, "_lib", None)
    with pytest.raises(ImportError):
        gk.lib()
    with pytest.raises(ImportError):
        gk.gracekv_budget_for_ratio(1, 2, 1024, 8.0)


def test_device_entry_points_reject_host_tensors(gk):
    bf = torch.bfloat16
    K = torch.zeros(1, 2, 64, 64, dtype=bf)
    Q = torch.zeros(1, 2, 4, 64, dtype=bf)
    st = torch.zeros(1, 2, 4)
    with pytest.raises(ValueError, match="CUDA"):
        gk.gracekv_row_stats_noalloc(K, Q, 0, 64, st, st, st)
    W = torch.zeros(1, 128, 2 * 64, dtype=bf)
    o = torch.zeros(1, 2, 4, 64, dtype=bf)
    with pytest.raises(ValueError, match="CUDA"):
        gk.gracekv_head_sensitivity(W, o, 2)
    with pytest.raises(ValueError, match="CUDA"):
        gk.Decoder(K[0, 0], K[0, 0], torch.zeros(64), torch.tensor([0, 32, 64]), L=1, G=2, Hq=2)


def test_host_buffer_pass_rejects_device_or_strided_tensors(gk):
    # gracekv_compress_host takes host memory only; a strided view is refused
    # before the call (the library reads plain contiguous arrays)
    x = torch.zeros(4, 4)
    with pytest.raises(ValueError, match="contiguous host"):
        gk._host_ptr(x.t())
    assert gk._host_ptr(None) is None and gk._host_ptr(x).value == x.data_ptr()


def test_noalloc_refuses_mismatched_arguments_before_any_launch(gk):
    # a wrong dtype, a Q of another dtype or shape, or a short or non-fp32
    # output is refused in the binding: none of them reaches the library
    bf = torch.bfloat16
    K = torch.zeros(1, 2, 64, 64, dtype=bf)
    Q = torch.zeros(1, 2, 4, 64, dtype=bf)
    ok = torch.zeros(1, 2, 4)
    cases = [
        (K.half(), Q.half(), ok, "bf16 or fp32"),
        (K, Q.float(), ok, "K's dtype"),
        (K, torch.zeros(2, 2, 4, 64, dtype=bf), ok, "L or d"),
        (K, torch.zeros(1, 2, 4, 32, dtype=bf), ok, "L or d"),
        (K, Q, torch.zeros(7), "at least"),
        (K, Q, torch.zeros(1, 2, 4, dtype=torch.float64), "fp32"),
        (K[0], Q, ok, r"\[L, G, T, d\]"),
    ]
    for k, q, out, why in cases:
        with pytest.raises(gk.GraceKVError, match=why) as e:
            gk.gracekv_row_stats_noalloc(k, q, 0, 64, out, ok, ok)
        assert e.value.status == gk.GKV_EINVAL
