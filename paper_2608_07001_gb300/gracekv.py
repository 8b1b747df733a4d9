"""Python binding of the GraceKV compression library (include/gracekv.h).

Argument marshalling only: every step of the compression pass runs in the
CUDA kernels of libgracekv.so.  Tensors are torch CUDA tensors (device
memory); calls are enqueued on the current torch stream.  There is no CPU
fallback: importing this module fails if the library is missing.
"""
from __future__ import annotations

import ctypes as C
import dataclasses
import os
from typing import Optional

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIBPATH = os.path.join(_HERE, "libgracekv.so")

GKV_OK, GKV_EINVAL, GKV_EBUDGET, GKV_ENOMEM, GKV_ECUDA, GKV_ETIMEOUT = 0, 1, 2, 3, 4, 5
GKV_ENONFINITE, GKV_ESTATE, GKV_EUNSUPPORTED, GKV_ECAPACITY = 6, 7, 8, 9
GKV_F32, GKV_BF16 = 0, 1


class GkvParams(C.Structure):
    _fields_ = [
        ("L", C.c_int32), ("G", C.c_int32), ("Hq", C.c_int32), ("T", C.c_int32),
        ("d", C.c_int32), ("W", C.c_int32), ("dtype", C.c_int32),
        ("ctx_start", C.c_int32), ("ctx_end", C.c_int32), ("recent", C.c_int32),
        ("budget", C.c_int64), ("rope_base", C.c_double),
        ("n_min", C.c_int32), ("n_max", C.c_int32), ("n0", C.c_int32),
        ("lambda_stab", C.c_double), ("lambda_s", C.c_double), ("lambda_d", C.c_double),
        ("lambda_n", C.c_double), ("c_cut", C.c_double),
        ("seg_layers", C.c_int32 * 8), ("n_seg_layers", C.c_int32),
        ("windows", C.c_int32 * 4), ("n_windows", C.c_int32),
        ("k_cand", C.c_int32),
        ("lambda_kappa", C.c_double), ("lambda_Z", C.c_double), ("lambda_M", C.c_double),
        ("eps", C.c_double), ("base_frac", C.c_double),
        ("lambda_graph", C.c_double), ("alpha_floor", C.c_double),
        ("seg_mode", C.c_int32), ("quota_alloc", C.c_int32),
        ("floor_c", C.c_double), ("floor_gamma", C.c_double), ("floor_eta", C.c_double),
        ("floor_half", C.c_int32),
        ("eta_seed", C.c_double), ("rho_hop", C.c_double), ("m_seed", C.c_int32), ("r_hop", C.c_int32),
        ("dp_warmup", C.c_int32),
    ]


class GkvDecodeCache(C.Structure):
    _fields_ = [
        ("L", C.c_int32), ("G", C.c_int32), ("Hq", C.c_int32), ("d", C.c_int32),
        ("dtype", C.c_int32), ("K", C.c_void_p), ("V", C.c_void_p), ("log_m", C.c_void_p),
        ("offsets", C.c_void_p), ("n_entries", C.c_int64), ("K_app", C.c_void_p),
        ("V_app", C.c_void_p), ("app_cap", C.c_int32),
    ]


class GraceKVError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"gracekv status {status}: {msg}")
        self.status = status


_lib = None

EXPORTED = ["gracekv_default_params", "gracekv_budget_for_ratio", "gracekv_graph_layers",
            "gracekv_create",
            "gracekv_destroy", "gracekv_last_error", "gracekv_status_string", "gracekv_query",
            "gracekv_segment", "gracekv_score", "gracekv_build_trees", "gracekv_allocate", "gracekv_gather",
            "gracekv_export", "gracekv_profile", "gracekv_stats", "gracekv_row_stats_noalloc",
            "gracekv_compress_host", "gracekv_export_floor", "gracekv_head_sensitivity",
            "gracekv_set_graph_queries", "gracekv_decode_workspace_size", "gracekv_decode_append",
            "gracekv_decode_attention", "gracekv_decode_status"]


def lib() -> C.CDLL:
    """Load libgracekv.so (built by __graft_entry__.build()); raises if absent."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIBPATH):
        raise ImportError(f"{LIBPATH} is missing: build it with __graft_entry__.build()")
    L = C.CDLL(LIBPATH)
    vp, i32, i64 = C.c_void_p, C.c_int32, C.c_int64
    L.gracekv_default_params.argtypes = [C.POINTER(GkvParams)]
    L.gracekv_budget_for_ratio.argtypes = [i32, i32, i32, C.c_double]
    L.gracekv_budget_for_ratio.restype = i64
    L.gracekv_graph_layers.argtypes = [i32, C.POINTER(i32)]
    L.gracekv_graph_layers.restype = i32
    L.gracekv_create.argtypes = [C.POINTER(GkvParams), C.POINTER(vp)]
    L.gracekv_destroy.argtypes = [vp]
    L.gracekv_destroy.restype = None
    L.gracekv_last_error.argtypes = [vp]
    L.gracekv_last_error.restype = C.c_char_p
    L.gracekv_status_string.argtypes = [C.c_int]
    L.gracekv_status_string.restype = C.c_char_p
    L.gracekv_query.argtypes = [vp, C.POINTER(i32), C.POINTER(i32), C.POINTER(i64), C.POINTER(i32)]
    L.gracekv_segment.argtypes = [vp, vp, vp, i32, vp, vp, i32, C.POINTER(i32), vp, vp]
    L.gracekv_build_trees.argtypes = [vp, vp, vp, vp, vp, vp, i32, vp]
    L.gracekv_score.argtypes = [vp, vp, vp, vp]
    L.gracekv_compress_host.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, i64, C.POINTER(i64), vp]
    L.gracekv_allocate.argtypes = [vp, C.POINTER(i64), vp]
    L.gracekv_gather.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp, vp, vp, i64, vp]
    L.gracekv_export.argtypes = [vp, i64, C.POINTER(i64)] + [vp] * 18 + [vp]
    L.gracekv_export_floor.argtypes = [vp, vp, vp, C.POINTER(i64), vp]
    L.gracekv_set_graph_queries.argtypes = [vp, vp, i32]
    L.gracekv_head_sensitivity.argtypes = [vp, vp] + [i32] * 7 + [vp, vp, vp]
    L.gracekv_profile.argtypes = [vp, i32]
    L.gracekv_stats.argtypes = [vp, vp, i32, C.POINTER(i64), vp, i32]
    L.gracekv_row_stats_noalloc.argtypes = [vp, vp] + [i32] * 9 + [vp, vp, vp, vp]
    dcp = C.POINTER(GkvDecodeCache)
    L.gracekv_decode_workspace_size.argtypes = [dcp, C.POINTER(C.c_size_t)]
    L.gracekv_decode_append.argtypes = [dcp, i32, i32, i32, vp, vp, vp]
    L.gracekv_decode_attention.argtypes = [dcp, i32, i32, i32, vp, vp, vp, vp]
    L.gracekv_decode_status.argtypes = [vp, vp]
    _lib = L
    return L


def gracekv_default_params() -> GkvParams:
    p = GkvParams()
    lib().gracekv_default_params(C.byref(p))
    return p


def gracekv_budget_for_ratio(L: int, G: int, n_ctx: int, x: float) -> int:
    return int(lib().gracekv_budget_for_ratio(L, G, n_ctx, float(x)))


def gracekv_graph_layers(L: int) -> list:
    """The multi-hop relevance's graph layers for an L-layer model."""
    out = (C.c_int32 * 2)()
    n = int(lib().gracekv_graph_layers(int(L), out))
    if n < 0:
        _raise(GKV_EINVAL)
    return [int(out[k]) for k in range(n)]


graph_layers = gracekv_graph_layers


def gracekv_row_stats_noalloc(K, Q, c_lo: int, c_hi: int, row_m, row_Z, row_ZC, stream=None):
    """Row statistics without a context and without any device allocation.

    For callers that cannot call cudaMalloc (an engine owning the device's
    memory pool, or a loop that cannot afford an allocation's synchronisation):
    the scratch is a fixed 4 MiB array inside the library.  Outputs are
    caller-provided [L, Hq, W] fp32 CUDA tensors.  Overlapping calls race.
    Every argument is checked here before the library is called (a wrong
    element size or a short output would otherwise become an out-of-bounds
    device access); a mismatch raises GraceKVError(GKV_EINVAL).
    """
    def bad(why):
        return GraceKVError(GKV_EINVAL, "row_stats_noalloc: " + why)

    if K.dim() != 4 or Q.dim() != 4:
        raise bad("K is [L, G, T, d] and Q is [L, Hq, W, d]")
    L, G, T, d = K.shape
    Hq, W = Q.shape[1], Q.shape[2]
    if K.dtype not in (torch.bfloat16, torch.float32):
        raise bad(f"K must be bf16 or fp32, not {K.dtype}")
    if Q.dtype != K.dtype:
        raise bad(f"Q must have K's dtype {K.dtype}, not {Q.dtype}")
    if Q.shape[0] != L or Q.shape[3] != d:
        raise bad(f"Q {tuple(Q.shape)} does not match K {tuple(K.shape)} in L or d")
    for name, o in (("row_m", row_m), ("row_Z", row_Z), ("row_ZC", row_ZC)):
        if o.dtype != torch.float32 or o.numel() < L * Hq * W:
            raise bad(f"{name} must be fp32 with at least L*Hq*W = {L * Hq * W} elements")
        if o.device != K.device:
            raise bad(f"{name} is on {o.device}, K on {K.device}")
    if Q.device != K.device:
        raise bad(f"Q is on {Q.device}, K on {K.device}")
    dt = GKV_BF16 if K.dtype == torch.bfloat16 else GKV_F32
    st = lib().gracekv_row_stats_noalloc(_ptr(K), _ptr(Q), L, G, Hq, T, d, W, dt, c_lo, c_hi,
                                         _ptr(row_m), _ptr(row_Z), _ptr(row_ZC), _stream(stream))
    if st != GKV_OK:
        raise GraceKVError(st, lib().gracekv_status_string(st).decode())


def gracekv_head_sensitivity(W_O, o, G: int, stream=None):
    """omega [L, G] (fp32, device) from W_O [L, D, Hq*d] and o [L, Hq, U, d] (bf16)."""
    L, D, _ = W_O.shape
    _, Hq, U, d = o.shape
    om = torch.empty(L, G, dtype=torch.float32, device=W_O.device)
    scratch = torch.empty(L * G * 65, dtype=torch.float32, device=W_O.device)
    st = lib().gracekv_head_sensitivity(_ptr(W_O), _ptr(o), L, G, Hq, d, D, U, GKV_BF16, _ptr(om),
                                        _ptr(scratch), _stream(stream))
    if st != GKV_OK:
        raise GraceKVError(st, lib().gracekv_status_string(st).decode())
    return om


def _host_ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if t.is_cuda or not t.is_contiguous():
        raise ValueError("tensors must be contiguous host tensors")
    return C.c_void_p(t.data_ptr())


def _ptr(t: Optional[torch.Tensor]):
    if t is None:
        return None
    if not t.is_cuda or not t.is_contiguous():
        raise ValueError("tensors must be contiguous CUDA tensors")
    return C.c_void_p(t.data_ptr())


def _stream(stream=None):
    s = stream if stream is not None else torch.cuda.current_stream()
    return C.c_void_p(s.cuda_stream)


def make_params(L, G, Hq, T, d, W, *, dtype, budget, rope_base, ctx_start=0, ctx_end=None,
                **overrides) -> GkvParams:
    p = gracekv_default_params()
    p.L, p.G, p.Hq, p.T, p.d, p.W = L, G, Hq, T, d, W
    p.dtype = GKV_BF16 if dtype in (torch.bfloat16, "bf16") else GKV_F32
    p.ctx_start = ctx_start
    p.ctx_end = T if ctx_end is None else ctx_end
    p.budget = int(budget)
    p.rope_base = float(rope_base)
    for k, v in overrides.items():
        if k == "windows":
            for i, w in enumerate(v):
                p.windows[i] = w
            p.n_windows = len(v)
        elif k == "seg_layers":
            for i, w in enumerate(v):
                p.seg_layers[i] = w
            p.n_seg_layers = len(v)
        else:
            setattr(p, k, v)
    return p


class Context:
    """Owns a gracekv_ctx; the four stage calls follow the C ABI one to one."""

    def __init__(self, params: GkvParams):
        self.params = params
        h = C.c_void_p()
        st = lib().gracekv_create(C.byref(params), C.byref(h))
        if st != GKV_OK:
            raise GraceKVError(st, lib().gracekv_status_string(st).decode())
        self.h = h
        r, nc, bf, js = C.c_int32(), C.c_int32(), C.c_int64(), C.c_int32()
        lib().gracekv_query(self.h, C.byref(r), C.byref(nc), C.byref(bf), C.byref(js))
        self.recent, self.n_c, self.b_free = r.value, nc.value, bf.value

    def close(self):
        if getattr(self, "h", None):
            lib().gracekv_destroy(self.h)
            self.h = None

    __del__ = close

    def _check(self, st: int):
        if st != GKV_OK:
            msg = lib().gracekv_last_error(self.h).decode()
            raise GraceKVError(st, msg or lib().gracekv_status_string(st).decode())

    def gracekv_segment(self, V, slot_starts, hidden=None, surprisal=None, kappa=None, stream=None) -> int:
        n = C.c_int32()
        Dh = 0 if hidden is None else hidden.shape[-1]
        self._check(lib().gracekv_segment(self.h, _ptr(V), _ptr(hidden), Dh, _ptr(surprisal),
                                          _ptr(slot_starts), slot_starts.numel() - 1, C.byref(n),
                                          _ptr(kappa), _stream(stream)))
        return n.value

    def gracekv_compress_host(self, K, V, Q, out: "Cache", omega=None, stream=None) -> int:
        """The whole pass from host tensors (pinned for the full copy rate)
        into the host cache `out`; returns the number of entries."""
        n = C.c_int64()
        hp = [_host_ptr(t) for t in (K, V, Q, omega, out.K, out.V, out.pos, out.log_m, out.src_lo,
                                     out.src_hi, out.offsets)]
        self._check(lib().gracekv_compress_host(self.h, *hp, out.K.shape[0], C.byref(n), _stream(stream)))
        return n.value

    def gracekv_score(self, K, Q, stream=None):
        self._check(lib().gracekv_score(self.h, _ptr(K), _ptr(Q), _stream(stream)))

    def gracekv_build_trees(self, K, V, Q, omega=None, slot_starts=None, n_slots=0, stream=None):
        self._check(lib().gracekv_build_trees(self.h, _ptr(K), _ptr(V), _ptr(Q), _ptr(omega),
                                              _ptr(slot_starts), n_slots, _stream(stream)))

    def gracekv_allocate(self, stream=None) -> int:
        n = C.c_int64()
        self._check(lib().gracekv_allocate(self.h, C.byref(n), _stream(stream)))
        return n.value

    def gracekv_gather(self, K, V, out: "Cache", stream=None):
        self._check(lib().gracekv_gather(self.h, _ptr(K), _ptr(V), _ptr(out.K), _ptr(out.V),
                                         _ptr(out.pos), _ptr(out.log_m), _ptr(out.src_lo),
                                         _ptr(out.src_hi), _ptr(out.offsets), out.K.shape[0],
                                         _stream(stream)))

    STAGES = ("segment", "row_stats", "token_values", "unit_trees", "allocate", "gather", "floor",
              "multihop")

    def gracekv_set_graph_queries(self, Qg):
        """Qg [n_graph, Hq, T, d] bf16: queries of every position at the graph layers."""
        self._check(lib().gracekv_set_graph_queries(self.h, _ptr(Qg), Qg.shape[0]))
        self._Qg = Qg

    def gracekv_export_floor(self, stream=None) -> dict:
        """The singleton floor of the last tree build (host arrays)."""
        import numpy as np
        p = self.params
        LG = p.L * p.G
        acc = np.zeros((LG, self.n_c), np.uint8)
        f = np.zeros((LG, self.n_c), np.float32)
        bf = C.c_int64()
        self._check(lib().gracekv_export_floor(self.h, C.c_void_p(acc.ctypes.data), C.c_void_p(f.ctypes.data),
                                               C.byref(bf), _stream(stream)))
        return dict(accepted=acc, f=f, B_floor=bf.value)

    def gracekv_profile(self, enable: bool = True):
        self._check(lib().gracekv_profile(self.h, int(enable)))

    def gracekv_stats(self):
        """(per-stage ms since the last call, kernels launched so far, tree work counters)."""
        import numpy as np
        ms = np.zeros(len(self.STAGES), np.float32)
        work = np.zeros(6, np.uint64)
        n = C.c_int64()
        self._check(lib().gracekv_stats(self.h, C.c_void_p(ms.ctypes.data), len(ms), C.byref(n),
                                        C.c_void_p(work.ctypes.data), len(work)))
        names = ("scan_steps", "cand_evals", "cand_len_sum", "units", "dp_chunks", "dp_rerun")
        return dict(zip(self.STAGES, ms.tolist())), n.value, dict(zip(names, map(int, work)))

    def gracekv_export(self, node_cap: Optional[int] = None, stream=None) -> dict:
        """Host copy of the trees and selection (introspection for tests)."""
        import numpy as np
        p = self.params
        js = C.c_int32()
        lib().gracekv_query(self.h, None, None, None, C.byref(js))
        J = js.value
        nu = p.L * p.G * J
        cap = node_cap or p.L * p.G * 2 * self.n_c
        nrow = p.L * p.Hq * p.W
        arr = dict(unit_first=np.zeros(nu + 1, np.int64), unit_Uadd=np.zeros(nu, np.float32),
                   unit_Ddrop=np.zeros(nu, np.float32), add_sel=np.zeros(nu, np.uint8),
                   a=np.zeros(cap, np.int32), b=np.zeros(cap, np.int32),
                   child0=np.zeros(cap, np.int32), nchild=np.zeros(cap, np.int32),
                   cost=np.zeros(cap, np.int32), D=np.zeros(cap, np.float32),
                   R=np.zeros(cap, np.float32), U=np.zeros(cap, np.float32),
                   kappa=np.zeros(cap, np.float32), split_sel=np.zeros(cap, np.uint8),
                   row_m=np.zeros(nrow, np.float32), row_Z=np.zeros(nrow, np.float32),
                   row_ZC=np.zeros(nrow, np.float32), rtok=np.zeros(p.L * p.G * self.n_c, np.float32))
        order = ["unit_first", "unit_Uadd", "unit_Ddrop", "add_sel", "a", "b", "child0", "nchild",
                 "cost", "D", "R", "U", "kappa", "split_sel", "row_m", "row_Z", "row_ZC", "rtok"]
        nn = C.c_int64()
        self._check(lib().gracekv_export(self.h, cap, C.byref(nn),
                                         *[C.c_void_p(arr[k].ctypes.data) for k in order],
                                         _stream(stream)))
        n = nn.value
        for k in ["a", "b", "child0", "nchild", "cost", "D", "R", "U", "kappa", "split_sel"]:
            arr[k] = arr[k][:n]
        arr["J"] = J
        return arr


@dataclasses.dataclass
class Cache:
    """Ragged compressed cache (device tensors, capacity rows)."""
    K: torch.Tensor
    V: torch.Tensor
    pos: torch.Tensor
    log_m: torch.Tensor
    src_lo: torch.Tensor
    src_hi: torch.Tensor
    offsets: torch.Tensor

    @staticmethod
    def empty_host(cap: int, d: int, LG: int, dtype) -> "Cache":
        """Page-locked host arrays (the output of gracekv_compress_host)."""
        c = Cache.empty(cap, d, LG, dtype, device="cpu")
        return Cache(*(t.pin_memory() for t in (c.K, c.V, c.pos, c.log_m, c.src_lo, c.src_hi, c.offsets)))

    @staticmethod
    def empty(cap: int, d: int, LG: int, dtype, device="cuda") -> "Cache":
        i32 = dict(dtype=torch.int32, device=device)
        return Cache(torch.empty(cap, d, dtype=dtype, device=device),
                     torch.empty(cap, d, dtype=dtype, device=device),
                     torch.empty(cap, **i32), torch.empty(cap, dtype=torch.float32, device=device),
                     torch.empty(cap, **i32), torch.empty(cap, **i32),
                     torch.empty(LG + 1, dtype=torch.int64, device=device))


class Compressor:
    """Runs the four stages on one context with preallocated outputs."""

    def __init__(self, params: GkvParams, device="cuda"):
        self.ctx = Context(params)
        p = params
        self.params = p
        dt = torch.bfloat16 if p.dtype == GKV_BF16 else torch.float32
        self.slots = torch.empty(self.ctx.n_c + 2, dtype=torch.int32, device=device)
        self.kappa = torch.empty(p.T, dtype=torch.float32, device=device)
        cap = p.budget + p.L * p.G * (p.T - (p.ctx_end - p.ctx_start)) + 8
        self.cache = Cache.empty(cap, p.d, p.L * p.G, dt, device)
        self.n_slots = 0
        self.n_entries = 0
        self._side = None

    def __call__(self, K, V, Q, omega=None, hidden=None, surprisal=None, slot_starts=None,
                 stream=None, Qg=None) -> "Cache":
        c = self.ctx
        if Qg is not None:          # multi-hop relevance: the graph layers' queries
            c.gracekv_set_graph_queries(Qg)
        # the score passes (K, Q only) run on a second stream while the
        # segmentation runs; the tree build waits for them
        main = stream if stream is not None else torch.cuda.current_stream()
        if self._side is None:
            self._side = torch.cuda.Stream(device=K.device)
        self._side.wait_stream(main)
        c.gracekv_score(K, Q, self._side)
        K.record_stream(self._side)
        Q.record_stream(self._side)
        self.n_slots = c.gracekv_segment(V, self.slots, hidden, surprisal, self.kappa, main)
        if slot_starts is not None:
            c.gracekv_build_trees(K, V, Q, omega, slot_starts, slot_starts.numel() - 1, stream)
        else:
            c.gracekv_build_trees(K, V, Q, omega, None, 0, stream)
        self.n_entries = c.gracekv_allocate(stream)
        c.gracekv_gather(K, V, self.cache, stream)
        return self.cache


def _raise(st: int):
    if st != GKV_OK:
        raise GraceKVError(st, lib().gracekv_status_string(st).decode())


class Decoder:
    """Decoding attention on a packed cache (gracekv_decode_* of the C ABI).

    K, V [E, d], log_m [E] fp32 and offsets [L*G + 1] int64 are the device
    outputs of gracekv_gather (or any cache in that layout); the append area
    [L, G, app_cap, d] and the workspace are allocated here.  ``n_app`` counts
    the appended rows; ``append`` adds one row to every (l, g) of the layers
    it is given and ``attention`` reads the packed entries plus the first
    ``n_app`` appended rows.
    """

    def __init__(self, K, V, log_m, offsets, *, L: int, G: int, Hq: int, app_cap: int = 0):
        d = K.shape[1]
        if K.numel() == 0:              # no packed entry at all: pass a valid address
            K = V = torch.zeros(1, d, dtype=K.dtype, device=K.device)
            log_m = torch.zeros(1, dtype=torch.float32, device=K.device)
        self.dtype = K.dtype
        dt = GKV_BF16 if K.dtype == torch.bfloat16 else GKV_F32
        self.K_app = torch.empty(L, G, max(app_cap, 1), d, dtype=K.dtype, device=K.device)
        self.V_app = torch.empty_like(self.K_app)
        self._keep = (K, V, log_m, offsets)
        ptr = lambda t: _ptr(t).value
        self.desc = GkvDecodeCache(L, G, Hq, d, dt, ptr(K), ptr(V), ptr(log_m), ptr(offsets),
                                   K.shape[0], ptr(self.K_app), ptr(self.V_app), app_cap)
        n = C.c_size_t()
        _raise(lib().gracekv_decode_workspace_size(C.byref(self.desc), C.byref(n)))
        self.workspace = torch.zeros(n.value, dtype=torch.uint8, device=K.device)
        self.L, self.G, self.Hq, self.d = L, G, Hq, d
        self.n_app = 0

    def append(self, k_new, v_new, l0: int = 0, stream=None):
        """k_new, v_new [n_layers, G, d]: row n_app of layers l0.. (n_app is
        advanced when the call covers the last layer)."""
        nl = k_new.shape[0]
        _raise(lib().gracekv_decode_append(C.byref(self.desc), l0, nl, self.n_app, _ptr(k_new),
                                           _ptr(v_new), _stream(stream)))
        if l0 + nl == self.L:
            self.n_app += 1

    def attention(self, q, l0: int = 0, out=None, stream=None):
        """q [n_layers, Hq, d] -> out [n_layers, Hq, d] fp32."""
        nl = q.shape[0]
        if out is None:
            out = torch.empty(nl, self.Hq, self.d, dtype=torch.float32, device=q.device)
        _raise(lib().gracekv_decode_attention(C.byref(self.desc), l0, nl, self.n_app, _ptr(q),
                                              _ptr(out), _ptr(self.workspace), _stream(stream)))
        return out

    def status(self, stream=None):
        _raise(lib().gracekv_decode_status(_ptr(self.workspace), _stream(stream)))
