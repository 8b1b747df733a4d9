#!/usr/bin/env python3
"""Benchmark of the GraceKV compression pass on GB300.

One step = the whole pass (segment, build trees, allocate, gather) over one
synthetic request of the workload, inputs resident in HBM.  Default workload:
Llama-3-8B-shaped cache, 32 layers x 8 KV heads x 128K tokens x d 128, bf16,
64 observation queries, 32x compression (B_total = L G T / 32).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload NAME] [--ratio X] [--no-e2e]

Under torchrun each rank compresses its own request on its own GPU (independent
requests, no collective): value = requests x T tokens / max-over-ranks time.
--impl reference times the CPU oracle (the paper's definitions in plain C,
single thread) on a bounded sample of the same workload and extrapolates its
tokens/s linearly in L*G*T.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np
import torch

METRIC = "context tokens compressed/sec per GB300 and % of HBM roofline (vs CPU oracle)"
PEAK_FALLBACK = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                 "sm_max_mhz": 2070.0}
FP32_LANES = 128
# DRAM bytes of one compression in the dominant stage, from an ncu capture
# (profiles/unit_build_llama128k_2layers_32x.md: the 2-layer slice's 2.29 GB
# scaled by 16 to 32 layers); reported only for the workload it was taken on
STAGE_TRAFFIC = {("unit_trees", "llama128k@32x"): (36.62e9, "ncu dram bytes of every unit_build launch "
                                                           "of one compression on the 2-layer slice x 16")}


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d, "measured"
    return PEAK_FALLBACK, "fallback"


class ClockSampler:
    """nvidia-smi clock/throttle sampling during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu: int):
        self.gpu = gpu
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.t = threading.Thread(target=self._read, daemon=True)
            self.t.start()
        except (OSError, FileNotFoundError):
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def stop(self):
        if not self.proc:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for ln in self.lines:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


def _oracle_sample(args):
    """Child process: the oracle pass on the bounded sample, pinned to one
    host core when the platform allows it; returns (seconds, cores, cpu)."""
    wname, ratio, T_s = args
    cores = None
    try:
        allowed = sorted(os.sched_getaffinity(0))
        os.sched_setaffinity(0, {allowed[0]})
        cores = len(os.sched_getaffinity(0))
    except (AttributeError, OSError):
        pass
    import oracle as O
    from paper_2608_07001_gb300 import synth
    w = synth.WORKLOADS[wname]
    x = synth.make_inputs(w, layers=[0], heads=[0], T=T_s)
    L1, G1, T1, d = x.K.shape
    B = max(int(L1 * G1 * T1 // ratio), 4 * L1 * G1 + 1)
    slots = None if x.slots is None else x.slots
    t0 = time.perf_counter()
    O.run(x.K, x.V, x.Q, B, w.rope_base, slot_starts=slots)
    return time.perf_counter() - t0, cores


def host_info():
    """nproc and the CPU model of the host the oracle runs on."""
    model = None
    try:
        for ln in open("/proc/cpuinfo"):
            k = ln.split(":")[0].strip().lower()
            if k in ("model name", "cpu model", "hardware"):
                model = ln.split(":", 1)[1].strip()
                break
    except OSError:
        pass
    if model is None:
        try:
            out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
            for ln in out.splitlines():
                if ln.lower().startswith("model name"):
                    model = ln.split(":", 1)[1].strip()
                    break
        except (OSError, subprocess.SubprocessError):
            pass
    return {"nproc": os.cpu_count(), "cpu_model": model}


REF_TOKENS = 4096


def cpu_baseline(w, ratio: float, T_s: int = REF_TOKENS):
    """The oracle as it stands on one layer x one KV head x T_s tokens of the
    workload's recipe (for a workload with supplied slots, the recipe's slots
    of that length), in a spawned child pinned to one host core: about 10 s
    of CPU work.  Its tokens/s is extrapolated linearly in L G T."""
    import multiprocessing as mp
    with mp.get_context("spawn").Pool(1) as pool:
        dt, cores = pool.apply(_oracle_sample, ((w.name, ratio, T_s),))
    value = T_s / (dt * w.L * w.G)
    sample = (f"oracle pipeline (segmentation, row statistics, token values, trees, heap "
              f"allocation, gather) on 1 layer x 1 KV head x {T_s} tokens ({dt:.1f} s on one "
              f"host core), extrapolated linearly to {w.L} x {w.G} x {w.T}")
    return value, dt, sample, (cores or 1)


def max_over_ranks(x: float, dist, device) -> float:
    """The largest x over the ranks of the process group (x itself when dist
    is None): the job's time is its slowest rank's."""
    if dist is None:
        return float(x)
    t = torch.tensor([float(x)], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_rate(world: int, tokens: int, steps: int, seconds: float) -> float:
    """Context tokens/s of the whole job: every rank compresses its own
    request of `tokens` tokens per step."""
    return world * tokens * steps / seconds


def run_reference(args, w):
    """Reference arm: the CPU oracle, timed on the host cores."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    vals = []
    for i in range(args.warmup + args.steps):
        v, dt, sample, cores = cpu_baseline(w, args.ratio, T_s=args.ref_tokens)
        if i >= args.warmup:
            vals.append((v, dt))
    value = statistics.median(v for v, _ in vals)
    ms = statistics.median(dt for _, dt in vals) * 1e3 * (w.L * w.G * w.T / args.ref_tokens)
    out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
           "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference",
           "config": workload_config(w, args.ratio),
           "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                            "sample": sample, **host_info()},
           "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out))


def workload_config(w, ratio, L=None):
    L = w.L if L is None else L
    name = w.name if L == w.L else f"{w.name}[{L} layers]"
    return {"workload": f"{name}@{int(ratio)}x", "L": L, "G": w.G, "Hq": w.Hq, "d": w.d,
            "T": w.T, "W": w.W, "ratio": ratio, "dtype": w.dtype,
            "l2": "inputs larger than L2 (no flush needed)"}


def decode_leg(args, w, comp, L, G, Hq, d, dev):
    """Decoding on the cache the pass just wrote (Eq. app_decode_logit).

    One decode step of one token: for every layer, the new token's K/V is
    appended to its (l, g) (multiplicity 1) and the attention of the Hq query
    heads runs over the packed entries plus the appended rows.  Timed two
    ways, CUDA events on the launching stream, after warm-up:
      * all_layers: one attention launch over the L layers (the bandwidth
        figure of the kernel; it sets the roofline below),
      * per_layer:  L x (append + attention) launches, replayed from a CUDA
        graph (the per-token cost when the model runs layer by layer).
    The packed cache is larger than L2, so repeated steps read it from HBM.
    """
    from paper_2608_07001_gb300 import gracekv as gk
    c = comp.cache
    E = comp.n_entries
    n_app = args.decode_app
    dec = gk.Decoder(c.K[:max(E, 1)], c.V[:max(E, 1)], c.log_m[:max(E, 1)], c.offsets,
                     L=L, G=G, Hq=Hq, app_cap=n_app + 1)
    gen = torch.Generator(device=dev).manual_seed(7)
    dt = c.K.dtype
    dec.K_app.copy_(torch.randn(dec.K_app.shape, generator=gen, device=dev).to(dt))
    dec.V_app.copy_(torch.randn(dec.V_app.shape, generator=gen, device=dev).to(dt))
    q = torch.randn(L, Hq, d, generator=gen, device=dev).to(dt)
    k_new = torch.randn(L, G, d, generator=gen, device=dev).to(dt)
    v_new = torch.randn(L, G, d, generator=gen, device=dev).to(dt)
    out = torch.empty(L, Hq, d, device=dev, dtype=torch.float32)
    qs = [q[l:l + 1] for l in range(L)]
    ks = [k_new[l:l + 1] for l in range(L)]
    vs = [v_new[l:l + 1] for l in range(L)]
    outs = [out[l:l + 1] for l in range(L)]

    def step_all():
        dec.n_app = n_app
        dec.append(k_new, v_new)                      # row n_app of every (l, g); n_app + 1 rows
        dec.attention(q, out=out)

    def step_layers():
        for l in range(L):
            dec.n_app = n_app
            dec.append(ks[l], vs[l], l0=l)
            dec.n_app = n_app + 1
            dec.attention(qs[l], l0=l, out=outs[l])

    s = torch.cuda.current_stream(dev)
    for _ in range(max(args.warmup, 3)):
        step_all()
        step_layers()
    torch.cuda.synchronize(dev)
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        step_layers()
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize(dev)
    reps = 50
    e = [torch.cuda.Event(enable_timing=True) for _ in range(6)]
    e[0].record(s)
    for _ in range(reps):
        dec.attention(q, out=out)                    # the attention kernel alone
    e[1].record(s)
    for _ in range(reps):
        step_all()
    e[2].record(s)
    for _ in range(reps):
        g.replay()
    e[3].record(s)
    torch.cuda.synchronize(dev)
    dec.status()
    t_kern = e[0].elapsed_time(e[1]) / reps
    t_all = e[1].elapsed_time(e[2]) / reps
    t_layers = e[2].elapsed_time(e[3]) / reps
    elem = c.K.element_size()
    rows = E + L * G * (n_app + 1)
    # algorithmic bytes of one attention launch over all layers: every packed
    # entry (K row, V row, log m), every appended row (K, V), the offsets,
    # the queries and the fp32 outputs
    byt = (E * (2 * d * elem + 4) + L * G * (n_app + 1) * 2 * d * elem + (L * G + 1) * 8
           + L * Hq * d * (elem + 4))
    pk, pk_kind = peaks()
    ach = byt / (t_kern / 1e3) / 1e9
    return {"workload": f"decode step on the {w.name}@{int(args.ratio)}x packed cache "
                        f"({E} entries) + {n_app + 1} appended rows per (l, g)",
            "entries_read": rows, "bytes_per_launch": byt,
            "us_attention_all_layers": t_kern * 1e3,
            "us_per_token_all_layers": t_all * 1e3,
            "us_per_token_per_layer_graph": t_layers * 1e3,
            "tokens_per_s_per_layer_graph": 1e3 / t_layers,
            "roofline": {"kernel": "decode_tc_kernel", "bound": "hbm", "achieved": ach,
                         "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": ach / pk["hbm_gbs"],
                         "peak_kind": pk_kind, "traffic": None}}


def sensitivity_leg(args, w, D=4096, U=32):
    """omega (Eq. app_head_sensitivity) from a synthetic output projection
    W_O [L, D, Hq d] and head outputs o [L, Hq, U, d] of the workload's shape;
    the pass reads W_O once, so its bytes set the roofline."""
    from paper_2608_07001_gb300 import gracekv as gk
    dev = torch.device("cuda")
    gen = torch.Generator(device=dev).manual_seed(11)
    W = (torch.randn(w.L, D, w.Hq * w.d, generator=gen, device=dev) / w.d ** 0.5).to(torch.bfloat16)
    o = torch.randn(w.L, w.Hq, U, w.d, generator=gen, device=dev).to(torch.bfloat16)
    for _ in range(3):
        gk.gracekv_head_sensitivity(W, o, w.G)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    reps = 20
    e0.record()
    for _ in range(reps):
        gk.gracekv_head_sensitivity(W, o, w.G)
    e1.record()
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    byt = W.numel() * 2 + o.numel() * 2
    pk, pk_kind = peaks()
    ach = byt / (ms / 1e3) / 1e9
    return {"shape": f"L {w.L}, Hq {w.Hq}, d {w.d}, D {D}, U {U}", "ms": ms, "bytes": byt,
            "roofline": {"kernel": "sens_tile_kernel", "bound": "hbm", "achieved": ach,
                         "peak": pk["hbm_gbs"], "unit": "GB/s", "frac": ach / pk["hbm_gbs"],
                         "peak_kind": pk_kind, "traffic": None}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="llama128k")
    ap.add_argument("--ratio", type=float, default=32.0)
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--ref-tokens", type=int, default=REF_TOKENS,
                    help="tokens of the oracle's bounded sample (cpu_baseline and --impl reference)")
    ap.add_argument("--layers", type=int, default=0,
                    help="compress only the first N layers (small cases for profiler captures)")
    ap.add_argument("--no-decode", action="store_true",
                    help="skip the decoding-attention leg on the compressed cache")
    ap.add_argument("--decode-only", action="store_true",
                    help="compress once, then time only the decoding attention")
    ap.add_argument("--decode-app", type=int, default=64,
                    help="tokens already appended to every (l, g) when decoding is timed")
    ap.add_argument("--sensitivity-only", action="store_true",
                    help="time only the layer-KV-head sensitivity on the workload's shape")
    ap.add_argument("--alpha-floor", type=float, default=None,
                    help="singleton-floor cap alpha (the library default when omitted)")
    ap.add_argument("--lambda-graph", type=float, default=0.0,
                    help="multi-hop relevance weight lambda (0: the four-stage pass alone); "
                         "graph-layer queries are synthesised on the device, and the "
                         "host-buffer pass, which takes no graph queries, is not timed")
    ap.add_argument("--ablation", default="none", choices=["none", "wo_cs", "wo_ga"],
                    help="the paper's w/o CS (uniform slots, midpoint cuts) or w/o GA "
                         "(fixed per-(l, g) capacity) variant")
    args = ap.parse_args()

    from paper_2608_07001_gb300 import synth
    w = synth.WORKLOADS[args.workload]
    if args.sensitivity_only:
        print(json.dumps({"head_sensitivity": sensitivity_leg(args, w)}))
        return
    if args.impl == "reference":
        run_reference(args, w)
        return

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    from paper_2608_07001_gb300 import gracekv as gk
    dev = torch.device("cuda", local)
    layers = list(range(args.layers)) if args.layers > 0 else None
    x = synth.make_inputs(w, device=dev, layers=layers)
    K, V, Q = x.K, x.V, x.Q
    L, G, T, d = K.shape
    n_sms = torch.cuda.get_device_properties(dev).multi_processor_count
    # a workload with a supplied partition (the skewed one) passes its slots
    slots = None if x.slots is None else torch.as_tensor(x.slots, dtype=torch.int32, device=dev)
    B = gk.gracekv_budget_for_ratio(L, G, T, args.ratio)
    abl = {"none": {}, "wo_cs": dict(seg_mode=1, k_cand=0, lambda_kappa=0.0),
           "wo_ga": dict(quota_alloc=1)}[args.ablation]
    if args.alpha_floor is not None:
        abl = dict(abl, alpha_floor=args.alpha_floor)
    Qg = None
    if args.lambda_graph > 0:
        abl = dict(abl, lambda_graph=args.lambda_graph)
        args.no_e2e = True
        Qg = synth.make_graph_queries(w, gk.graph_layers(K.shape[0]), device=dev)
    p = gk.make_params(L, G, Q.shape[1], T, d, Q.shape[2], dtype=K.dtype, budget=B,
                       rope_base=w.rope_base, **abl)
    comp = gk.Compressor(p, device=dev)
    stream = torch.cuda.current_stream(dev)

    def barrier():
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize(dev)

    if args.decode_only:
        comp(K, V, Q, Qg=Qg, slot_starts=slots)
        torch.cuda.synchronize(dev)
        dec = decode_leg(args, w, comp, L, G, Q.shape[1], d, dev)
        if rank == 0:
            print(json.dumps({"decode": dec}))
        return

    for _ in range(args.warmup):
        comp(K, V, Q, Qg=Qg, slot_starts=slots)
    comp.ctx.gracekv_profile(True)
    comp.ctx.gracekv_stats()
    _, launches0, _ = comp.ctx.gracekv_stats()
    barrier()
    clk = ClockSampler(local)
    clk.start()
    time.sleep(0.3)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        comp(K, V, Q, Qg=Qg, slot_starts=slots)
    e1.record(stream)
    barrier()
    clocks = clk.stop()
    ms_total = e0.elapsed_time(e1)
    stage_ms, launches1, work = comp.ctx.gracekv_stats()
    comp.ctx.gracekv_profile(False)
    ms_total = max_over_ranks(ms_total, dist, dev)
    ms_step = ms_total / args.steps
    value = whole_job_rate(world, T, args.steps, ms_total / 1e3)
    E = comp.n_entries

    # ---- roofline ----------------------------------------------------------------
    pk, pk_kind = peaks()
    elem = 2 if K.dtype == torch.bfloat16 else 4
    floor_bytes = L * G * T * 2 * d * elem + E * (2 * d * elem + 16)
    hbm = {"floor_bytes": floor_bytes, "achieved_gbs": floor_bytes / (ms_step / 1e3) / 1e9,
           "peak_gbs": pk["hbm_gbs"], "peak_kind": pk_kind}
    hbm["frac"] = hbm["achieved_gbs"] / hbm["peak_gbs"]
    per_step = {k: v / args.steps for k, v in stage_ms.items()}
    dom = max(per_step, key=per_step.get)
    Wp = Q.shape[2]
    if dom == "unit_trees":
        # probe scans (W*d FMA per token step), candidate evaluation (logit,
        # residual and ||M||^2: 4 W d FMA), prototype sums (3 d per token),
        # probe weights of every token (W d FMA)
        flops = (2 * Wp * d * work["scan_steps"] + 8 * Wp * d * work["cand_evals"]
                 + 6 * d * work["cand_len_sum"] + 2 * Wp * d * L * G * comp.ctx.n_c)
        peak = n_sms * FP32_LANES * 2 * pk.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        ach = flops / (per_step[dom] / 1e3) / 1e12
        tr = STAGE_TRAFFIC.get((dom, workload_config(w, args.ratio, L)["workload"]))
        roof = {"kernel": "unit_build_kernel", "bound": "alu", "achieved": ach, "peak": peak,
                "unit": "TFLOP/s", "frac": ach / peak, "traffic": None if tr is None else tr[0],
                "peak_basis": f"{n_sms} SMs x {FP32_LANES} fp32 lanes x 2 x max SM clock"}
        if tr is not None:
            roof["traffic_basis"] = tr[1]
    elif dom in ("row_stats", "token_values"):
        flops = 2 * L * Q.shape[1] * Wp * d * (T if dom == "row_stats" else comp.ctx.n_c)
        peak = n_sms * FP32_LANES * 2 * pk.get("sm_max_mhz", 2070.0) * 1e6 / 1e12
        ach = flops / (per_step[dom] / 1e3) / 1e12
        roof = {"kernel": dom, "bound": "alu", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
                "frac": ach / peak, "traffic": None}
    else:
        byt = L * G * T * 2 * d * elem if dom == "gather" else floor_bytes
        ach = byt / (per_step[dom] / 1e3) / 1e9
        roof = {"kernel": dom, "bound": "hbm", "achieved": ach, "peak": pk["hbm_gbs"],
                "unit": "GB/s", "frac": ach / pk["hbm_gbs"], "traffic": None}

    # ---- end to end through the C ABI with host buffers ---------------------------
    e2e = None
    if not args.no_e2e:
        Kh = torch.empty_like(K, device="cpu").pin_memory()
        Vh = torch.empty_like(V, device="cpu").pin_memory()
        Qh = torch.empty_like(Q, device="cpu").pin_memory()
        Kh.copy_(K); Vh.copy_(V); Qh.copy_(Q)
        c = comp.cache
        hc = gk.Cache.empty_host(c.K.shape[0], d, L * G, K.dtype)

        if slots is None:
            def e2e_step():
                # the library copies the inputs layer group by layer group on a
                # copy stream and starts each group's work as it lands
                return comp.ctx.gracekv_compress_host(Kh, Vh, Qh, hc)
        else:
            # a supplied partition: the device API with the copies in the
            # step (the host-buffer call segments the context itself)
            Kd, Vd, Qd = torch.empty_like(K), torch.empty_like(V), torch.empty_like(Q)
            sh = x.slots.astype(np.int32)

            def e2e_step():
                Kd.copy_(Kh, non_blocking=True)
                Vd.copy_(Vh, non_blocking=True)
                Qd.copy_(Qh, non_blocking=True)
                sd = torch.from_numpy(sh).to(dev, non_blocking=False)
                cache = comp(Kd, Vd, Qd, slot_starts=sd)
                n = comp.n_entries
                for k_ in ("K", "V", "pos", "log_m", "src_lo", "src_hi"):
                    getattr(hc, k_)[:n].copy_(getattr(cache, k_)[:n], non_blocking=True)
                hc.offsets.copy_(cache.offsets, non_blocking=True)
                torch.cuda.synchronize(dev)
                return n

        e2e_step()
        barrier()
        t0 = time.perf_counter()
        for _ in range(args.e2e_steps):
            n = e2e_step()
        barrier()
        dt = time.perf_counter() - t0
        dt = max_over_ranks(dt, dist, dev)
        h2d = sum(t_.numel() * t_.element_size() for t_ in (K, V, Q)) + (0 if slots is None else slots.numel() * 4)
        d2h = n * (2 * d * elem + 16) + hc.offsets.numel() * 8
        e2e = {"value": whole_job_rate(world, T, args.e2e_steps, dt), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        v, dt, sample, cores = cpu_baseline(w, args.ratio, T_s=args.ref_tokens)
        cpu = {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle", "sample": sample,
               **host_info()}

    dec = None
    if not args.no_decode:
        dec = decode_leg(args, w, comp, L, G, Q.shape[1], d, dev)

    if rank == 0:
        out = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world,
               "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
               "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
               "dtype": "bf16" if K.dtype == torch.bfloat16 else "f32", "data": "synthetic",
               "config": dict(workload_config(w, args.ratio, L), B_total=B, entries=E,
                              slots=comp.n_slots, parallelism=f"replicas{world}",
                              alpha_floor=p.alpha_floor, lambda_graph=p.lambda_graph,
                              **({"ablation": args.ablation} if args.ablation != "none" else {})),
               "roofline": roof, "hbm_pass": hbm, "stages_ms": per_step, "tree_work": work,
               "cpu_baseline": cpu, "e2e": e2e,
               "gpu_launches": launches1 - launches0, "clocks": clocks, "decode": dec}
        print(json.dumps(out))
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
