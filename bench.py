#!/usr/bin/env python
"""Benchmark of the OrderMoE MoE-layer hot path on GB300.

One step = one pass of the hot path over one batch: router + softmax + top-k
+ server-expert selection, permutation, grouped SwiGLU expert FFN (gate/up,
down) and weighted combine -- eight kernels of libordermoe.so, nothing else.
Default workload: the Mixtral-8x7B-shaped prefill layer (T = 4096 tokens,
d = 4096, E = 8, top-2, d_ff = 14336, 4 logical servers), synthetic seeded
inputs drawn on the device. The offline plan (similarity, grouping,
placement, tables) runs once through the library before timing.

Prints one JSON line (rank 0). `--impl reference` times the CPU oracle on a
bounded sample of the same workload instead.
"""
import argparse
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "MoE-layer tokens/s on 1 GB300 (route+select+FFN) and % of tensor/HBM roofline"
UNIT = "tokens/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}

# DRAM bytes (read + write) per launch of the gate/up GEMM at the mixtral_prefill workload, from
# the recorded ncu capture of that kernel, valid only while the
# kernel sources hash to the values recorded with it.
GATE_UP_TRAFFIC = {
    "bytes": 1960575488 + 229206784,  # dram__bytes_read.sum + dram__bytes_write.sum, one launch
    "sha256": {"paper_2607_17154_gb300/csrc/grouped_gemm.cu":
               "37d3c35e5807598734e8f1340faa5ee978a2cdf8c753a74a149166cbb1bfcf13",
               "paper_2607_17154_gb300/csrc/common.cuh":
               "f9203679569dac2a7615b946e342f582a518ee0b5532bbda0ead03f68f9af7a9"},
}


def gate_up_traffic(workload):
    """The recorded traffic if the kernel is unchanged since the capture, else None."""
    import hashlib
    if workload != "mixtral_prefill":
        return None
    for rel, digest in GATE_UP_TRAFFIC["sha256"].items():
        with open(os.path.join(ROOT, rel), "rb") as f:
            if hashlib.sha256(f.read()).hexdigest() != digest:
                return None
    return GATE_UP_TRAFFIC["bytes"]


def gate_up_kernel_name(R, E, dff):
    """The gate/up kernel the library picks for R permuted rows (grouped_gemm.cu)."""
    if R < 256 * E:
        return "ffn_gemm_kernel<gate_up> (tcgen05, one CTA, 128-row tiles)"
    return "ffn_gemm_pair_kernel<gate_up> (tcgen05 CTA pairs)"


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=500)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--workload", default="mixtral_prefill")
    p.add_argument("--theta", type=float, default=None,
                   help="similarity threshold theta of the grouping (default: the workload's)")
    p.add_argument("--seed", type=int, default=0)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-extras", action="store_true",
                   help="mixtral_prefill: skip timing the other workloads after the main line")
    p.add_argument("--lookahead", type=int, default=1,
                   help="selection horizon H (Eqs. 41-43) for the decode stack; 1 = myopic")
    p.add_argument("--memory-ratio", type=float, default=None,
                   help="memory budget ratio of the offline plan (Section VI-G): server capacity "
                        "over one copy of the experts; above 1 the spare memory holds replicas "
                        "(Eqs. 32-35). Default: 1.0 for the decode stack, 2.0 for the plan")
    p.add_argument("--eager", action="store_true",
                   help="decode stack: launch every kernel from the host instead of replaying "
                        "each step as one CUDA graph")
    p.add_argument("--n-cal", type=int, default=None,
                   help="calibration tokens of the offline plan (default: the workload's; a "
                        "smaller count makes a short profiling case of the same kernels)")
    p.add_argument("--cpu-seconds", type=float, default=15.0,
                   help="target CPU seconds of the oracle baseline sample")
    return p.parse_args()


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


BURST_REGION_S = 1.0


def tensor_peak(pk, pk_kind, clocks, region_s):
    """The bf16 peak that applies to a kernel timed inside a region of
    region_s seconds: the burst figure (best single cuBLAS GEMM) when the
    region is short (under BURST_REGION_S) and no power cap was active while
    it ran, else the sustained figure (cuBLAS back to back for seconds under
    the power cap). Returns (peak, which, why, burst, sustained)."""
    burst = float(pk.get("bf16_tflops", FALLBACK_PEAKS["bf16_tflops"]))
    sustained = float(pk.get("bf16_tflops_sustained", FALLBACK_PEAKS["bf16_tflops_sustained"]))
    capped = "sw_power_cap" in (clocks or {}).get("reasons", [])
    if region_s < BURST_REGION_S and not capped:
        why = "timed region %.3f s < %.1f s, no power cap seen" % (region_s, BURST_REGION_S)
        return burst, "burst", why, burst, sustained
    why = ("sw_power_cap active during the timed region" if capped else
           "timed region %.3f s >= %.1f s" % (region_s, BURST_REGION_S))
    return sustained, "sustained", why, burst, sustained


def tensor_roofline(kernel, achieved, pk, pk_kind, clocks, region_s, **extra):
    """Roofline object of a tensor-bound kernel, its fraction of both measured
    bf16 peaks, and which one applies."""
    peak, which, why, burst, sustained = tensor_peak(pk, pk_kind, clocks, region_s)
    out = {"kernel": kernel, "bound": "tensor", "achieved": round(achieved, 1), "peak": peak,
           "unit": "TFLOP/s", "frac": round(achieved / peak, 4),
           "frac_burst": round(achieved / burst, 4), "frac_sustained": round(achieved / sustained, 4),
           "peak_applies": which, "peak_reason": why,
           "peak_source": "%s bf16_tflops%s" % (pk_kind, "" if which == "burst" else "_sustained")}
    out.update(extra)
    return out


# ----------------------------------------------------------------- clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, gpu_index):
        self.index = gpu_index
        self.proc = None

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
                 "-lms", "100", "-i", str(self.index)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, smax, reasons = [], [], set()
        for line in out.splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1])); smax.append(float(f[2]))
            except ValueError:
                continue
            for name, v in zip(self.NAMES, f[5:9]):
                if v.lower() == "active":
                    reasons.add(name)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


def gpu_index(local_rank):
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        items = [v.strip() for v in vis.split(",") if v.strip()]
        if local_rank < len(items):
            return items[local_rank]
    return str(local_rank)


# ----------------------------------------------------------------- distributed
class Dist:
    """Replicas only: ranks share nothing on the data path; the process group
    serves the timing barrier and the max-over-ranks reduction."""

    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local_rank = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        if self.world > 1:
            import torch.distributed as dist
            backend = os.environ.get("ORDERMOE_BENCH_BACKEND", "nccl")
            dist.init_process_group(backend=backend)
            self.pg = dist

    def barrier(self, device=None):
        if self.pg is not None:
            if device is not None and self.pg.get_backend() == "nccl":
                self.pg.barrier(device_ids=[device.index])
            else:
                self.pg.barrier()

    def max(self, value, device=None):
        if self.pg is None:
            return value
        import torch
        t = torch.tensor([float(value)], dtype=torch.float64,
                         device=device if self.pg.get_backend() == "nccl" else "cpu")
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg is not None:
            self.pg.destroy_process_group()


# ----------------------------------------------------------------- our arm
def setup_gpu(w, seed, device):
    """Inputs on the device, then the offline plan through the library."""
    import torch
    from paper_2607_17154_gb300 import binding as B
    from paper_2607_17154_gb300 import synth

    inp = synth.layer_inputs(w, seed=seed, device=device)
    home = torch.as_tensor(inp["home"]).to(device)
    Xcal = synth.calibration(w.n_cal, w.d, seed, device=device)
    sim = torch.empty(1, w.E, w.E, dtype=torch.float32, device=device)
    counts = torch.empty(1, w.E, dtype=torch.int32, device=device)
    ws = torch.empty(B.ordermoe_similarity_workspace_bytes(1, w.E, w.n_cal), dtype=torch.uint8,
                     device=device)
    t0 = time.perf_counter()
    B.ordermoe_similarity(inp["Wr"], Xcal, 1, w.E, w.d, w.n_cal, w.k, sim, counts, ws)
    group = torch.empty(1, w.E, dtype=torch.int32, device=device)
    ngroups = torch.empty(1, dtype=torch.int32, device=device)
    theta = torch.empty(1, dtype=torch.float32, device=device)
    placement = torch.empty(1, w.M, w.E, dtype=torch.uint8, device=device)
    used = torch.empty(w.M, dtype=torch.float64, device=device)
    status = torch.empty(1, dtype=torch.int32, device=device)
    p = torch.ones(1, w.E, dtype=torch.float64, device=device)
    C = torch.full((w.M,), w.E / w.M, dtype=torch.float64, device=device)
    B.ordermoe_place(sim, counts, 1, w.E, w.M, w.theta_min, w.theta_max, w.theta, 0.5, 0.5, 0.5,
                     0.5, p, C, group, ngroups, theta, None, placement, used, status)
    sp = synth.server_params(w.M, w.d, w.dff, seed)
    f64 = lambda a: torch.as_tensor(a, dtype=torch.float64).to(device)
    tables = torch.zeros(B.ordermoe_tables_bytes(w.E, w.M), dtype=torch.uint8, device=device)
    B.ordermoe_build_tables(sim[0], group[0], placement[0], w.theta, w.qbar, f64(sp.F), f64(sp.B),
                            f64(sp.tau), sp.z, sp.c, sp.omega_T, sp.omega_Q, tables)
    torch.cuda.synchronize(device)
    plan_ms = (time.perf_counter() - t0) * 1e3
    code, detail = B.ordermoe_device_error()
    if code:
        raise RuntimeError("device error %d (%d) in the offline plan" % (code, detail))
    return inp, home, tables, {"plan_ms": round(plan_ms, 3), "n_groups": int(ngroups.item()),
                               "place_status": int(status.item())}


def run_ours(args, dist):
    import torch
    from paper_2607_17154_gb300 import binding as B
    from paper_2607_17154_gb300 import synth

    device = torch.device("cuda", dist.local_rank)
    torch.cuda.set_device(device)
    B.lib()
    over = {}
    if args.n_cal:
        over["n_cal"] = args.n_cal
    if args.theta is not None:
        over["theta"] = args.theta
    w = synth.workload(args.workload, **over)
    if w.name == "decode_stack":
        return run_decode(args, dist, w, device)
    if w.name == "similarity":
        return run_similarity(args, dist, w, device)
    inp, home, tables, plan = setup_gpu(w, args.seed + 1000 * dist.rank, device)
    T, E, d, k, dff = w.T, w.E, w.d, w.k, w.dff
    R = T * k
    X, Wr, W1, W3, W2 = (inp[n] for n in ("X", "Wr", "W1", "W3", "W2"))
    f = lambda *s, dt: torch.empty(*s, dtype=dt, device=device)
    idx, wts, ch = f(T, k, dt=torch.int32), f(T, k, dt=torch.float32), f(T, k, dt=torch.int32)
    sv, kd = f(T, k, dt=torch.uint8), f(T, k, dt=torch.uint8)
    counters = torch.zeros(4, dtype=torch.int32, device=device)
    offsets, row_token, row_of = f(E + 1, dt=torch.int32), f(R, dt=torch.int32), f(T, k, dt=torch.int32)
    Xp, H, Yp = f(R, d, dt=torch.bfloat16), f(R, dff, dt=torch.bfloat16), f(R, d, dt=torch.bfloat16)
    y = f(T, d, dt=torch.bfloat16)
    ws = f(B.ordermoe_dispatch_workspace_bytes(T, k, E), dt=torch.uint8)
    stream = torch.cuda.current_stream(device)

    def step(ev0=None, ev1=None, cnt=None):
        B.ordermoe_route_select(X, Wr, None, T, E, d, k, 1, tables, home, None, None, None, idx,
                                wts, ch, sv, kd, cnt)
        B.ordermoe_dispatch(ch, X, T, k, E, d, offsets, row_token, row_of, Xp, ws)
        if ev0 is not None:
            ev0.record(stream)
        B.ordermoe_expert_gate_up(Xp, offsets, R, W1, W3, E, d, dff, H)
        if ev1 is not None:
            ev1.record(stream)
        B.ordermoe_expert_down(H, offsets, R, W2, E, d, dff, Yp)
        B.ordermoe_combine(Yp, row_of, wts, T, k, d, y)

    def step_phases():
        return [
            ("route_select", lambda: B.ordermoe_route_select(X, Wr, None, T, E, d, k, 1, tables, home,
                                                              None, None, None, idx, wts, ch, sv, kd,
                                                              None)),
            ("dispatch", lambda: B.ordermoe_dispatch(ch, X, T, k, E, d, offsets, row_token, row_of,
                                                     Xp, ws)),
            ("expert_gate_up", lambda: B.ordermoe_expert_gate_up(Xp, offsets, R, W1, W3, E, d, dff, H)),
            ("expert_down", lambda: B.ordermoe_expert_down(H, offsets, R, W2, E, d, dff, Yp)),
            ("combine", lambda: B.ordermoe_combine(Yp, row_of, wts, T, k, d, y)),
        ]

    # route_select 1 (2 for more than 16 experts: the lane selection kernel),
    # dispatch 4, gate/up 1, down 1, combine 1
    KERNELS_PER_STEP = 8 + (1 if E > 16 else 0)
    step(cnt=counters)     # one counted pass for the execution-type breakdown
    for _ in range(max(args.warmup, 3)):
        step()
    ev0 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    ev1 = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps)]
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(gpu_index(dist.local_rank))
    sampler.start()
    dist.barrier(device)
    torch.cuda.synchronize(device)
    start.record(stream)
    for i in range(args.steps):
        step(ev0[i], ev1[i])
    stop.record(stream)
    torch.cuda.synchronize(device)
    dist.barrier(device)
    clocks = sampler.stop()
    elapsed_ms = start.elapsed_time(stop)
    gu_ms = statistics.mean(a.elapsed_time(b) for a, b in zip(ev0, ev1))
    code, detail = B.ordermoe_device_error()
    if code:
        raise RuntimeError("device error %d (%d) during the timed steps" % (code, detail))
    elapsed_ms = dist.max(elapsed_ms, device)
    breakdown = phase_breakdown(step_phases, stream, reps=20)
    total_tokens = T * args.steps * dist.world
    value = total_tokens / (elapsed_ms / 1e3)

    # end to end through the C ABI with host buffers (pinned), copies timed:
    # ordermoe_layer_forward_batches over queues of E2E_QUEUE batches, each
    # batch's copies overlapping its neighbours' compute
    e2e = None
    if not args.no_e2e:
        E2E_QUEUE = 16
        scratch = torch.empty(B.ordermoe_layer_batches_scratch_bytes(T, E, d, dff, k),
                              dtype=torch.uint8, device=device)
        desc = B.make_layer_desc(T, Wr, W1, W3, W2, tables, k, scratch)
        Xh = X.cpu().unsqueeze(0).expand(E2E_QUEUE, T, d).contiguous().pin_memory()
        hh = home.cpu().unsqueeze(0).expand(E2E_QUEUE, T).contiguous().pin_memory()
        yh = torch.empty(E2E_QUEUE, T, d, dtype=torch.bfloat16).pin_memory()
        B.ordermoe_layer_forward_batches(desc, E2E_QUEUE, T, Xh, hh, yh)
        calls = max(1, min(args.steps, 200) // E2E_QUEUE)
        n_e2e = calls * E2E_QUEUE
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        dist.barrier(device)
        torch.cuda.synchronize(device)
        a.record(stream)
        for _ in range(calls):
            B.ordermoe_layer_forward_batches(desc, E2E_QUEUE, T, Xh, hh, yh)
        b.record(stream)
        torch.cuda.synchronize(device)
        dist.barrier(device)
        e_ms = dist.max(a.elapsed_time(b), device)
        e2e = {"value": round(T * n_e2e * dist.world / (e_ms / 1e3), 1), "unit": UNIT,
               "h2d_bytes_per_step": T * d * 2 + T, "d2h_bytes_per_step": T * d * 2,
               "steps": n_e2e,
               "api": "ordermoe_layer_forward_batches, %d batches per call" % E2E_QUEUE}
        code, detail = B.ordermoe_device_error()
        if code:
            raise RuntimeError("device error %d (%d) during the e2e steps" % (code, detail))

    pk, pk_kind = peaks()
    gu_flop = 2.0 * R * d * 2 * dff
    achieved = gu_flop / (gu_ms / 1e3) / 1e12
    layer_flop = 2.0 * R * 3 * d * dff + 2.0 * T * d * E
    out = {
        "metric": METRIC, "value": round(value, 1), "unit": UNIT, "n_gpus": dist.world,
        "steps": args.steps, "warmup": max(args.warmup, 3),
        "ms_per_step": round(elapsed_ms / args.steps, 4), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "T": T, "d": d, "E": E, "k": k, "d_ff": dff, "M": w.M,
                   "similarity_groups": w.n_clusters, "theta": w.theta, "qbar": w.qbar,
                   "home": w.home, "seed": args.seed, "parallelism": "replicas",
                   "l2": "inputs larger than L2: %.2f GB of expert weights read every step"
                         % (3 * E * d * dff * 2 / 1e9)},
        "roofline": tensor_roofline(
            gate_up_kernel_name(T * k, E, dff), achieved, pk, pk_kind, clocks, elapsed_ms / 1e3,
            traffic=gate_up_traffic(w.name), flop_per_launch=gu_flop, ms_per_launch=round(gu_ms, 4),
            layer_tflops=round(layer_flop / (elapsed_ms / args.steps / 1e3) / 1e12, 1),
            layer_frac=round(layer_flop / (elapsed_ms / args.steps / 1e3) / 1e12
                             / tensor_peak(pk, pk_kind, clocks, elapsed_ms / 1e3)[0], 4)),
        "e2e": e2e,
        "gpu_launches": KERNELS_PER_STEP * args.steps,
        "breakdown_ms": breakdown,
        "clocks": clocks,
        "exec_types": dict(zip(["local_exact", "local_sub", "remote_exact", "remote_sub"],
                               counters.cpu().tolist())),
        "rows_per_expert": torch.diff(offsets).cpu().tolist(),
        "plan": plan,
    }
    if dist.rank == 0 and dist.world == 1 and not args.no_cpu_baseline:
        out["cpu_baseline"] = cpu_baseline(w, inp, args.seed, args.cpu_seconds)
    if w.name == "mixtral_prefill" and not args.no_extras:
        torch.cuda.empty_cache()
        out["other_workloads"] = other_workloads(args, dist, device)
    return out


EXTRA_STEPS = 50


def other_workloads(args, dist, device):
    """The other full-size workloads, each timed in this run like the main
    one (CUDA events around K steps after W warm-up steps, clocks sampled
    during the region), reported compactly: the fine-grained layer, the
    decode stack (myopic and with the paper's default horizon H = 3) and the
    offline plan."""
    import copy

    import torch
    from paper_2607_17154_gb300 import synth
    sub = copy.copy(args)
    sub.steps = min(args.steps, EXTRA_STEPS)
    sub.warmup = max(3, min(args.warmup, 5))
    sub.no_cpu_baseline = True
    sub.no_e2e = True
    sub.no_extras = True
    sub.theta = None
    sub.n_cal = None
    out = {}
    # fine-grained layer: E = 64, top-6, Zipf homes
    sub.workload = "fine_grained"
    fg = run_ours(sub, dist)
    r = fg["roofline"]
    out["fine_grained"] = {
        "value": fg["value"], "unit": UNIT, "steps": sub.steps, "ms_per_step": fg["ms_per_step"],
        "gate_up": {k: r[k] for k in ("kernel", "achieved", "frac", "frac_burst", "frac_sustained",
                                      "peak_applies", "ms_per_launch")},
        "layer_tflops": r["layer_tflops"], "layer_frac": r["layer_frac"],
        "breakdown_ms": fg["breakdown_ms"], "clocks": fg["clocks"],
        "gpu_launches": fg["gpu_launches"]}
    del fg
    torch.cuda.empty_cache()
    # decode stack on the residual map, H = 1 and H = 3
    w = synth.workload("decode_stack")
    sub.workload = "decode_stack"
    sub.memory_ratio = None
    S = decode_setup(sub, dist, w, device, 1)
    dec = {}
    for H in (1, 3):
        ms, clocks, stack, *_ = decode_timed(sub, dist, w, device, S, H)
        line = decode_line(sub, dist, w, ms, clocks, H, S)
        dec["H%d" % H] = {"value": line["value"], "unit": UNIT, "steps": sub.steps,
                          "ms_per_step": line["ms_per_step"],
                          "hbm": {k: line["roofline"][k] for k in ("achieved", "peak", "frac", "unit",
                                                                   "peak_source")},
                          "clocks": clocks, "gpu_launches": line["gpu_launches"]}
        del stack
    dec["config"] = line["config"]
    out["decode_stack"] = dec
    del S
    torch.cuda.empty_cache()
    # offline plan: similarity + grouping + placement + redundancy + coverage
    w = synth.workload("similarity")
    sub.workload = "similarity"
    pl = run_similarity(sub, dist, w, device)
    out["similarity_plan"] = {
        "value": pl["value"], "unit": pl["unit"], "metric": pl["metric"], "steps": sub.steps,
        "ms_per_step": pl["ms_per_step"],
        "tensor": {k: pl["roofline"][k] for k in ("achieved", "frac", "frac_burst", "frac_sustained",
                                                  "peak_applies")},
        "clocks": pl["clocks"], "gpu_launches": pl["gpu_launches"]}
    del pl
    torch.cuda.empty_cache()
    return out


def phase_breakdown(phases_fn, stream, reps=20):
    """Mean time of each phase of a step (CUDA events around each C-ABI call),
    measured after the timed region; informational, not part of `value`."""
    import torch
    names = [n for n, _ in phases_fn()]
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)] for _ in range(reps)]
    for r in range(reps):
        ev[r][0].record(stream)
        for i, (_, fn) in enumerate(phases_fn()):
            fn()
            ev[r][i + 1].record(stream)
    torch.cuda.synchronize()
    return {n: round(statistics.mean(ev[r][i].elapsed_time(ev[r][i + 1]) for r in range(reps)), 4)
            for i, n in enumerate(names)}


def timed_region(args, dist, device, fn):
    """W warm-up calls, then K timed calls between barriers and synchronizes,
    CUDA events on the current stream; returns (max-over-ranks ms, clocks)."""
    import torch
    for _ in range(max(args.warmup, 3)):
        fn()
    stream = torch.cuda.current_stream(device)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    sampler = ClockSampler(gpu_index(dist.local_rank))
    sampler.start()
    dist.barrier(device)
    torch.cuda.synchronize(device)
    a.record(stream)
    for _ in range(args.steps):
        fn()
    b.record(stream)
    torch.cuda.synchronize(device)
    dist.barrier(device)
    clocks = sampler.stop()
    return dist.max(a.elapsed_time(b), device), clocks


def plan_coverage(B, group, ng, x, L, E, M, device):
    """Local group coverage (Eq. 32) of a placement: covered (server, group)
    pairs over M * sum_l K_l."""
    import torch
    covered = torch.empty(L, dtype=torch.int32, device=device)
    B.ordermoe_coverage(group, x, L, E, M, None, covered)
    return {"coverage": round(covered.sum().item() / (M * int(ng.sum().item())), 4)}


def edge_cost_windows(args, w, device, layers, Xs, home, tabs, stride, P, H, sim, group, x, theta,
                      sp, windows=3, kappa=0.1):
    """Untimed: the edge cost (Eqs. 13-20) of one step's decisions over the
    layers, the same for the exact-only decisions on the same deployment
    (substitution off), the utility (Eq. 23), and `windows` rounds of weight
    adaptation (Eq. 45), each rebuilding the tables with the new weights."""
    import torch
    from paper_2607_17154_gb300 import binding as B
    L, T, E, M, k = w.L, w.T, w.E, w.M, w.k
    rec = [torch.empty(L, T, k, dtype=dt, device=device) for dt in (torch.int32, torch.int32, torch.uint8)]
    wtmp = torch.empty(T, k, device=device)
    ktmp = torch.empty(T, k, dtype=torch.uint8, device=device)
    loc = torch.empty_like(home)
    qhat = torch.empty(T, device=device)
    f64 = lambda a: torch.as_tensor(a, dtype=torch.float64).to(device)
    gF, gB, gt = f64(sp.F), f64(sp.B), f64(sp.tau)
    th = theta.cpu().tolist()

    def build(buf, omega_T, omega_Q, exact=False):
        for l in range(L):
            B.ordermoe_build_tables(sim[l], group[l], x[l], 2.0 if exact else th[l], w.qbar, gF, gB,
                                    gt, sp.z, sp.c, omega_T, omega_Q, buf[l * stride:(l + 1) * stride])

    def select_pass(buf):
        loc.copy_(home); qhat.zero_()
        for l in range(L):
            Hl = min(H, L - l)
            B.ordermoe_route_select_lookahead(Xs[l], layers[l]["W_r"], None, T, E, w.d, k, 1,
                                              buf[l * stride:], stride, Hl,
                                              P[l:l + Hl - 1].contiguous() if Hl > 1 else None,
                                              home, loc, qhat, None, rec[0][l], wtmp, rec[1][l],
                                              rec[2][l], ktmp)

    def cost(buf):
        d = torch.empty(T, dtype=torch.float64, device=device)
        q = torch.empty(T, dtype=torch.float64, device=device)
        n = torch.empty(T, dtype=torch.int32, device=device)
        B.ordermoe_trajectory_cost(rec[0], rec[1], rec[2], home, L, T, k, E, buf, stride, M, gF, gB,
                                   gt, sp.z, sp.c, d, q, n)
        return d, q, n

    exact_tabs = torch.zeros_like(tabs)
    build(exact_tabs, sp.omega_T, sp.omega_Q, exact=True)
    select_pass(exact_tabs)
    dref, _, nref = cost(exact_tabs)
    select_pass(tabs)
    # per-server load (slot executions per server over the step) and the
    # distribution of the accumulated loss q^ against the budget after the last layer
    load = torch.bincount(rec[2].reshape(-1).to(torch.int64), minlength=M).cpu().tolist()
    qh = qhat.float().cpu()
    edges = [round(w.qbar * i / 10, 4) for i in range(11)]
    qhist = torch.histc(qh, bins=10, min=0.0, max=float(w.qbar)).to(torch.int64).tolist()
    out = torch.empty(5, dtype=torch.float64, device=device)
    stream = torch.cuda.current_stream(device)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    ev[0].record(stream)
    d, q, n = cost(tabs)
    B.ordermoe_utility(d, dref, q, T, w.qbar, sp.omega_T, sp.omega_Q, kappa, out)
    ev[1].record(stream)
    torch.cuda.synchronize(device)
    first = out.cpu().tolist()
    res = {
        "mean_delay_ms": round(d.mean().item() * 1e3, 4),
        "mean_delay_exact_only_ms": round(dref.mean().item() * 1e3, 4),
        "mean_loss": round(q.mean().item(), 5), "qbar": w.qbar,
        "transfers_per_1k_tokens": round(n.sum().item() * 1000.0 / T, 1),
        "transfers_per_1k_tokens_exact_only": round(nref.sum().item() * 1000.0 / T, 1),
        "traffic_bytes_per_1k_tokens": round(n.sum().item() * sp.z * 1000.0 / T, 1),
        "U": round(first[0], 4), "Tbar": round(first[1], 4), "Qbar": round(first[2], 4),
        "cost_and_utility_us": round(ev[0].elapsed_time(ev[1]) * 1e3, 1),
        "server_load": load,
        "qhat_hist": {"edges": edges, "counts": qhist},
    }
    # adaptation windows: each prices one step under the current weights
    wT, wQ = first[3], first[4]
    trace = [[sp.omega_T, round(first[1], 4), round(first[2], 4)]]
    work = torch.zeros_like(tabs)
    for _ in range(windows):
        build(work, wT, wQ)
        select_pass(work)
        d, q, n = cost(work)
        B.ordermoe_utility(d, dref, q, T, w.qbar, wT, wQ, kappa, out)
        o = out.cpu().tolist()
        trace.append([round(wT, 4), round(o[1], 4), round(o[2], 4)])
        wT, wQ = o[3], o[4]
    res["adaptation"] = {"kappa": kappa, "omega_T_Tbar_Qbar_per_window": trace}
    return res


def decode_setup(args, dist, w, device, H):
    """The decode stack on the residual map: weights of every layer, the
    calibration pass through the unmodified stack (similarity, counts and
    transitions of each layer on the inputs it sees), the placement with b_m
    carried over the layers (Alg. 1), optional replicas, and the tables."""
    import torch
    from paper_2607_17154_gb300 import binding as B
    from paper_2607_17154_gb300 import synth
    from paper_2607_17154_gb300.layer import calibrate_stack
    seed = args.seed + 1000 * dist.rank
    L, E, M = w.L, w.E, w.M
    layers = []
    for l in range(L):
        inp = synth.layer_inputs(w, seed=seed, layer=l, device=device)
        layers.append({"W_r": inp["Wr"], "W1": inp["W1"], "W3": inp["W3"], "W2": inp["W2"]})
    home = torch.as_tensor(synth.layer_inputs(w, seed=seed, with_ffn=False)["home"]).to(device)
    cal = calibrate_stack(layers, synth.calibration(w.n_cal, w.d, seed, device=device), w.k, M)
    sim, counts, P = cal["sim"], cal["counts"], cal["P"]
    del cal
    group = torch.empty(L, E, dtype=torch.int32, device=device)
    ng = torch.empty(L, dtype=torch.int32, device=device)
    theta = torch.empty(L, dtype=torch.float32, device=device)
    x = torch.empty(L, M, E, dtype=torch.uint8, device=device)
    used = torch.empty(M, dtype=torch.float64, device=device)
    st = torch.empty(1, dtype=torch.int32, device=device)
    imp = torch.empty(L, E, dtype=torch.float64, device=device)
    ratio = 1.0 if args.memory_ratio is None else args.memory_ratio
    pmem = torch.ones(L, E, dtype=torch.float64, device=device)
    Cm = (torch.full((M,), L * E / M, dtype=torch.float64, device=device) if ratio == 1.0 else
          torch.as_tensor(synth.capacities(M, L * E, ratio, seed), dtype=torch.float64).to(device))
    B.ordermoe_place(sim, counts, L, E, M, w.theta_min, w.theta_max, w.theta, 0.5, 0.5, 0.5, 0.5,
                     pmem, Cm, group, ng, theta, imp, x, used, st)
    plan = plan_coverage(B, group, ng, x, L, E, M, device)
    if ratio > 1.0:
        pi = torch.as_tensor(synth.token_shares(home.cpu().numpy(), M), dtype=torch.float64).to(device)
        reps = torch.empty(M, dtype=torch.int32, device=device)
        B.ordermoe_replicate(group, imp, pmem, Cm, pi, L, E, M, x, used, reps)
        plan.update({"replicas": int(reps.sum().item()),
                     "coverage_after": plan_coverage(B, group, ng, x, L, E, M, device)["coverage"]})
    sp = synth.server_params(M, w.d, w.dff, seed)
    f64 = lambda a: torch.as_tensor(a, dtype=torch.float64).to(device)
    th = theta.cpu().tolist()
    stride = B.ordermoe_tables_bytes(E, M)
    tabs = torch.zeros(L * stride, dtype=torch.uint8, device=device)
    for l in range(L):
        B.ordermoe_build_tables(sim[l], group[l], x[l], th[l], w.qbar, f64(sp.F), f64(sp.B),
                                f64(sp.tau), sp.z, sp.c, sp.omega_T, sp.omega_Q,
                                tabs[l * stride:(l + 1) * stride])
    h0 = synth.hidden(w.T, w.d, seed + 5000, device=device)
    return {"layers": layers, "home": home, "sim": sim, "group": group, "x": x, "theta": theta,
            "P": P, "tabs": tabs, "stride": stride, "sp": sp, "plan": plan, "ratio": ratio,
            "h0": h0}


def decode_timed(args, dist, w, device, S, H):
    """Times graph-replayed (or eager) decode steps of the stack S with
    horizon H; returns (ms, clocks, stack, hs, xs, loc, qhat)."""
    import torch
    from paper_2607_17154_gb300.layer import LayerStack
    L = w.L
    stack = LayerStack(S["layers"], S["tabs"], w.k, w.T, device, H=H, stride=S["stride"], P=S["P"])
    home = S["home"]
    hs = [S["h0"]] + [torch.empty_like(S["h0"]) for _ in range(L)]
    xs = [torch.empty_like(S["h0"]) for _ in range(L + 1)]
    loc = home.clone()
    qhat = torch.zeros(w.T, device=device)

    def reset():
        loc.copy_(home)
        qhat.zero_()

    if not args.eager:
        graph = stack.capture_residual(hs, xs, home, loc, qhat, prologue=reset)
        step = graph.replay
    else:
        def step():
            reset()
            stack.step_residual(hs, xs, home, loc, qhat)
    ms, clocks = timed_region(args, dist, device, step)
    return ms, clocks, stack, hs, xs, loc, qhat


def decode_launches(w, H):
    """Kernels of one decode step: the first layer's RMSNorm, then per layer
    route_select 1 (2 with a look-ahead horizon H > 1 or more than 16
    experts: a separate selection kernel), dispatch 2 (one block ranks up to
    4096 entries) or 4, gate/up 1, down 1 and the residual combine 1."""
    route = 1 if (H == 1 and w.E <= 16) else 2
    return 1 + (route + 3 + (2 if w.T * w.k <= 4096 else 4)) * w.L


def run_decode(args, dist, w, device):
    """Decode stack: one step = 32 MoE layers over a batch of 128 tokens on the
    residual map (h_{l+1} = h_l + y_l, each layer reading RMSNorm(h_l)), with
    the selection state carried across layers; bound by streaming the expert
    weights from HBM."""
    import torch
    from paper_2607_17154_gb300 import binding as B
    H = max(1, args.lookahead)
    S = decode_setup(args, dist, w, device, H)
    L, E = w.L, w.E
    ms, clocks, stack, hs, xs, loc, qhat = decode_timed(args, dist, w, device, S, H)
    code, detail = B.ordermoe_device_error()
    if code:
        raise RuntimeError("device error %d (%d)" % (code, detail))
    home, tabs, stride, P, layers = S["home"], S["tabs"], S["stride"], S["P"], S["layers"]
    # execution types of one step's decisions (untimed)
    kinds = torch.zeros(4, dtype=torch.int32, device=device)
    loc.copy_(home); qhat.zero_()
    stack.step_residual(hs, xs, home, loc, qhat, counters=kinds)
    exec_types = dict(zip(["local_exact", "local_sub", "remote_exact", "remote_sub"],
                          kinds.cpu().tolist()))
    # decision time: the selection alone (router + top-k + Alg. 2) over the 32 layers, on the
    # layer inputs of that step
    f = lambda *sh, dt: torch.empty(*sh, dtype=dt, device=device)
    sel = [f(w.T, w.k, dt=dt) for dt in (torch.int32, torch.float32, torch.int32, torch.uint8, torch.uint8)]
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    stream = torch.cuda.current_stream(device)
    ev[0].record(stream)
    for _ in range(5):
        loc.copy_(home); qhat.zero_()
        for l in range(L):
            Hl = min(H, L - l)
            B.ordermoe_route_select_lookahead(xs[l], layers[l]["W_r"], None, w.T, E, w.d, w.k, 1,
                                              tabs[l * stride:], stride, Hl,
                                              P[l:l + Hl - 1].contiguous() if Hl > 1 else None,
                                              home, loc, qhat, None, *sel)
    ev[1].record(stream)
    torch.cuda.synchronize(device)
    select_ms_per_layer = ev[0].elapsed_time(ev[1]) / (5 * L)
    edge = edge_cost_windows(args, w, device, layers, xs[:L], home, tabs, stride, P, H, S["sim"],
                             S["group"], S["x"], S["theta"], S["sp"])
    out = decode_line(args, dist, w, ms, clocks, H, S)
    out.update({"plan": S["plan"], "exec_types": exec_types, "edge": edge,
                "selection_ms_per_layer": round(select_ms_per_layer, 4),
                "selection_us_per_token_layer": round(select_ms_per_layer * 1e3 / w.T, 4)})
    return out


def decode_line(args, dist, w, ms, clocks, H, S):
    step_s = ms / args.steps / 1e3
    wbytes = 3.0 * w.E * w.d * w.dff * 2 * w.L
    pk, pk_kind = peaks()
    achieved = wbytes / step_s / 1e9
    peak = float(pk.get("hbm_gbs", FALLBACK_PEAKS["hbm_gbs"]))
    return {
        "metric": METRIC, "value": round(w.T * args.steps * dist.world / (ms / 1e3), 1), "unit": UNIT,
        "n_gpus": dist.world, "steps": args.steps, "warmup": max(args.warmup, 3),
        "ms_per_step": round(ms / args.steps, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "layers": w.L, "T": w.T, "d": w.d, "E": w.E, "k": w.k,
                   "d_ff": w.dff, "M": w.M, "lookahead_H": H, "memory_ratio": S["ratio"],
                   "inter_layer": "h_{l+1} = h_l + y_l, layer input RMSNorm(h_l)",
                   "cuda_graph": not args.eager,
                   "l2": "inputs larger than L2: %.1f GB of expert weights" % (wbytes / 1e9)},
        "roofline": {"kernel": "whole decode step (expert weight streaming)", "bound": "hbm",
                     "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                     "frac": round(achieved / peak, 4), "traffic": None,
                     "peak_source": "%s hbm_gbs" % pk_kind, "bytes_per_step": wbytes},
        # plus the look-ahead selection pass on every layer that looks ahead
        # (all but the last when H > 1)
        "gpu_launches": (decode_launches(w, H)
                         + sum(min(H, w.L - l) > 1 for l in range(w.L))) * args.steps,
        "clocks": clocks,
        "lookahead_H": H,
    }


def plan_launches(L, E):
    """Kernels of one ordermoe_plan call: on the tensor-core path (E in {8,
    16, 32, 64}, L E <= 4096) the layers go in blocks of 512 logit columns,
    the last block in two halves when there is more than one, and each block
    launches the logits GEMM, the Gram, its reduction, the similarities and
    one grouping + placement kernel (5); otherwise the similarity takes 5 and
    the placement 2. Replication and coverage add 1 each."""
    if E in (8, 16, 32, 64) and L * E <= 4096:
        part = max(1, 512 // E)
        nfull = (L + part - 1) // part
        last_n = L - (nfull - 1) * part
        blocks = nfull + (1 if nfull > 1 and last_n >= 2 else 0)
        return 5 * blocks + 2
    return 5 + 2 + 2


def run_similarity(args, dist, w, device):
    """Offline similarity of 24 layers x 64 experts over 262144 calibration
    tokens (Eqs. 3-5), then grouping and placement (Eqs. 6, 24-31)."""
    import torch
    from paper_2607_17154_gb300 import binding as B
    from paper_2607_17154_gb300 import synth
    L, E, d, N = w.L, w.E, w.d, w.n_cal
    seed = args.seed + 1000 * dist.rank
    Wr = torch.stack([synth.router_weights(E, d, w.n_clusters, seed=seed + 500 + l, device=device)
                      for l in range(L)])
    Xcal = synth.calibration(N, d, seed, device=device)
    sim = torch.empty(L, E, E, dtype=torch.float32, device=device)
    counts = torch.empty(L, E, dtype=torch.int32, device=device)
    ws = torch.empty(B.ordermoe_plan_workspace_bytes(L, E, N), dtype=torch.uint8, device=device)
    group = torch.empty(L, E, dtype=torch.int32, device=device)
    ng = torch.empty(L, dtype=torch.int32, device=device)
    theta = torch.empty(L, dtype=torch.float32, device=device)
    x = torch.empty(L, w.M, E, dtype=torch.uint8, device=device)
    used = torch.empty(w.M, dtype=torch.float64, device=device)
    st = torch.empty(1, dtype=torch.int32, device=device)
    imp = torch.empty(L, E, dtype=torch.float64, device=device)
    reps = torch.empty(w.M, dtype=torch.int32, device=device)
    covered = torch.empty(L, dtype=torch.int32, device=device)
    p = torch.ones(L, E, dtype=torch.float64, device=device)
    ratio = 2.0 if args.memory_ratio is None else args.memory_ratio
    C = torch.as_tensor(synth.capacities(w.M, L * E, ratio, seed), dtype=torch.float64).to(device)
    # pi_m of Eq. 33 from a non-uniform (Zipf 1.1) user-server association
    pi = torch.as_tensor(synth.token_shares(synth.homes(65536, w.M, seed, "zipf1.1"), w.M),
                         dtype=torch.float64).to(device)

    def step():  # one call: similarity (no logits kept), grouping, placement, redundancy, coverage
        B.ordermoe_plan(Wr, Xcal, L, E, d, N, w.k, w.M, w.theta_min, w.theta_max, w.theta, 0.5, 0.5,
                        0.5, 0.5, p, C, pi, sim, counts, group, ng, theta, imp, x, used, st, reps,
                        None, covered, ws)

    ms, clocks = timed_region(args, dist, device, step)
    code, detail = B.ordermoe_device_error()
    if code:
        raise RuntimeError("device error %d (%d)" % (code, detail))
    step_s = ms / args.steps / 1e3
    flop = 2.0 * N * L * E * d + 2.0 * L * N * E * E
    pk, pk_kind = peaks()
    achieved = flop / step_s / 1e12
    return {
        "metric": "calibration tokens/s through the offline similarity + grouping + placement",
        "value": round(N * args.steps * dist.world / (ms / 1e3), 1), "unit": "tokens/s",
        "n_gpus": dist.world, "steps": args.steps, "warmup": max(args.warmup, 3),
        "ms_per_step": round(ms / args.steps, 4), "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": w.name, "layers": L, "E": E, "d": d, "N": N, "groups": w.n_clusters,
                   "M": w.M, "k_freq": w.k, "memory_ratio": ratio},
        "roofline": tensor_roofline(
            "ordermoe_plan: similarity (tcgen05 logits + Gram) + group + place + replicate + "
            "coverage (whole plan)", achieved, pk, pk_kind, clocks, ms / 1e3, traffic=None,
            flop_per_step=flop),
        "gpu_launches": plan_launches(L, E) * args.steps,
        "n_groups": ng.cpu().tolist()[:3], "place_status": int(st.item()),
        "replicas": int(reps.sum().item()),
        "coverage": round(covered.sum().item() / (w.M * int(ng.sum().item())), 4),
        "clocks": clocks,
    }


# ----------------------------------------------------------------- oracle side
def oracle_setup(w, inp, seed):
    """Host copies of the inputs and the oracle's own plan and tables."""
    import numpy as np

    import oracle
    from paper_2607_17154_gb300 import synth
    bits = synth.bits
    host = {n: bits(inp[n]) for n in ("X", "Wr", "W1", "W3", "W2")}
    home = np.asarray(inp["home"].cpu() if hasattr(inp["home"], "cpu") else inp["home"], np.uint8)
    Xcal = bits(synth.calibration(w.n_cal, w.d, seed, device=inp["X"].device))
    sim, H = oracle.similarity(host["Wr"], Xcal, return_H=True)
    counts = oracle.expert_counts(np.ascontiguousarray(H.T), w.k)
    group, K, _ = oracle.group(sim, counts, w.theta)
    imp = oracle.importance(sim, counts, group)
    x, _, _ = oracle.place(group[None], imp[None], np.ones((1, w.E)), np.full(w.M, w.E / w.M))
    sp = synth.server_params(w.M, w.d, w.dff, seed)
    tab = oracle.tables(sim, group, x[0], w.theta, w.qbar, sp.F, sp.B, sp.tau, sp.z, sp.c,
                        sp.omega_T, sp.omega_Q)
    return host, home, tab


def oracle_tokens(w, host, home, tab, toks):
    """The oracle's whole hot path for the listed tokens."""
    import numpy as np

    import oracle
    Xs = np.ascontiguousarray(host["X"][toks])
    logits = oracle.router_logits(Xs, host["Wr"])
    idx, wt = oracle.topk(logits, w.k)
    h = home[toks]
    chosen, _, _, _, _ = oracle.select(idx, tab, h, h.copy(), np.zeros(len(toks), np.float32))
    off, rt, row_of = oracle.dispatch(chosen, w.E)
    Xp = oracle.gather_rows(Xs, rt)
    row_e = np.repeat(np.arange(w.E), np.diff(off)).astype(np.int32)
    _, Y = oracle.ffn_rows(Xp, row_e, host["W1"], host["W3"], host["W2"])
    return oracle.combine(Y, row_of, wt)


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count() or 1


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.split(":")[0].strip() in ("Model name", "Model"):
                name = line.split(":", 1)[1].strip()
                if name and not name.isdigit():
                    return name
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith(("model name", "cpu part")):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return "unknown"


def tiny_oracle_rate(seed, threads):
    """Tokens/s of the whole oracle path on the tiny layer (T 64, d 256, E 8,
    top-2, d_ff 512) with the given OpenMP thread count."""
    import numpy as np

    import oracle
    from paper_2607_17154_gb300 import synth
    w = synth.workload("tiny")
    inp = synth.layer_inputs(w, seed=seed)
    host, home, tab = oracle_setup(w, inp, seed)
    prev = oracle.threads()
    oracle.set_threads(threads)
    try:
        toks = np.arange(w.T)
        oracle_tokens(w, host, home, tab, toks)
        reps, t0 = 0, time.perf_counter()
        while reps < 3 or time.perf_counter() - t0 < 1.0:
            oracle_tokens(w, host, home, tab, toks)
            reps += 1
        dt = time.perf_counter() - t0
    finally:
        oracle.set_threads(prev)
    return {"value": round(w.T * reps / dt, 1), "unit": UNIT, "threads": threads,
            "sample": "all %d tokens of the tiny layer, %d passes, %.2f s" % (w.T, reps, dt)}


def cpu_baseline(w, inp, seed, target_s):
    import numpy as np

    import oracle
    host, home, tab = oracle_setup(w, inp, seed)
    rng = np.random.default_rng(seed)
    t0 = time.perf_counter()
    oracle_tokens(w, host, home, tab, np.sort(rng.choice(w.T, 4, replace=False)))
    per_tok = max((time.perf_counter() - t0) / 4, 1e-6)
    n = int(min(w.T, max(4, target_s / per_tok)))
    toks = np.sort(rng.choice(w.T, n, replace=False))
    t0 = time.perf_counter()
    oracle_tokens(w, host, home, tab, toks)
    dt = time.perf_counter() - t0
    return {"value": round(n / dt, 3), "unit": UNIT, "cores": oracle.threads(), "kind": "oracle",
            "sample": "%d of the %d tokens of one %s layer through the whole oracle path "
                      "(router, top-k, selection, permutation, SwiGLU FFN, combine), %.1f s"
                      % (n, w.T, w.name, dt),
            "cpu_model": cpu_model(), "host_cpus": cpu_cores(), "omp_threads": oracle.threads(),
            "tiny_1_thread": tiny_oracle_rate(seed, 1),
            "tiny_all_threads": tiny_oracle_rate(seed, oracle.threads()),
            "other_workloads": cpu_other_workloads(seed, inp["X"].device)}


def cpu_other_workloads(seed, device, budget_s=3.0):
    """The oracle on bounded samples of the other workloads, each scaled to
    that workload's unit and labelled with its sample: tokens of the
    fine-grained layer; tokens of one decode layer, scaled to the 32-layer
    step; calibration tokens of one similarity layer, scaled to 24 layers."""
    import numpy as np

    import oracle
    from paper_2607_17154_gb300 import synth
    out = {}
    rng = np.random.default_rng(seed)

    def sample_rate(w, inp, layers):
        host, home, tab = oracle_setup(w, inp, seed)
        t0 = time.perf_counter()
        oracle_tokens(w, host, home, tab, np.arange(2))
        per_tok = max((time.perf_counter() - t0) / 2, 1e-6)
        n = int(min(w.T, max(2, budget_s / per_tok)))
        toks = np.sort(rng.choice(w.T, n, replace=False))
        t0 = time.perf_counter()
        oracle_tokens(w, host, home, tab, toks)
        dt = time.perf_counter() - t0
        return n, dt, n / dt / layers

    w = synth.workload("fine_grained")
    n, dt, v = sample_rate(w, synth.layer_inputs(w, seed=seed, device=device), 1)
    out["fine_grained"] = {"value": round(v, 3), "unit": UNIT,
                           "sample": "%d of the %d tokens of the layer, whole oracle path, %.1f s"
                                     % (n, w.T, dt)}
    w = synth.workload("decode_stack")
    n, dt, v = sample_rate(w, synth.layer_inputs(w, seed=seed, device=device), w.L)
    out["decode_stack"] = {"value": round(v, 3), "unit": UNIT,
                           "sample": "%d of the %d tokens of one of the %d layers, whole oracle path, "
                                     "%.1f s; the step rate extrapolated as one layer's rate / %d"
                                     % (n, w.T, w.L, dt, w.L)}
    w = synth.workload("similarity")
    Wr = synth.bits(synth.router_weights(w.E, w.d, w.n_clusters, seed=seed + 500, device=device))
    n = 4096
    Xs = synth.bits(synth.calibration(n, w.d, seed, device=device))
    t0 = time.perf_counter()
    sim, H = oracle.similarity(Wr, Xs, return_H=True)
    oracle.expert_counts(np.ascontiguousarray(H.T), w.k)
    dt = time.perf_counter() - t0
    out["similarity"] = {"value": round(n / dt / w.L, 1), "unit": "tokens/s",
                         "sample": "%d calibration tokens through one of the %d layers (logits, "
                                   "cosine similarity, counts), %.1f s; the plan rate extrapolated "
                                   "as one layer's rate / %d; grouping and placement not timed"
                                   % (n, w.L, dt, w.L)}
    return out


def run_reference(args, dist):
    """The CPU oracle as it stands, each step a bounded sample of the workload."""
    import numpy as np
    import torch

    import oracle
    from paper_2607_17154_gb300 import synth
    w = synth.workload(args.workload)
    device = "cuda" if torch.cuda.is_available() else "cpu"
    inp = synth.layer_inputs(w, seed=args.seed, device=device)
    host, home, tab = oracle_setup(w, inp, args.seed)
    rng = np.random.default_rng(args.seed)
    t0 = time.perf_counter()
    oracle_tokens(w, host, home, tab, np.sort(rng.choice(w.T, 2, replace=False)))
    per_tok = max((time.perf_counter() - t0) / 2, 1e-6)
    budget = 150.0
    n = int(max(1, min(w.T, budget / max(1, args.steps + args.warmup) / per_tok)))
    for _ in range(args.warmup):
        oracle_tokens(w, host, home, tab, np.sort(rng.choice(w.T, n, replace=False)))
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_tokens(w, host, home, tab, np.sort(rng.choice(w.T, n, replace=False)))
    dt = time.perf_counter() - t0
    value = n * args.steps / dt
    sample = ("%d of the %d tokens of one %s layer per step through the whole oracle path"
              % (n, w.T, w.name))
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 3), "unit": UNIT,
        "n_gpus": dist.world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(dt / args.steps * 1e3, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "T": w.T, "d": w.d, "E": w.E, "k": w.k, "d_ff": w.dff,
                   "M": w.M, "tokens_per_step": n},
        "cpu_baseline": {"value": round(value, 3), "unit": UNIT, "cores": oracle.threads(),
                         "kind": "oracle", "sample": sample, "cpu_model": cpu_model(),
                         "host_cpus": cpu_cores(), "omp_threads": oracle.threads()},
        "e2e": {"value": round(value, 3), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }


def main():
    args = parse()
    dist = Dist()
    try:
        if args.impl == "reference":
            if dist.rank != 0:
                return
            out = run_reference(args, dist)
        else:
            out = run_ours(args, dist)
        if dist.rank == 0:
            print(json.dumps(out), flush=True)
    finally:
        dist.close()


if __name__ == "__main__":
    main()
