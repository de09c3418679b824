"""Benchmark of the quantized widely-linear layer on a LLaMA-2-7B-shaped linear stack.

Workload (headline): 32 decoder layers x {q, k, v, o, gate, up, down} (hidden 4096, intermediate
11008), every weight Student-t(df=4, std 0.02), converted and quantized with T=2 stages; one
step = one decode token (batch 1, bf16 activations with 1% outlier channels) through all 224
quantized linears, as a decoder layer feeds them: q, k, v on one input (one grouped call), o,
gate and up on one input (one grouped call), down; 4 calls per layer (--ungrouped: 7). Metric:
decode GB/s = algorithmic bytes (packed codes + scales + x + y of every linear) per second,
against the HBM copy peak. The 1.62 GB of codes per step exceed the L2 many times over, so no
L2 flush is needed between steps.

Further objects on the same line (each timed with CUDA events on the launching stream):
* decode_chain: the same step as one persistent launch (fairy2i_wl_matmul_chain, 128 calls,
  call c reading its input only after call c - 1's outputs are written);
* batches: the stack at batch 8 and 64 (per-token time), the MLP layers (gate, up, down) at
  batch 1, 4 and 16 and the attention projections (4096 -> 4096) at batch 1, each over all 32
  layers' weights so that the codes come from HBM;
* quantize: convert and quantize of the 4096 -> 11008 layer (T = 1, 2, 3), GB/s;
* prefill: the tensor-core GEMM path on 2048 tokens through the 4096 -> 11008 and
  11008 -> 4096 layers at T = 1, 2, 3 (effective TOPS = 8 n m B / time, and the MMA work
  16 T n m B / time against the bf16 tensor peak), each launch timed alone after an L2 flush;
* lut_cpu: the look-up-table matmul on the host cores (one 4096 -> 4096 linear, one token);
* cpu_baseline: the float64 oracle on the host cores (all cores, and one thread) on a bounded
  sample (layer 0's q and k at the headline batch).

--impl reference times the CPU oracle on the host cores on the same sample as cpu_baseline and
reports the same metric.

Multi-GPU: the layer is not partitioned across ranks; N ranks run N independent replicas
(weak scaling) and value = bytes of all ranks / max over ranks of the timed region.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import numpy as np  # noqa: E402
import torch  # noqa: E402

from paper_2512_02901_gb300 import synth  # noqa: E402

METRIC = "WL {±1,±i} matmul: decode GB/s vs HBM peak; prefill effective TOPS"
WORKLOAD = "llama2-7b-linear-stack-decode"
T_STAGES = 2
HBM_NOMINAL_GBS = 7900.0
SAMPLE_LINEARS = 2   # layer 0's first linears (q, k) timed by cpu_baseline and --impl reference


def peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            p = json.load(f)
        return float(p["hbm_gbs"]), float(p["bf16_tflops"]), "measured"
    except Exception:
        return 6800.0, 1900.0, "fallback"


# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) per launch, from ncu captures of the
# current kernels: one decoder layer's decode launches (every layer has the same shapes; grouped:
# q/k/v, o, gate/up, down; ungrouped: seven), and one T = 2 prefill launch of the 4096 -> 11008
# layer on 2048 tokens. Per call and decode kernel: "fp8" = the warp-MMA kernel, "stream" = the
# persistent tcgen05 kernel's one-token form.
DECODE_DRAM_BYTES = {
    "fp8": {"q,k,v": 12.621e6, "o": 4.232e6, "gate,up": 22.582e6, "down": 11.323e6,
            "q": 4.231e6, "k": 4.231e6, "v": 4.231e6, "gate": 11.309e6, "up": 11.309e6},
    "stream": {"q,k,v": 12.655e6, "o": 4.265e6, "gate,up": 22.618e6, "down": 11.357e6},
}
PREFILL_T2_UP_DRAM_BYTES = 28.121e6 + 36.813e6
# ncu sm__pipe_tensor_cycles_active of the same prefill launch (T = 2, up layer, 2048 tokens)
PREFILL_T2_UP_TENSOR_PIPE_PCT = 54.9


def decode_kernel(c, path, sms):
    """The decode kernel the library runs for a call at batch <= 2 (bf16 x): the automatic path
    takes the persistent tcgen05 kernel's one-token form, token by token."""
    if path == 1:
        return "fp8"
    if path == 5:
        return "chain"
    return "stream"


def decode_traffic(calls, path, B, sms):
    """ncu DRAM bytes of one step's decode launches (batch 1), summed per call from captures of
    the kernels this run uses; None where no capture exists for a call."""
    if B != 1:
        return None
    total = 0.0
    for c in calls:
        name = ",".join(m["name"] for m in c["members"])
        v = DECODE_DRAM_BYTES[decode_kernel(c, path, sms)].get(name)
        if v is None:
            return None
        total += v
    return int(total)


PREFILL_TOKENS = 2048
PREFILL_LAYERS = (("up", 11008, 4096, 0), ("down", 4096, 11008, 1))   # (name, out, in, seed idx)


def layer_shapes(layers: int):
    out = []
    for L in range(layers):
        for pi, (name, rows, cols) in enumerate(synth.PROJECTIONS):
            out.append((L, pi, name, rows, cols))
    return out


def layer_bytes(rows, cols, B, T=T_STAGES, x_bytes=2):
    n, m = (rows + 1) // 2, (cols + 1) // 2
    codes = T * 2 * n * m // 4            # 2 bits per complex weight
    return codes + T * 16 + B * cols * x_bytes + B * rows * 4


# --------------------------------------------------------------------------------------------
class Clocks:
    """nvidia-smi sampler running during the timed region."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "20"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        rows = []
        for line in open(self.path):
            f = [c.strip() for c in line.split(",")]
            if len(f) >= 9:
                rows.append(f)
        os.unlink(self.path)
        if not rows:
            return None
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if "Active" in r[5 + i]
                          and "Not" not in r[5 + i]})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": reasons,
                "samples": len(rows)}


# --------------------------------------------------------------------------------------------
def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(local)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(v: float, world: int) -> float:
    if world == 1:
        return v
    import torch.distributed as dist
    t = torch.tensor([v], dtype=torch.float64, device="cuda" if torch.cuda.is_available() else "cpu")
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --------------------------------------------------------------------------------------------
GROUPS = (("q", "k", "v"), ("o",), ("gate", "up"), ("down",))   # linears sharing an input


def build_linears(F, layers: int, dev):
    """Converts + quantizes every linear of the stack on the GPU: [layer][name] -> dict."""
    out = []
    for L in range(layers):
        lin = {}
        for (_, pi, name, rows, cols) in layer_shapes(1):
            seed = synth.weight_seed("stack", L, pi)
            R = synth.student_t_weight(rows, cols, seed, device=dev)
            U, W = F.convert(R)
            del R
            codes, scales = F.quantize(U, W, T_STAGES)
            del U, W
            lin[name] = dict(L=L, name=name, seed=seed, rows=rows, cols=cols, codes=codes,
                             scales=scales)
        out.append(lin)
    torch.cuda.synchronize()
    status = F.get_status()
    if status != 0:
        raise RuntimeError(f"quantize status {status}")
    return out


def make_calls(linears, B: int, dev, groups=GROUPS):
    """The calls of a step over `linears` at batch B: per call the input x and its member
    linears with their outputs. The inputs of all calls are views of one buffer, the outputs of
    another, so that a step's activations reach the device and its results the host in one copy
    each."""
    cols_of = {name: cols for (_, _, name, _, cols) in layer_shapes(1)}
    rows_of = {name: rows for (_, _, name, rows, _) in layer_shapes(1)}
    x_all = torch.empty(len(linears) * sum(B * cols_of[g[0]] for g in groups),
                        dtype=torch.bfloat16, device=dev)
    y_all = torch.empty(len(linears) * sum(B * rows_of[nm] for g in groups for nm in g),
                        dtype=torch.float32, device=dev)
    xo = yo = 0
    calls = []
    for lin in linears:
        for g in groups:
            first = lin[g[0]]
            ys = []
            for nm in g:
                ys.append(y_all[yo:yo + B * rows_of[nm]].view(B, rows_of[nm]))
                yo += B * rows_of[nm]
            x = x_all[xo:xo + B * first["cols"]].view(B, first["cols"])
            xo += B * first["cols"]
            x.copy_(synth.outlier_activations(B, first["cols"],
                                              synth.activation_seed(first["seed"], B), device=dev))
            calls.append(dict(x=x, rows=first["rows"], cols=first["cols"], ys=ys,
                              members=[lin[nm] for nm in g]))
    return calls, x_all, y_all


def step_launches(ncalls: int, B: int, path: int, T: int = T_STAGES) -> int:
    """Kernel launches of one step of `ncalls` (grouped) bf16 calls: one per call on the automatic
    path (B = 1 on a decode kernel, 2 <= B <= 4 on the chained kernel, larger batches on the
    prefill GEMM, T = 3 from 512 tokens on as two launches); one per call and per 4 tokens on the
    chained kernel chosen explicitly (path 5)."""
    if path == 5:
        return ncalls * ((B + 3) // 4)
    if T == 3 and B >= 512:
        return 2 * ncalls
    return ncalls


def call_bytes(c, B):
    """Algorithmic bytes of one call: every member's codes, scales and y, the shared x once."""
    per = [layer_bytes(m["rows"], m["cols"], B) for m in c["members"]]
    return sum(per) - (len(per) - 1) * B * c["cols"] * 2


def run_call(F, c, path=0, stream=None):
    if len(c["members"]) == 1:
        m = c["members"][0]
        F.wl_matmul(c["x"], m["codes"], m["scales"], c["rows"], y=c["ys"][0], path=path,
                    stream=stream)
    else:
        F.wl_matmul_group(c["x"], [m["codes"] for m in c["members"]],
                          [m["scales"] for m in c["members"]], c["rows"], ys=c["ys"], path=path,
                          stream=stream)


def graphed(fn, stream, warmup: int):
    """fn captured once in a CUDA graph on `stream` (after `warmup` eager runs); returns the
    replay."""
    with torch.cuda.stream(stream):
        for _ in range(max(warmup, 1)):
            fn()
    stream.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=stream):
        fn()
    stream.synchronize()
    return g.replay


def time_replays(run, stream, reps: int, warmup: int = 3) -> float:
    """Milliseconds per run() over `reps` runs (CUDA events on `stream`)."""
    with torch.cuda.stream(stream):
        for _ in range(warmup):
            run()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            run()
        e1.record(stream)
    stream.synchronize()
    return e0.elapsed_time(e1) / reps


def run_ours(args, world, rank, local):
    from paper_2512_02901_gb300 import binding as F
    from paper_2512_02901_gb300 import build as B_
    B_.build()
    F.load()
    dev = torch.device("cuda", local)
    B = args.batch
    groups = GROUPS if not args.ungrouped else tuple((nm,) for g in GROUPS for nm in g)
    linears = build_linears(F, args.layers, dev)
    calls, x_all, y_all = make_calls(linears, B, dev, groups)
    step_bytes = sum(call_bytes(c, B) for c in calls)
    nlinears = sum(len(c["members"]) for c in calls)
    launches_per_step = step_launches(len(calls), B, args.decode_path)

    def step():
        for c in calls:
            run_call(F, c, args.decode_path)

    stream = torch.cuda.Stream(device=dev)
    run = step if args.no_graph else graphed(step, stream, args.warmup)
    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            run()
    stream.synchronize()

    clocks = Clocks(torch.cuda.current_device() if "CUDA_VISIBLE_DEVICES" not in os.environ else local)
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    barrier(world)
    torch.cuda.synchronize()
    clocks.start()
    # the sampler sees the GPU under load for ~0.3 s before the timed region as well
    t_end = time.perf_counter() + 0.3
    with torch.cuda.stream(stream):
        while time.perf_counter() < t_end:
            run()
            stream.synchronize()
    barrier(world)
    torch.cuda.synchronize()
    with torch.cuda.stream(stream):
        e0.record(stream)
        for _ in range(args.steps):
            run()
        e1.record(stream)
    stream.synchronize()
    torch.cuda.synchronize()
    barrier(world)
    clk = clocks.stop()
    ms = e0.elapsed_time(e1)
    ms = max_over_ranks(ms, world)
    ms_step = ms / args.steps
    value = world * step_bytes * args.steps / (ms * 1e-3) / 1e9
    st = F.get_status()
    if st != 0:
        raise RuntimeError(f"device status {st} after the timed region")

    # end to end through the public call with host buffers: per step the inputs of all
    # linears go host->device from pinned memory and every output comes back to the host (one
    # copy each way: the calls' inputs and outputs are views of x_all and y_all).
    x_host = x_all.cpu().pin_memory()
    y_host = torch.empty(y_all.shape, dtype=torch.float32).pin_memory()
    h2d = x_host.numel() * x_host.element_size()
    d2h = y_host.numel() * 4

    def e2e_step():
        x_all.copy_(x_host, non_blocking=True)
        run()
        y_host.copy_(y_all, non_blocking=True)

    e2e_steps = max(1, min(args.steps, 50))
    barrier(world)
    ms_e2e = max_over_ranks(time_replays(e2e_step, stream, e2e_steps, args.warmup) * e2e_steps,
                            world)
    st = F.get_status()
    if st != 0:
        raise RuntimeError(f"device status {st} after the end-to-end steps")
    e2e_value = world * step_bytes * e2e_steps / (ms_e2e * 1e-3) / 1e9

    hbm, _, peak_kind = peaks()
    achieved = step_bytes / (ms_step * 1e-3) / 1e9
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    traffic = decode_traffic(calls, args.decode_path, B, sms)
    kernels = (sorted({decode_kernel(c, args.decode_path, sms) for c in calls}) if B == 1 else
               ["chain"] if (B <= 4 and args.decode_path == 0) or args.decode_path == 5 else [])
    kname = ("wl_matmul decode (all launches of the step: "
             + " + ".join({"fp8": "warp-MMA", "stream": "persistent tcgen05",
                           "chain": "chained tcgen05"}[k] for k in kernels)
             + ")") if kernels else "wl_matmul (all launches of the step: tcgen05 GEMM)"
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": "GB/s", "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_step, 5),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "data": "synthetic (seeded Student-t weights, N(0,1) bf16 activations with 1% x20 "
                "outlier channels)",
        "config": {"workload": WORKLOAD, "layers": args.layers, "linears": nlinears,
                   "calls_per_step": launches_per_step,
                   "grouping": "none" if args.ungrouped else "qkv, o, gate+up, down (shared x)",
                   "decode_path": args.decode_path,
                   "T": T_STAGES, "batch": B, "x_dtype": "bf16",
                   "bytes_per_step": step_bytes, "cuda_graph": not args.no_graph,
                   "l2": "inputs larger than L2 (packed codes per step >> 129 MB)",
                   "parallelism": f"replicas{world}"},
        "e2e": {"value": round(e2e_value, 2), "unit": "GB/s", "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h},
        "gpu_launches": launches_per_step * args.steps,
        "roofline": {"bound": "hbm", "achieved": round(achieved, 1), "peak": hbm,
                     "unit": "GB/s", "frac": round(achieved / hbm, 4),
                     "frac_nominal": round(achieved / HBM_NOMINAL_GBS, 4),
                     "traffic": traffic,
                     "peak_kind": f"{peak_kind} hbm_gbs (burst copy); frac_nominal against "
                                  f"{HBM_NOMINAL_GBS:.0f} GB/s nominal",
                     "kernel": kname},
        "clocks": clk,
    }
    del x_host, y_host
    if B == 1 and not args.ungrouped and not args.no_chain:
        line["decode_chain"] = run_chain(F, calls, dev, step_bytes, args)
    del calls, x_all, y_all
    torch.cuda.empty_cache()
    if not args.no_sweep:
        line["batches"] = run_batches(F, linears, dev, args)
    del linears
    torch.cuda.empty_cache()
    if not args.no_quantize:
        line["quantize"] = run_quantize(F, dev)
    if not args.no_prefill:
        line["prefill"] = run_prefill(F, dev, args.prefill_steps, max(args.warmup, 3))
    if rank == 0 and not args.no_lut:
        line["lut_cpu"] = run_lut(F)
    if rank == 0 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(B, budget_s=args.cpu_budget, count=args.ref_linears)
    return line


def run_chain(F, calls, dev, step_bytes, args):
    """The step as one launch of the chained decode kernel."""
    hbm, _, peak_kind = peaks()
    tup = [(c["x"], [m["codes"] for m in c["members"]], [m["scales"] for m in c["members"]],
            c["ys"], c["rows"]) for c in calls]
    arr = F.chain_calls(tup)
    ws = F.chain_workspace(len(tup), dev)
    stream = torch.cuda.Stream(device=dev)
    run = graphed(lambda: F.wl_matmul_chain(None, T_STAGES, workspace=ws, stream=stream, arr=arr),
                  stream, 2)
    reps = max(5, min(args.steps, 50))
    ms = time_replays(run, stream, reps, max(args.warmup, 3))
    if F.get_status() != 0:
        raise RuntimeError("device status after the chained decode")
    gbs = step_bytes / (ms * 1e-3) / 1e9
    return {"workload": f"{WORKLOAD} (batch 1), one launch", "calls": len(tup),
            "us_per_step": round(ms * 1e3, 1), "value": round(gbs, 1), "unit": "GB/s",
            "frac": round(gbs / hbm, 4), "frac_nominal": round(gbs / HBM_NOMINAL_GBS, 4),
            "peak_kind": f"{peak_kind} hbm_gbs", "gpu_launches": reps}


def run_batches(F, linears, dev, args):
    """Other batches: the whole stack at batch 8 and 64 (per token), the MLP layers at batch 1,
    4 and 16, the attention projections at batch 1; every figure runs over all layers' weights
    (codes from HBM), through the automatic path."""
    hbm, _, _ = peaks()
    stream = torch.cuda.Stream(device=dev)
    out = []
    cases = [("stack", GROUPS, 8), ("stack", GROUPS, 64),
             ("mlp gate+up, down", (("gate", "up"), ("down",)), 1),
             ("mlp gate+up, down", (("gate", "up"), ("down",)), 4),
             ("mlp gate+up, down", (("gate", "up"), ("down",)), 16),
             ("attention q, k, v, o (4096->4096 each)", (("q",), ("k",), ("v",), ("o",)), 1)]
    for name, groups, B in cases:
        calls, x_all, y_all = make_calls(linears, B, dev, groups)
        nbytes = sum(call_bytes(c, B) for c in calls)
        nlin = sum(len(c["members"]) for c in calls)

        def step():
            for c in calls:
                run_call(F, c, 0, stream)

        run = graphed(step, stream, 1)
        reps = 5 if B >= 16 else 10
        ms = time_replays(run, stream, reps, 2)
        if F.get_status() != 0:
            raise RuntimeError(f"device status after batch {B} ({name})")
        gbs = nbytes / (ms * 1e-3) / 1e9
        rec = {"case": name, "batch": B, "layers": len(linears), "linears": nlin,
               "us_per_pass": round(ms * 1e3, 1), "value": round(gbs, 1), "unit": "GB/s",
               "frac": round(gbs / hbm, 4)}
        if name == "stack":
            rec["us_per_token"] = round(ms * 1e3 / B, 2)
        if name.startswith("attention"):
            rec["us_per_linear"] = round(ms * 1e3 / nlin, 2)
        if name.startswith("mlp"):
            rec["us_per_layer"] = round(ms * 1e3 / len(linears), 2)
        rec["path"] = ("persistent tcgen05, one-token form" if B == 1 else
                       "chained tcgen05, one launch per call" if B <= 4 else
                       "tcgen05 GEMM (%d-token tiles; K split over CTA pairs where the "
                       "tiles fill the SMs poorly)" % (32 if B <= 32 else 64))
        out.append(rec)
        del calls, x_all, y_all
    torch.cuda.empty_cache()
    return out


def run_quantize(F, dev):
    """convert + quantize of the 4096 -> 11008 layer: median of 5 timed runs each (L2 flushed
    before each), GB/s of the traffic each makes: convert reads R and writes U, W; quantize reads
    U, W T + 1 times (T stage passes and the pack pass) and writes the codes."""
    hbm, _, _ = peaks()
    rows, cols = 11008, 4096
    n, m = (rows + 1) // 2, (cols + 1) // 2
    R = synth.student_t_weight(rows, cols, synth.weight_seed("prefill", 0), device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    stream = torch.cuda.Stream(device=dev)
    stream.wait_stream(torch.cuda.current_stream())

    def timed(fn, reps=5):
        ts = []
        with torch.cuda.stream(stream):
            for i in range(reps + 2):
                flush.zero_()
                e0 = torch.cuda.Event(enable_timing=True)
                e1 = torch.cuda.Event(enable_timing=True)
                e0.record(stream)
                fn()
                e1.record(stream)
                if i >= 2:
                    ts.append((e0, e1))
        stream.synchronize()
        return statistics.median(a.elapsed_time(b) for a, b in ts)

    res = {}
    U, W = F.convert(R, stream=stream)
    ms_c = timed(lambda: F.convert(R, stream=stream))
    conv_bytes = rows * cols * 4 + 2 * n * m * 8
    res["convert"] = {"us": round(ms_c * 1e3, 1), "bytes": conv_bytes,
                      "gbs": round(conv_bytes / (ms_c * 1e-3) / 1e9, 1),
                      "frac": round(conv_bytes / (ms_c * 1e-3) / 1e9 / hbm, 4)}
    res["quantize"] = []
    for T in (1, 2, 3):
        ws = torch.empty(F.quantize_workspace_bytes(n, m, T), dtype=torch.uint8, device=dev)
        codes, scales = F.quantize(U, W, T, workspace=ws, stream=stream)
        ms_q = timed(lambda: F.quantize(U, W, T, codes=codes, scales=scales, workspace=ws,
                                        stream=stream))
        code_bytes = T * 2 * n * m // 4
        traffic = (T + 1) * 2 * n * m * 8 + code_bytes
        once = 2 * n * m * 8 + code_bytes
        res["quantize"].append({"T": T, "us": round(ms_q * 1e3, 1), "bytes": traffic,
                                "gbs": round(traffic / (ms_q * 1e-3) / 1e9, 1),
                                "frac": round(traffic / (ms_q * 1e-3) / 1e9 / hbm, 4),
                                "one_read_gbs": round(once / (ms_q * 1e-3) / 1e9, 1)})
        del codes, scales, ws
    if F.get_status() != 0:
        raise RuntimeError("device status after the quantize timing")
    del R, U, W, flush
    torch.cuda.empty_cache()
    res["workload"] = f"{cols}->{rows} layer (complex {m}->{n}), fp32 weights"
    res["timing"] = "median of 5 CUDA-event times, L2 flushed before each"
    return res


def run_prefill(F, dev, steps: int, warmup: int):
    """Prefill GEMM on 2048 tokens: per layer and T, the median over `steps` launches, each timed
    alone (CUDA events on the launching stream) after a 256 MB L2 flush."""
    _, bf16, peak_kind = peaks()
    stream = torch.cuda.Stream(device=dev)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    rows_out, roof = [], None
    clocks = Clocks(torch.cuda.current_device())
    clocks.start()
    for (name, rows, cols, idx) in PREFILL_LAYERS:
        seed = synth.weight_seed("prefill", idx)
        R = synth.student_t_weight(rows, cols, seed, device=dev)
        U, W = F.convert(R)
        del R
        codes, scales = F.quantize(U, W, 3)     # stages 0..T-1 of a T = 3 quantization are the
        del U, W                                # T-stage quantization (prefix of the buffers)
        x = synth.outlier_activations(PREFILL_TOKENS, cols,
                                      synth.activation_seed(seed, PREFILL_TOKENS), device=dev)
        y = torch.empty((PREFILL_TOKENS, rows), dtype=torch.float32, device=dev)
        n, m = (rows + 1) // 2, (cols + 1) // 2
        # The set-up ran on the current stream (and y may reuse the blocks of U, W): the timed
        # launches on `stream` start after it.
        stream.wait_stream(torch.cuda.current_stream())
        for T in (1, 2, 3):
            times = []
            with torch.cuda.stream(stream):
                for i in range(warmup + steps):
                    flush.zero_()
                    e0 = torch.cuda.Event(enable_timing=True)
                    e1 = torch.cuda.Event(enable_timing=True)
                    e0.record(stream)
                    F.wl_matmul(x, codes, scales, rows, y=y, stream=stream, T=T)
                    e1.record(stream)
                    if i >= warmup:
                        times.append((e0, e1))
            stream.synchronize()
            st = F.get_status()
            if st != 0:
                raise RuntimeError(f"device status {st} after the prefill launches")
            us = statistics.median(a.elapsed_time(b) for a, b in times) * 1e3
            eff = 8.0 * n * m * PREFILL_TOKENS / (us * 1e-6) / 1e12
            mma = 2 * T * eff
            rows_out.append({"layer": f"{name} {cols}->{rows}", "T": T, "us": round(us, 1),
                             "effective_tops": round(eff, 1), "mma_tflops": round(mma, 1),
                             "tensor_frac": round(mma / bf16, 4)})
            if name == "up" and T == T_STAGES:
                roof = {"bound": "tensor", "achieved": round(mma, 1), "peak": bf16,
                        "unit": "TFLOP/s", "frac": round(mma / bf16, 4),
                        "traffic": int(PREFILL_T2_UP_DRAM_BYTES),
                        "ncu_tensor_pipe_active_pct": PREFILL_T2_UP_TENSOR_PIPE_PCT,
                        "peak_kind": f"{peak_kind} bf16_tflops (burst)",
                        "kernel": f"wl_prefill_kernel<{T}> (up {cols}->{rows}, "
                                  f"{PREFILL_TOKENS} tokens)"}
        del codes, scales, x, y
    clk = clocks.stop()
    del flush
    return {"workload": f"prefill {PREFILL_TOKENS} tokens x (4096->11008, 11008->4096), bf16 x",
            "metric": "effective TOPS = 8 n m B / time; MMA work 16 T n m B / time",
            "timing": "median of per-launch CUDA-event times, L2 flushed before each launch",
            "layers": rows_out, "roofline": roof, "clocks": clk,
            "gpu_launches": len(rows_out) * steps}


def run_lut(F):
    """The host look-up-table matmul (Sec. 3.4) on one 4096 -> 4096 linear (layer 0's q, codes
    made by the GPU quantizer), one int8 token, all host cores and one."""
    dev = torch.device("cuda", torch.cuda.current_device())
    rows, cols = 4096, 4096
    seed = synth.weight_seed("stack", 0, 0)
    R = synth.student_t_weight(rows, cols, seed, device=dev)
    U, W = F.convert(R)
    codes, scales = F.quantize(U, W, T_STAGES)
    codes, scales = codes.cpu(), scales.cpu()
    del R, U, W
    x = synth.outlier_activations(1, cols, synth.activation_seed(seed, 1)).float()
    xq, delta = F.lut_quantize_x(x)
    nb = layer_bytes(rows, cols, 1, x_bytes=1)
    out = {"workload": "4096->4096 linear (complex 2048->2048), T = 2, one int8 token",
           "unit": "GB/s (packed codes + scales + x + y)"}
    for label, nt in (("all_cores", os.cpu_count() or 1), ("one_thread", 1)):
        F.lut_matmul(xq, delta, codes, scales, rows, nthreads=nt)
        reps, t0 = 0, time.perf_counter()
        while True:
            F.lut_matmul(xq, delta, codes, scales, rows, nthreads=nt)
            reps += 1
            if time.perf_counter() - t0 > 1.0 or reps >= 200:
                break
        sec = (time.perf_counter() - t0) / reps
        out[label] = {"threads": nt, "us": round(sec * 1e6, 1),
                      "value": round(nb / sec / 1e9, 3)}
    return out


# --------------------------------------------------------------------------------------------
def _oracle_layer(rows, cols, seed, B):
    import oracle as O
    R = synth.student_t_weight(rows, cols, seed).numpy()
    U, W = O.convert(R)
    codes, scales = O.quantize(U, W, T_STAGES)
    x = synth.outlier_activations(B, cols, synth.activation_seed(seed, B)).float().numpy()
    return codes, scales, x


def _threads():
    try:
        from threadpoolctl import threadpool_info
        return max(int(i.get("num_threads", 1)) for i in threadpool_info()) or 1
    except Exception:
        if os.environ.get("OMP_NUM_THREADS") == "1":
            return 1
        return os.cpu_count() or 1


def oracle_sample(B: int, count: int = SAMPLE_LINEARS):
    """The oracle's inputs for the bounded sample: layer 0's first `count` linears at batch B."""
    shapes = layer_shapes(1)[:max(1, count)]
    return [(rows, cols, name, _oracle_layer(rows, cols, synth.weight_seed("stack", L, pi), B))
            for (L, pi, name, rows, cols) in shapes]


def time_oracle(prepared, budget_s: float):
    """Passes of the oracle's wl_matmul (float64 numpy, as it stands) over the sample until the
    time budget is used (at least one pass): GB/s of the algorithmic bytes."""
    import oracle as O
    B = prepared[0][3][2].shape[0]
    nbytes = sum(layer_bytes(r, c, B) for r, c, _, _ in prepared)
    passes, spent = 0, 0.0
    while passes == 0 or spent < budget_s:
        t0 = time.perf_counter()
        for rows, cols, _, (codes, scales, x) in prepared:
            O.wl_matmul(x, codes, scales, rows)
        spent += time.perf_counter() - t0
        passes += 1
    return nbytes * passes / spent / 1e9, passes, spent


def cpu_baseline(B: int, budget_s: float = 10.0, count: int = SAMPLE_LINEARS):
    """The oracle on the host cores: BLAS with its default threads (all cores) in this process,
    and one thread in a child process started with the thread-count variables set to 1."""
    prepared = oracle_sample(B, count)
    gbs, passes, spent = time_oracle(prepared, budget_s)
    names = ",".join(f"0.{nm}" for _, _, nm, _ in prepared)
    res = {"value": round(gbs, 5), "unit": "GB/s", "cores": _threads(), "kind": "oracle",
           "sample": f"oracle wl_matmul over linears {names} of the stack, batch {B}, "
                     f"{passes} passes ({spent:.1f} s); setup (oracle convert+quantize) untimed"}
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    try:
        out = subprocess.run([sys.executable, os.path.abspath(__file__), "--oracle-sample-only",
                              "--batch", str(B), "--cpu-budget", str(budget_s),
                              "--ref-linears", str(count)],
                             env=env, capture_output=True, text=True, timeout=600)
        one = json.loads(out.stdout.strip().splitlines()[-1])
        res["one_thread"] = {"value": one["value"], "unit": "GB/s", "cores": 1,
                             "sample": one["sample"]}
    except Exception as e:   # noqa: BLE001
        res["one_thread"] = {"unavailable": f"{type(e).__name__}"}
    return res


def run_reference(args, world, rank):
    if rank != 0:
        return None
    prepared = oracle_sample(args.batch, args.ref_linears)
    import oracle as O

    def step():
        for rows, cols, _, (codes, scales, x) in prepared:
            O.wl_matmul(x, codes, scales, rows)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    sec = time.perf_counter() - t0
    step_bytes = sum(layer_bytes(r, c, args.batch) for r, c, _, _ in prepared)
    value = step_bytes * args.steps / sec / 1e9
    names = ",".join(f"0.{nm}" for _, _, nm, _ in prepared)
    return {
        "impl": "reference", "metric": METRIC, "value": round(value, 5), "unit": "GB/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(sec / args.steps * 1e3, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic (same seeds as the GPU arm)",
        "config": {"workload": WORKLOAD, "layers": args.layers, "T": T_STAGES,
                   "batch": args.batch, "x_dtype": "bf16",
                   "sample_per_step": f"linears {names} (the bounded sample cpu_baseline times)"},
        "e2e": {"value": round(value, 5), "unit": "GB/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
        "cpu_baseline": {"value": round(value, 5), "unit": "GB/s", "cores": _threads(),
                         "kind": "oracle", "sample": f"linears {names} per step"},
    }


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=300)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--batch", type=int, default=1)
    ap.add_argument("--layers", type=int, default=32)
    ap.add_argument("--no-graph", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-budget", type=float, default=8.0)
    ap.add_argument("--ref-linears", type=int, default=SAMPLE_LINEARS,
                    help="linears of layer 0 in the oracle sample (cpu_baseline, reference arm)")
    ap.add_argument("--no-prefill", action="store_true")
    ap.add_argument("--no-sweep", action="store_true")
    ap.add_argument("--no-chain", action="store_true")
    ap.add_argument("--no-quantize", action="store_true")
    ap.add_argument("--no-lut", action="store_true")
    ap.add_argument("--ungrouped", action="store_true")
    ap.add_argument("--prefill-steps", type=int, default=10)
    ap.add_argument("--oracle-sample-only", action="store_true", help=argparse.SUPPRESS)
    ap.add_argument("--decode-path", type=int, default=0, choices=[0, 1, 4, 5],
                    help="decode kernel: 0 automatic, 1 warp-MMA, 4 persistent tcgen05, "
                         "5 chained kernel per call")
    args = ap.parse_args()
    if args.oracle_sample_only:
        prepared = oracle_sample(args.batch, args.ref_linears)
        gbs, passes, spent = time_oracle(prepared, args.cpu_budget)
        names = ",".join(f"0.{nm}" for _, _, nm, _ in prepared)
        print(json.dumps({"value": round(gbs, 5),
                          "sample": f"linears {names}, batch {args.batch}, {passes} passes "
                                    f"({spent:.1f} s), one thread"}))
        return
    world, rank, local = dist_setup()
    if args.impl == "reference":
        line = run_reference(args, world, rank)
    else:
        line = run_ours(args, world, rank, local)
    if rank == 0 and line is not None:
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
