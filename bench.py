#!/usr/bin/env python
"""Benchmark of the masked-linear hot path on one GB300.

Default workload (one step): one prefill of 512 tokens through a 28-layer
Llama-3.2-3B-shaped linear stack (per layer Q|K|V 3072 -> 5120, O 3072 ->
3072, Gate|Up 3072 -> 16384, Down 8192 -> 3072), fp32, Laplace noise at
eps = 1, each layer seeded on its own.  A step draws and adds the mask of every
input group of every layer (fused with the fp16 split the tensor-core product
reads), runs the masked products with the unmask fused into their epilogues
(Y = X~ W^T - C), and carries its share of the correction bank: each product
call multiplies the step's 512 masked rows together with the 512 noise rows of
the same draw of the next bank cycle (8 draws per cycle), whose products are
the corrections that cycle's step subtracts.  So any number of steps times the
whole method: prefill plus its correction.  ``--schedule banked`` runs the
separate bank instead (8 draws of corrections per group refilled beside the
steps on a lower-priority stream).  The weights (45 GB with their splits) are
far larger than L2.

Also reported on the same stack: the online prefill alone, the bank refill
alone, the product kernels per launch (the roofline), decode at one token per
step (tokens/s), the cancellation bound on every output of the first and last
layer, Down on its own (its binary32 output is dominated by cancellation,
which is why the paper keeps it in the enclave, and in binary64), the oracle
on the host cores (cpu_baseline) and end to end through host memory (e2e).

``--workload llama_layer`` is the one-layer, 128-token workload; the other
``--workload`` values measure the Qwen workloads, the LM head and the
comparators and print their own line.  ``--impl reference`` times the fp64
CPU oracle on a bounded sample of the same workload instead.
"""

import argparse
import faulthandler
import json
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "masked-linear TFLOP/s & ms/prefill (Llama-3B shapes), % of roofline, oracle match"
UNIT = "TFLOP/s"
TF32_OVER_BF16 = 1.1 / 2.25  # nominal dense TF32 : BF16 tensor rate on GB300
DRAWS = 8
STACK_LAYERS, STACK_TOKENS, STACK_SEED, STACK_INPUT_SEED = 28, 512, 7, 11


def stack_workload(layers, tokens, mech, eps):
    what = ("one llama-3.2-3b-shaped layer" if layers == 1 else
            f"llama-3.2-3b-shaped linear stack, {layers} layers")
    return (f"{what} (Q|K|V, O, Gate|Up, Down), prefill of {tokens} tokens, fp32, {mech} eps={eps:g}, per-layer "
            f"seeds, corrections precomputed in banks of {DRAWS} draws (each step carries 1/{DRAWS} of the next "
            f"cycle's banks)")


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=24)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--eps", type=float, default=1.0)
    ap.add_argument("--path", default="auto")
    ap.add_argument("--tokens", type=int, default=None, help="rows per step (stack: 512, llama_layer: 128)")
    ap.add_argument("--layers", type=int, default=STACK_LAYERS, help="layers of the stack workload")
    ap.add_argument("--mech", default=None, help="noise law (stack: laplace, llama_layer: gaussian)")
    ap.add_argument("--cpu-sample-rows", type=int, default=4)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-decode", action="store_true", help="stack: skip the one-token decode measurement")
    ap.add_argument("--decode-steps", type=int, default=256)
    ap.add_argument("--rows", type=str, default=None,
                    help="qwen_sweep: comma-separated row counts (default 1,4,16,64,256,1024; the mask measured "
                         "on 10^9 elements only with the default)")
    ap.add_argument("--schedule", choices=["stacked", "banked"], default="stacked",
                    help="stack workload: stacked (each product also computes the next cycle's correction of its "
                         "draw) or banked (the next cycle's banks of 1/8 of the layers beside each step)")
    ap.add_argument("--workload", default="llama_stack",
                    choices=["llama_stack", "llama_layer", "llama_stack_detail", "qwen_stack", "qwen_sweep",
                             "down_fp64", "slalom", "lm_head"],
                    help="llama_stack (default): the headline line; llama_layer: one layer at 128 tokens; the "
                         "others measure the other workloads and print their own line")
    a = ap.parse_args(argv)
    if a.workload == "llama_layer":  # one layer of the same stack code, at 128 tokens, no decode
        a.layers = 1
        a.no_decode = True
    if a.tokens is None:
        a.tokens = STACK_TOKENS if a.workload == "llama_stack" else 128
    if a.mech is None:
        a.mech = "laplace" if a.workload == "llama_stack" else "gaussian"
    return a


def peaks():
    p = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            m = json.load(f)
        p.update({k: float(m[k]) for k in ("hbm_gbs", "bf16_tflops", "bf16_tflops_sustained") if k in m})
        p["source"] = "measured"
    except (OSError, ValueError, KeyError):
        pass
    return p


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.proc = None
        time.sleep(0.3)
        return self

    def __exit__(self, *exc):
        if self.proc is None:
            return
        time.sleep(0.2)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        self.lines = [l for l in out.splitlines() if l.strip()]

    def summary(self):
        if self.proc is None or not getattr(self, "lines", None):
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in self.lines:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 7:
                continue
            try:
                sm.append(float(parts[0]))
                smax.append(float(parts[1]))
            except ValueError:
                continue
            for n, v in zip(names, parts[3:7]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        loaded = [s for s in sm if s > 0.5 * max(sm)] or sm
        return {"sm_mhz": statistics.median(loaded), "sm_max_mhz": max(smax), "reasons": sorted(reasons),
                "samples": len(sm)}


def profiled_traffic(profile="tc_gemm_fp16x3_llama_online_and_bank.md", field="traffic_bytes_per_step"):
    """A DRAM byte count from a committed ncu summary, if it was taken on the current tensor-core
    kernel source (else None)."""
    import hashlib
    prof = os.path.join(ROOT, "profiles", profile)
    src = os.path.join(ROOT, "paper_2609_15039_gb300", "csrc", "gemm_tc.cu")
    try:
        fields = dict(line.split(":", 1) for line in open(prof).read().splitlines()
                      if line.startswith((field + ":", "kernel_source_sha256_prefix:")))
        digest = hashlib.sha256(open(src, "rb").read()).hexdigest()
    except (OSError, ValueError):
        return None, "no profile"
    if not digest.startswith(fields.get("kernel_source_sha256_prefix", "-").strip()):
        return None, "kernel changed since the ncu capture"
    if field not in fields:
        return None, "no such figure in the profile"
    return float(fields[field]), "ncu capture of the same kernel source (profiles/" + profile + ")"


def max_over_ranks(x, device):
    """The job's figure for a per-rank time: the largest over the ranks (one replica per GPU, so the
    job is as slow as its slowest replica); x itself when the job has one rank."""
    import torch
    import torch.distributed as dist
    if not dist.is_initialized() or dist.get_world_size() == 1:
        return x
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_rate(world, units_per_step, ms):
    """Whole-job rate of `world` replicas that each do units_per_step in ms per step (weak scaling:
    the work per rank is fixed, the job's grows with the ranks)."""
    return world * units_per_step / (ms * 1e-3)


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


# ----------------------------------------------------------------------------- reference arm
def oracle_sample(model, M, rows, eps, mech, seed, deltas, weights_cpu, inputs_cpu, offsets=None):
    """The oracle on the first ``rows`` tokens of every group: noise, mask, products, unmask.
    offsets: {group: first Philox block of the draw} (default 0)."""
    from oracle import linear, philox
    out = {}
    flops = 0
    for gi, (g, K, names) in enumerate(model.input_groups()):
        X = inputs_cpu[g][:rows]
        off = (offsets or {}).get(g, 0)
        eta = philox.noise((rows, K), deltas[g], eps, mech, seed, stream_id=gi, offset=off)
        Xt = linear.mask(X, eta)
        for name in names:
            W = weights_cpu[name]
            r = linear.masked_linear(Xt, W)
            C = linear.precompute_noise_product(eta, W)
            out[name] = linear.unmask(r.astype("float32"), C.astype("float32"))
            flops += 2 * 2 * rows * K * W.shape[0]
    return out, flops


def cpu_setup(model, M, weight_seed=None, input_seed=None):
    """Seeded inputs of one layer on the host (the stack's layer 0 when seeds are given, else the
    one-layer workload's), and the noise scales of Thms. 1-3 from the oracle."""
    import numpy as np
    from oracle import sensitivity as osens
    from paper_2609_15039_gb300 import workloads as wl
    if weight_seed is None:
        weights = {name: wl.weight(N, K, seed=200 + pi).numpy() for pi, (name, K, N, g) in
                   enumerate(model.projections())}
        inputs = {g: wl.activations(M, K, seed=100 + gi).numpy() for gi, (g, K, _n) in
                  enumerate(model.input_groups())}
    else:
        weights = {name: wl.weight(N, K, seed=wl.layer_seed(weight_seed, 0, pi)).numpy()
                   for pi, (name, K, N, g) in enumerate(model.projections())}
        inputs = {g: wl.activations(M, K, seed=wl.layer_seed(input_seed, 0, 50 + gi)).numpy()
                  for gi, (g, K, _n) in enumerate(model.input_groups())}
    ones = np.ones(model.d_model)
    norms = {n: osens.spectral_norm(weights[n], iters=30) for n in ("v", "up", "gate")}
    deltas = {"qkv": osens.delta_layernorm(ones), "gateup": osens.delta_layernorm(ones),
              "o": osens.delta_attention(ones, norms["v"]),
              "down": osens.delta_activation(ones, None, model.d_ff, norms["up"], norms["gate"])}
    return weights, inputs, deltas


def run_reference(args):
    """The fp64 CPU oracle, as it stands, on a bounded sample of the workload's step: the first
    rows of every input group of one layer per step (stack: its layer 0)."""
    world, rank, _ = dist_env()
    if rank != 0:
        return
    from paper_2609_15039_gb300 import workloads as wl
    model, M = wl.LLAMA_3_2_3B, args.tokens
    weights, inputs, deltas = cpu_setup(model, M, STACK_SEED, STACK_INPUT_SEED)
    workload = stack_workload(args.layers, M, args.mech, args.eps)
    rows = args.cpu_sample_rows
    for w in range(args.warmup):
        oracle_sample(model, M, rows, args.eps, args.mech, 1000 + w, deltas, weights, inputs)
    t0 = time.perf_counter()
    flops = 0
    for s in range(args.steps):
        _, f = oracle_sample(model, M, rows, args.eps, args.mech, 2000 + s, deltas, weights, inputs)
        flops += f
    dt = time.perf_counter() - t0
    value = flops / dt / 1e12
    sample = (f"first {rows} of {M} tokens of every input group of one layer (all 7 projections: noise, mask, "
              f"masked product, correction, unmask in fp64) per step")
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": workload, "tokens": M, "eps": args.eps, "mech": args.mech},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }))


# ----------------------------------------------------------------------------- our arm
def run_workload(args):
    """bench.py --workload llama_stack | qwen_stack | qwen_sweep: one JSON line of that workload."""
    import torch
    from paper_2609_15039_gb300 import measure
    world, rank, local = dist_env()
    torch.cuda.set_device(local)
    with ClockSampler(local) as clocks:
        if args.workload == "qwen_sweep" and args.rows:
            res = measure.qwen_sweep(Ms=tuple(int(m) for m in args.rows.split(",")), mask_elements=10 ** 6)
        else:
            res = measure.WORKLOADS[args.workload]()
    if args.workload == "llama_stack_detail":
        value, unit, ms = res["prefill"]["tflops"], UNIT, res["prefill"]["ms_per_prefill"]
    elif args.workload == "qwen_stack":
        first = next(iter(res["prefill"].values()))
        value, unit, ms = first["tflops"], UNIT, first["ms_per_prefill"]
    elif args.workload == "slalom":
        first = next(iter(res["compare"].values()))["qkv"]
        value, unit, ms = first["slalom_us"] / first["ours_us"], "slalom time / this path's time (QKV)", \
            first["ours_us"] / 1e3
    elif args.workload == "down_fp64":
        first = next(iter(res["down"].values()))["binary64"]
        value, unit, ms = first["mean_err"], "mean abs error of the recovered Down output", first["us_per_call"] / 1e3
    elif args.workload == "lm_head":
        first = next(iter(res["lm_head"].values()))
        value, unit, ms = first["tflops"], UNIT, first["ms_per_step"]
    else:
        last = list(res["sweep"].values())[-1]
        value, unit, ms = last["tflops"], UNIT, last["online_ms"]
    if rank == 0:
        print(json.dumps({"metric": METRIC, "value": value, "unit": unit, "n_gpus": world, "ms_per_step": ms,
                          "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
                          "data": "synthetic", "config": {"workload": res.pop("workload")}, "clocks": clocks.summary(),
                          **res}))


def main():
    faulthandler.enable()  # a crash in native code prints the Python stack to stderr
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    if args.workload in ("llama_stack", "llama_layer"):
        return run_llama_stack(args)
    return run_workload(args)


def phase(msg):
    """Progress of the run on stderr (the JSON line goes to stdout)."""
    sys.stderr.write(f"[bench {time.strftime('%H:%M:%S')}] {msg}\n")
    sys.stderr.flush()


def path_peaks(pk):
    """Algorithmic flops per second at each path's instruction peak: FP16X3 = the measured
    sustained bf16 rate (fp16 runs at the bf16 rate) / 3 products per term; TF32X3 = that x the
    nominal TF32 : bf16 ratio; FP32 = 152 SMs x 128 lanes x 2 flops x 2.07 GHz (derived)."""
    return {"fp16x3": pk["bf16_tflops_sustained"] / 3.0,
            "tf32x3": pk["bf16_tflops_sustained"] * TF32_OVER_BF16 / 3.0,
            "fp32": 152 * 128 * 2 * 2.07e9 / 1e12}


PEAK_NOTE = ("fp16x3 = measured sustained bf16 (fp16 runs at the bf16 rate) / 3 products per term; tf32x3 = that x "
             "the nominal tf32/bf16 ratio (1.1/2.25, not measured); fp32 FMA = 152 SMs x 128 lanes x 2 flop x "
             "2.07 GHz (derived); hbm = measured copy bandwidth")


def _time_graphs(graph_of, s0, n, stream):
    """Replays graph_of(s) for s = s0 .. s0 + n - 1 with a CUDA event after each; per-step ms."""
    import torch
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    ev[0].record(stream)
    for i in range(n):
        graph_of(s0 + i).replay()
        ev[i + 1].record(stream)
    torch.cuda.synchronize()
    return [ev[i].elapsed_time(ev[i + 1]) for i in range(n)]


def run_llama_stack(args):
    """The headline line: prefill of 512 tokens through the 28-layer Llama-3.2-3B-shaped stack, each
    step carrying its share of the next bank cycle (see the module docstring)."""
    import numpy as np
    import torch
    import torch.distributed as dist
    from paper_2609_15039_gb300 import measure, spl, workloads as wl
    from paper_2609_15039_gb300.layer import MaskedStack, StackIO

    world, rank, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    model, L, M, D, mech, eps, path = wl.LLAMA_3_2_3B, args.layers, args.tokens, DRAWS, args.mech, args.eps, args.path
    stacked = args.schedule == "stacked"
    pk = peaks()
    ppk = path_peaks(pk)
    t_build = time.perf_counter()
    phase("building the stack")
    stack = MaskedStack.build(model, L, M, D, base_seed=STACK_SEED, device=dev, path=path, stacked=stacked)
    inputs = stack.inputs(STACK_INPUT_SEED, device=dev)
    layer0 = stack.layers[0]
    groups = layer0.groups
    if path == "auto":
        # a8 is evaluated per (shape, eps): on layer 0's weights and a masked sample of its input, and
        # the choice kept for every layer of the same shapes
        layer0.calibrate(inputs[0], eps, mech, stack.seeds[0])
        for layer in stack.layers[1:]:
            layer.paths = dict(layer0.paths)
        if stacked:  # the buffers follow the chosen paths
            for layer in stack.layers:
                layer.allocate_stacked(M, D, path, workspace=layer.workspace)
    rows = 2 * M if stacked else M  # rows of every product call
    if stacked:
        group_paths = {g.name: layer0.stacked[g.name]["path"] for g in groups}
    else:
        group_paths = {g.name: spl.PATH_NAMES[spl.spl_resolve_path(M, g.K, g.N, layer0.path_of(g, path, M))]
                       for g in groups}
    bank_ws = None if stacked else spl.workspace(max(l.workspace_bytes(M, D, path) for l in stack.layers), dev)
    stream = torch.cuda.current_stream(dev)
    for li, layer in enumerate(stack.layers):  # sets up every library call before capture
        if stacked:
            layer.stacked_step(inputs[li], eps, mech, stack.seeds[li], 0, 0, path=path)
        else:
            layer.refill(eps, mech, stack.seeds[li], 0, path=path)
            layer.online(inputs[li], eps, mech, stack.seeds[li], 0, 0, path=path)
    torch.cuda.synchronize()
    build_s = time.perf_counter() - t_build

    flops_layer = {g.name: 2 * M * g.K * g.N for g in groups}  # the masked product (online rows)
    flops_step = L * sum(flops_layer.values())  # the masked products of one prefill (algorithmic)

    # ---- the timed steps -----------------------------------------------------------------------
    phase("capturing the step graphs")
    if stacked:
        graphs, glaunch = stack.capture_stacked(inputs, eps, mech, path=path)
    else:
        graphs, glaunch = stack.capture_steps(inputs, eps, mech, bank_ws, path=path)
    graph_of = lambda s: graphs[(s // D) % 2][s % D]
    launches_of = lambda s: glaunch[(s // D) % 2][s % D]

    def prime(cycle):
        """Device-side Philox bases at ``cycle`` and that cycle's corrections in place."""
        if stacked:
            stack.start_stacked(cycle, graphs)
        else:
            stack.set_cycle(cycle)
            stack.refill_all(eps, mech, path, parity=cycle % 2, workspace=bank_ws)

    s = 2 * D  # every pass starts at a bank cycle
    phase("timed steps")
    prime(s // D)
    for _ in range(args.warmup):
        graph_of(s).replay()
        s += 1
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    t_start, t_end = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    s_timed = s
    with ClockSampler(local) as clocks:
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_push("timed")
        t_start.record(stream)
        for _ in range(args.steps):
            graph_of(s).replay()
            s += 1
        t_end.record(stream)
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_pop()
    if world > 1:
        dist.barrier()
    ms = max_over_ranks(t_start.elapsed_time(t_end) / args.steps, dev)
    gpu_launches = sum(launches_of(s_timed + i) for i in range(args.steps))
    st = spl.spl_get_device_status()
    if st != spl.SPL_OK:
        raise RuntimeError("device status " + spl.status_string(st))
    value = job_rate(world, flops_step, ms) / 1e12

    # ---- the product calls alone: CUDA event pairs around each, in graphs of the same steps ------
    ev = {}
    ev_alive = []  # every event recorded into a graph lives as long as the graph (a graph of both parities
                   # records its own events; the dict keeps the last captured ones)

    def timer(d, li, phase_, kind, group):
        if kind != "masked_linear_unmask":
            return
        e = torch.cuda.Event(enable_timing=True, external=True)
        e.record()
        ev_alive.append(e)
        ev.setdefault((d, li, group), [None, None])[0 if phase_ == "begin" else 1] = e

    phase("per-call timing pass")
    if stacked:
        ev_graphs, _ = stack.capture_stacked(inputs, eps, mech, path=path, timer=timer)
        c = -(-s // D) + 1
        stack.start_stacked(c, ev_graphs)
        for d in range(D):  # one cycle: each graph's events hold its last replay
            ev_graphs[c % 2][d].replay()
        torch.cuda.synchronize()
        s = (c + 1) * D
    else:
        ev_graphs, _ = stack.capture(inputs, eps, mech, path=path, refill=False, timer=timer)
        stack.set_cycle(1)
        _time_graphs(lambda i: ev_graphs[i % D], 0, D, stream)
    per_group = {}
    for (d, li, gname), (b, e) in ev.items():
        per_group.setdefault(gname, []).append(b.elapsed_time(e))
    del ev_graphs
    del ev_alive
    prod = {}
    for g in groups:
        t = per_group[g.name]
        avg = sum(t) / len(t)
        f = 2 * rows * g.K * g.N
        pp = ppk[group_paths[g.name]]
        prod[g.name] = {"calls": len(t), "rows": rows, "avg_us": 1e3 * avg, "tflops": f / (avg * 1e-3) / 1e12,
                        "path": group_paths[g.name], "peak": pp, "frac": f / (avg * 1e-3) / 1e12 / pp}
    prod_ms_layer = sum(p["avg_us"] for p in prod.values()) / 1e3
    call_flops_layer = sum(2 * rows * g.K * g.N for g in groups)
    prod_peak = call_flops_layer / sum(2 * rows * g.K * g.N / ppk[group_paths[g.name]] for g in groups)
    achieved = call_flops_layer / (prod_ms_layer * 1e-3) / 1e12
    traffic, traffic_note = (profiled_traffic("tc_stacked_fp16x3_llama_1024.md", "traffic_bytes_per_launch")
                             if stacked else
                             profiled_traffic("tc_prefill_fp16x3_llama_512.md", "traffic_bytes_per_launch"))
    what = (f"one call per input group and layer: the {M} masked rows of the step and, in the same launch, the "
            f"{M} noise rows of the next cycle's draw (their corrections), {rows} rows" if stacked else
            f"one call per input group and layer, {M} rows")
    roofline = {
        "bound": "tensor", "achieved": achieved, "peak": prod_peak, "unit": "TFLOP/s", "frac": achieved / prod_peak,
        "traffic": traffic,
        "kernel": ("tc_persistent_kernel / tc_gemm_kernel (FP16X3 on tcgen05) with the fused unmask: " + what +
                   f"; {len(groups) * L} calls per step"),
        "flops_per_launch": call_flops_layer / len(groups), "avg_launch_us": 1e3 * prod_ms_layer / len(groups),
        "per_group": prod, "share_of_step": L * prod_ms_layer / ms,
        "timing": ("CUDA event pairs (external event nodes, on the launching stream) around every product call of "
                   f"the {L} layers in graph-replayed steps (one bank cycle, {D} steps); achieved = the calls' "
                   "algorithmic flops (2 x rows x K x N) / their summed durations"),
        "traffic_note": traffic_note + "; DRAM bytes per call, averaged over the four calls of a layer",
        "peak_source": pk["source"], "peak_note": "sustained peak (the calls run back to back through the timed "
                                                  "steps); " + PEAK_NOTE}

    # ---- end to end: the same steps with every layer's input copied in from pinned host memory
    # and every output copied back, beside each step's graph, on a copy stream ------------------
    e2e = None
    if not args.no_e2e and stacked:
        phase("end-to-end pass")
        # every step copies its inputs of every layer in from page-locked host memory and its outputs
        # of every layer back (StackIO: one copy per input group in, one strided copy per group out,
        # the two directions on their own streams beside the graph replays); the last step's outputs
        # reach the host inside the timed region
        host_in = {g: torch.stack([inp[g] for inp in inputs]).cpu().pin_memory() for g in inputs[0]}
        io = StackIO(stack, host_in)
        h2d, d2h = io.bytes_per_step()
        e2e_graphs, _ = stack.capture_stacked(io.layer_inputs(), eps, mech, path=path)
        s = -(-s // D) * D + D
        stack.start_stacked(s // D, e2e_graphs)
        s_timed = s + max(2, args.warmup)
        while s < s_timed:  # no warm-up step copies in a timed step's inputs
            io.step(e2e_graphs, s, stop=s_timed)
            s += 1
        io.finish()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(args.steps):  # each timed step's inputs in and outputs out inside the region
            io.step(e2e_graphs, s, stop=s_timed + args.steps)
            s += 1
        io.finish()
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(e0.elapsed_time(e1) / args.steps, dev)
        e2e = {"value": job_rate(world, flops_step, e2e_ms) / 1e12, "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
               "copies": ("page-locked host memory; per step one copy in per input group (every layer's rows) and "
                          "one strided copy out per group (every layer's Y rows), inputs and outputs on their own "
                          f"streams beside the graph replays, inputs up to {io.sets - 1} steps ahead (StackIO); "
                          "every timed step's inputs go in and its outputs reach the host inside the timed region")}
        del e2e_graphs, io, host_in
    st = spl.spl_get_device_status()
    if st != spl.SPL_OK:
        raise RuntimeError("device status " + spl.status_string(st))

    # ---- the cancellation bound over every output of the first and last layer (an eager step) ---
    phase("bound check")
    check_cycle = -(-s // D) + 1
    check_outs = {}
    if stacked:
        stack.start_stacked(check_cycle, graphs)  # this cycle's corrections in place
        bound = {}
        for li in sorted({0, L - 1}):
            layer = stack.layers[li]
            outs = layer.stacked_step(inputs[li], eps, mech, stack.seeds[li], 0, check_cycle % 2, cycle=check_cycle,
                                      path=path)
            check_outs[li] = outs
            bc = layer.bound_check(inputs[li], outs, eps, mech, stack.seeds[li], check_cycle, 0)
            bound[f"layer{li}"] = {g: {"max_err_over_hard": v["max_err_over_hard"],
                                       "log_violation_pct": v["violation_pct"], "mean_err": v["mean_err"],
                                       "max_rel_err": v["max_err"] / v["max_abs_ref"] if v["max_abs_ref"] else 0.0}
                                   for g, v in bc.items()}
    else:
        bound = measure._bound(stack, inputs, eps, mech, 3 * D + 1, [0, L - 1])
        for lk, groups_bc in bound.items():
            for gname, v in groups_bc.items():
                v.pop("mean_log_bound", None)

    # ---- Down on its own path (Sec. 5.5): binary32 (the step's) and binary64, layer 0 -----------
    phase("binary64 Down")
    down = {}
    gd = layer0.group("down")
    gi = [g.name for g in groups].index("down")
    Xd = inputs[0]["down"]
    delta = layer0.deltas["down"]
    eta = torch.empty((M, gd.K), device=dev)
    xt64 = torch.empty((M, gd.K), dtype=torch.float64, device=dev)
    spl.spl_noise(eta, delta, eps, mech, stack.seeds[0], stream_id=gi, offset=0)
    spl.spl_noise_mask_f64(xt64, Xd, delta, eps, mech, stack.seeds[0], stream_id=gi, offset=0)
    ws64 = spl.workspace(spl.spl_f64_workspace_bytes(M, gd.K, gd.N), dev)
    C64 = torch.empty((M, gd.N), dtype=torch.float64, device=dev)
    spl.spl_precompute_noise_product_f64(C64, eta, gd.W, workspace=ws64)
    Y64 = torch.empty((M, gd.N), device=dev)
    spl.spl_masked_linear_unmask_f64(Y64, xt64, gd.W, C64, workspace=ws64)  # warm-up
    torch.cuda.synchronize()
    d0, d1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    d0.record(stream)
    spl.spl_masked_linear_unmask_f64(Y64, xt64, gd.W, C64, workspace=ws64)
    d1.record(stream)
    torch.cuda.synchronize()
    bc64 = spl.spl_bound_check(Y64, Xd, xt64.float().contiguous(), eta, gd.W)
    b32 = bound["layer0"]["down"]
    down = {"note": ("the paper keeps Down in the enclave (Sec. 5.5): its Delta (Thm. 3) is ~3e8, so the "
                     "binary32 recovered output is dominated by cancellation error, though inside the bound"),
            "binary32": {"path": group_paths["down"], "us_per_call": prod["down"]["avg_us"],
                         "rows_per_call": rows, "tflops": prod["down"]["tflops"], "max_rel_err": b32["max_rel_err"],
                         "mean_err": b32["mean_err"], "max_err_over_hard": b32["max_err_over_hard"]},
            "binary64": {"ms_per_call": d0.elapsed_time(d1), "rows": M,
                         "tflops": flops_layer["down"] / (d0.elapsed_time(d1) * 1e-3) / 1e12,
                         "max_rel_err": bc64["max_err"] / bc64["max_abs_ref"] if bc64["max_abs_ref"] else 0.0,
                         "mean_err": bc64["mean_err"]}}
    del eta, xt64, C64, Y64, ws64
    six = [n for n in prod if n != "down"]
    six_flops = sum(2 * rows * gg.K * gg.N for gg in groups if gg.name in six)
    six_ms = sum(prod[n]["avg_us"] for n in six) / 1e3
    offloaded = {"projections": "Q, K, V, O, Gate, Up", "tflops": six_flops / (six_ms * 1e-3) / 1e12,
                 "frac": six_flops / (six_ms * 1e-3) / 1e12 /
                 (six_flops / sum(2 * rows * gg.K * gg.N / ppk[group_paths[gg.name]] for gg in groups
                                  if gg.name in six)),
                 "max_rel_err": max(bound[lk][n]["max_rel_err"] for lk in bound for n in six),
                 "max_err_over_hard": max(bound[lk][n]["max_err_over_hard"] for lk in bound for n in six),
                 "timing": "product calls alone, from the roofline's event pairs"}

    # ---- cpu baseline + oracle match on the first rows of layer 0 (rank 0, N = 1 only) -----------
    cpu = match = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        phase("oracle on the host cores")
        from oracle import bounds, linear, philox
        nrows = args.cpu_sample_rows
        seed0 = stack.seeds[0]
        if stacked:
            cycle, d = check_cycle, 0
            outs = check_outs[0]
        else:
            cycle, d = 5, 3
            layer0.refill(eps, mech, seed0, cycle, path=path)
            outs = layer0.online(inputs[0], eps, mech, seed0, cycle, d, path=path)
        torch.cuda.synchronize()
        gpu_rows = {g: outs[g][:nrows].double().cpu().numpy() for g in outs}
        w_cpu = {g.name: g.W.cpu().numpy() for g in groups}
        x_cpu = {g: x[:nrows].cpu().numpy() for g, x in inputs[0].items()}
        t0, flops, reps, worst = time.perf_counter(), 0, 0, 0.0
        while True:
            for gi, g in enumerate(groups):
                X = x_cpu[g.name]
                eta = philox.noise((nrows, g.K), layer0.deltas[g.name], eps, mech, seed0, stream_id=gi,
                                   offset=layer0.block_offset(g, cycle, d))
                Xt = linear.mask(X, eta)
                r = linear.masked_linear(Xt, w_cpu[g.name])
                C = linear.precompute_noise_product(eta, w_cpu[g.name])
                linear.unmask(r.astype(np.float32), C.astype(np.float32))
                flops += 2 * 2 * nrows * g.K * g.N
                if reps == 0:
                    S = linear.abs_products(X, Xt, eta, w_cpu[g.name])
                    err = np.abs(gpu_rows[g.name] - linear.reference_output(X, w_cpu[g.name]))
                    worst = max(worst, float(np.max(err / bounds.hard_bound(*S, g.K))))
            reps += 1
            if time.perf_counter() - t0 > 10.0 or reps >= 50:
                break
        dt = time.perf_counter() - t0
        cpu = {"value": flops / dt / 1e12, "unit": UNIT, "cores": os.cpu_count(), "kind": "oracle", "seconds": dt,
               "sample": (f"first {nrows} of {M} tokens of every input group of layer 0 (all 7 projections: "
                          f"noise, mask, masked product, correction, unmask in fp64), {reps} repetitions; the rate "
                          f"is the sample's flops over its time")}
        match = {"rows_checked": nrows, "layer": 0, "max_err_over_hard_bound": worst, "pass": worst <= 1.0}

    # ---- the online prefill alone (masked products of 512 rows, no correction work) --------------
    phase("online prefill alone")
    del graphs
    torch.cuda.synchronize()
    for layer in stack.layers:
        layer.stacked = None
    torch.cuda.empty_cache()
    ws_on = spl.workspace(max(l.workspace_bytes(M, 1, path) for l in stack.layers), dev)
    for layer in stack.layers:
        layer.allocate(M, 1, path, workspace=ws_on)
    for li, layer in enumerate(stack.layers):
        layer.online(inputs[li], eps, mech, stack.seeds[li], 0, 0, path=path)
    torch.cuda.synchronize()
    on_graphs, on_launch = stack.capture(inputs, eps, mech, path=path, refill=False)
    stack.set_cycle(1)
    _time_graphs(lambda i: on_graphs[0], 0, 3, stream)
    on_times = _time_graphs(lambda i: on_graphs[0], 0, 8, stream)
    ms_online = sum(on_times) / len(on_times)
    del on_graphs

    # ---- decode at one token per step (the same layers, banks of D one-row draws) -----------------
    decode = None
    if not args.no_decode and stacked:
        phase("decode (stacked)")
        torch.cuda.synchronize()
        ws1 = spl.workspace(max(spl.spl_linear_workspace_bytes(2, g.K, g.N, "auto") for g in groups), dev)
        for layer in stack.layers:
            layer.allocate_stacked(1, D, workspace=ws1)
        del ws_on
        torch.cuda.empty_cache()
        inputs1 = stack.inputs(13, device=dev)
        dgraphs, dl = stack.capture_stacked(inputs1, eps, mech)
        dgraph_of = lambda s: dgraphs[(s // D) % 2][s % D]
        steps = max(D, args.decode_steps)
        stack.start_stacked(1, dgraphs)
        _time_graphs(dgraph_of, D, 2 * D, stream)  # cycles 1 and 2
        torch.cuda.nvtx.range_push("decode")
        times = _time_graphs(dgraph_of, 3 * D, steps, stream)
        torch.cuda.nvtx.range_pop()
        step_ms = sum(times) / steps
        dpaths = {g.name: layer0.stacked[g.name]["path"] for g in groups}
        step_bytes = sum(4 * g.K * g.N + 12 * g.K + 12 * g.N for g in groups) * L
        decode = {"steps": steps, "ms_per_token": step_ms, "tokens_per_s": 1e3 / step_ms,
                  "gbs": step_bytes / (step_ms * 1e-3) / 1e9, "peak_gbs": pk["hbm_gbs"],
                  "frac": step_bytes / (step_ms * 1e-3) / 1e9 / pk["hbm_gbs"], "bytes_per_step": step_bytes,
                  "paths": dpaths, "kernels_per_step": sum(sum(p) for p in dl) / (2 * D),
                  "fused_one_launch": all(layer0.stacked[g.name]["fused_mask"] for g in groups),
                  "schedule": ("stacked, one graph per token: every group's call draws the token's noise and the "
                               "next cycle's same-draw noise row, masks and multiplies both rows in one launch "
                               "of the decode kernel (bytes per step: every weight once, the token's x, C and Y, "
                               "both rows of x~ and the new correction)")}
        del dgraphs
        st = spl.spl_get_device_status()
        if st != spl.SPL_OK:
            raise RuntimeError("device status " + spl.status_string(st))
    elif not args.no_decode:
        phase("decode")
        torch.cuda.synchronize()
        ws1 = spl.workspace(max(l.workspace_bytes(1, D) for l in stack.layers), dev)
        for layer in stack.layers:
            layer.allocate(1, D, workspace=ws1)
        del ws_on
        torch.cuda.empty_cache()
        inputs1 = stack.inputs(13, device=dev)
        stack.step(inputs1, eps, mech, 0)
        torch.cuda.synchronize()
        bank_ws1 = spl.workspace(max(l.workspace_bytes(1, D) for l in stack.layers), dev)
        ov_graphs, ol = stack.capture_overlapped(inputs1, eps, mech, bank_ws1)
        cycles = max(1, -(-args.decode_steps // D))
        stack.start_overlapped(1, eps, mech)
        _time_graphs(lambda i: ov_graphs[(1 + i) % 2], 0, 2, stream)  # cycles 1 and 2
        times = _time_graphs(lambda i: ov_graphs[(3 + i) % 2], 0, cycles, stream)
        step_ms = sum(times) / (cycles * D)
        dpaths = {g.name: spl.PATH_NAMES[spl.spl_resolve_path(1, g.K, g.N, layer0.path_of(g, "auto", 1))]
                  for g in groups}
        step_bytes = sum(4 * g.K * g.N + 4 * g.K + 8 * g.N for g in groups) * L * (1 + 1.0 / D)
        decode = {"steps": cycles * D, "ms_per_token": step_ms, "tokens_per_s": 1e3 / step_ms,
                  "gbs": step_bytes / (step_ms * 1e-3) / 1e9, "peak_gbs": pk["hbm_gbs"],
                  "frac": step_bytes / (step_ms * 1e-3) / 1e9 / pk["hbm_gbs"], "bytes_per_step": step_bytes,
                  "paths": dpaths, "kernels_per_step": sum(ol) / len(ol) / D,
                  "schedule": ("whole-cycle graphs: each cycle's 8 one-token steps through every layer, and beside "
                               "them on a lower-priority stream the next cycle's corrections (bytes per step: every "
                               "weight once, x~, C and Y, plus 1/8 of the bank's weight reads)")}
        del ov_graphs
        st = spl.spl_get_device_status()
        if st != spl.SPL_OK:
            raise RuntimeError("device status " + spl.status_string(st))

    path_name = "+".join(sorted(set(group_paths.values())))
    schedule_note = (f"stacked: every product call multiplies the step's {M} masked rows and the {M} noise rows of "
                     f"the next cycle's same draw in one launch of {2 * M} rows, so each step computes 1/{D} of the "
                     "next cycle's corrections, summed exactly as the rows they will unmask"
                     if stacked else
                     f"banked: each step computes the next cycle's corrections of 1/{D} of the layers ({D} draws x "
                     f"{M} rows per group) on a lower-priority stream beside its prefill")
    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": ms, "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32",
        "path": path_name, "data": "synthetic",
        "config": {"workload": stack_workload(L, M, mech, eps), "layers": L, "tokens": M, "eps": eps, "mech": mech,
                   "bank_draws": D, "flops_per_step": flops_step,
                   "value": (f"algorithmic flops of the prefill's masked products (2 M K N per projection, {L} "
                             "layers) per second of the whole step: the prefill with its correction work"),
                   "bank_schedule": schedule_note,
                   "online_noise": "drawn again in each step's mask from the bank's Philox counters",
                   "l2": (f"weights {L * sum(g.K * g.N for g in groups) * 16 / 1e9:.1f} GB per step (fp32 + their "
                          "TF32 and fp16 splits) > 129 MB L2 (no flush needed)"),
                   "parallelism": "replicas" if world > 1 else "single", "setup_s": build_s},
        "prefill": {"ms_per_prefill_with_correction": ms, "tokens_per_s": M / (ms * 1e-3),
                    "online_only": {"ms_per_prefill": ms_online, "tflops": flops_step / (ms_online * 1e-3) / 1e12,
                                    "frac": flops_step / (ms_online * 1e-3) / 1e12 / prod_peak,
                                    "tokens_per_s": M / (ms_online * 1e-3), "kernels": on_launch[0],
                                    "what": f"the masked products of {M} rows with no correction work, timed alone"},
                    "correction_ms_per_prefill": ms - ms_online},
        "roofline": roofline,
        "gpu_launches": gpu_launches,
        "clocks": clocks.summary(),
    }
    if e2e is not None:
        result["e2e"] = e2e
    if decode is not None:
        result["decode"] = decode
    result["offloaded_six"] = offloaded
    result["down"] = down
    result["bound_check"] = bound
    if layer0.calibration:
        result["path_choice"] = {g: {"path": c["path"], **{f"{p}_max_err_over_hard": c[p]["max_err_over_hard"]
                                                          for p in ("fp32", "tf32x3", "fp16x3")}}
                                 for g, c in layer0.calibration.items()}
    if cpu is not None:
        result["cpu_baseline"] = cpu
        result["oracle_match"] = match
    if rank == 0:
        print(json.dumps(result))
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
