#!/usr/bin/env python
"""Benchmark of the masked-linear hot path on one GB300.

Workload (one step): one Llama-3.2-3B-shaped decoder layer's outsourced
linears (Q, K, V, O, Gate, Up, Down) at 128 prompt tokens, fp32, Gaussian
noise at eps = 1.  A step regenerates and adds the mask of each input group,
then runs the masked product with the unmask fused into its epilogue
(Y = X~ W^T - C).  Every 8 steps the correction bank is refilled: 8 masks
per group are drawn and their corrections C = eta W^T computed as one
product of 8 x 128 rows ("precomputed in a batch"), so each step carries an
eighth of that work.  The weights (0.4 GB per layer in fp32, plus the TF32
and fp16 splits) are larger than L2, so no step reuses L2-resident weights.
The arithmetic path of each input group is chosen by the bound check on a
masked sample (spl_choose_path) unless --path fixes it.

Prints one JSON line.  ``--impl reference`` times the fp64 CPU oracle on a
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
sys.path.insert(0, ROOT)

METRIC = "masked-linear TFLOP/s & ms/prefill (Llama-3B shapes), % of roofline, oracle match"
UNIT = "TFLOP/s"
TF32_OVER_BF16 = 1.1 / 2.25  # nominal dense TF32 : BF16 tensor rate on GB300
WORKLOAD = ("llama-3.2-3b-shaped layer (Q,K,V,O,gate,up,down), 128 tokens, fp32, gaussian eps=1, "
            "corrections precomputed in banks of 8 draws")
DRAWS = 8


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=32)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--eps", type=float, default=1.0)
    ap.add_argument("--path", default="auto")
    ap.add_argument("--tokens", type=int, default=128)
    ap.add_argument("--cpu-sample-rows", type=int, default=4)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-overlap", action="store_true",
                    help="compute each bank cycle's corrections before its steps instead of during the previous cycle")
    ap.add_argument("--stored-noise", action="store_true",
                    help="keep the bank's fp32 noise and mask each step with it instead of drawing it again")
    ap.add_argument("--workload", default="llama_layer",
                    choices=["llama_layer", "llama_stack", "qwen_stack", "qwen_sweep", "down_fp64", "slalom",
                             "lm_head"],
                    help="llama_layer (default): the headline line; the others measure the stack and sweep "
                         "workloads and print their own line")
    return ap.parse_args(argv)


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


def profiled_traffic():
    """DRAM bytes per step of the online product launches from the committed ncu summary, if it
    was taken on the current tensor-core kernel source (else None)."""
    import hashlib
    prof = os.path.join(ROOT, "profiles", "tc_gemm_fp16x3_llama_online_and_bank.md")
    src = os.path.join(ROOT, "paper_2609_15039_gb300", "csrc", "gemm_tc.cu")
    try:
        fields = dict(line.split(":", 1) for line in open(prof).read().splitlines()
                      if line.startswith(("traffic_bytes_per_step:", "kernel_source_sha256_prefix:")))
        digest = hashlib.sha256(open(src, "rb").read()).hexdigest()
    except (OSError, ValueError):
        return None, "no profile"
    if not digest.startswith(fields.get("kernel_source_sha256_prefix", "-").strip()):
        return None, "kernel changed since the ncu capture"
    return float(fields["traffic_bytes_per_step"]), "ncu capture of the same kernel source (profiles/)"


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
def oracle_sample(model, M, rows, eps, mech, seed, deltas, weights_cpu, inputs_cpu):
    """The oracle on the first ``rows`` tokens of every group: noise, mask, products, unmask."""
    from oracle import linear, philox
    out = {}
    flops = 0
    for gi, (g, K, names) in enumerate(model.input_groups()):
        X = inputs_cpu[g][:rows]
        eta = philox.noise((M, K), deltas[g], eps, mech, seed, stream_id=gi)[:rows]
        Xt = linear.mask(X, eta)
        for name in names:
            W = weights_cpu[name]
            r = linear.masked_linear(Xt, W)
            C = linear.precompute_noise_product(eta, W)
            out[name] = linear.unmask(r.astype("float32"), C.astype("float32"))
            flops += 2 * 2 * rows * K * W.shape[0]
    return out, flops


def cpu_setup(model, M):
    import numpy as np
    from oracle import sensitivity as osens
    from paper_2609_15039_gb300 import workloads as wl
    weights = {name: wl.weight(N, K, seed=200 + pi).numpy() for pi, (name, K, N, g) in enumerate(model.projections())}
    inputs = {g: wl.activations(M, K, seed=100 + gi).numpy() for gi, (g, K, _n) in enumerate(model.input_groups())}
    ones = np.ones(model.d_model)
    norms = {n: osens.spectral_norm(weights[n], iters=30) for n in ("v", "up", "gate")}
    deltas = {"qkv": osens.delta_layernorm(ones), "gateup": osens.delta_layernorm(ones),
              "o": osens.delta_attention(ones, norms["v"]),
              "down": osens.delta_activation(ones, None, model.d_ff, norms["up"], norms["gate"])}
    return weights, inputs, deltas


def run_reference(args):
    world, rank, _ = dist_env()
    if rank != 0:
        return
    from paper_2609_15039_gb300 import workloads as wl
    model, M = wl.LLAMA_3_2_3B, args.tokens
    weights, inputs, deltas = cpu_setup(model, M)
    rows = args.cpu_sample_rows
    for w in range(args.warmup):
        oracle_sample(model, M, rows, args.eps, "gaussian", 1000 + w, deltas, weights, inputs)
    t0 = time.perf_counter()
    flops = 0
    for s in range(args.steps):
        _, f = oracle_sample(model, M, rows, args.eps, "gaussian", 2000 + s, deltas, weights, inputs)
        flops += f
    dt = time.perf_counter() - t0
    value = flops / dt / 1e12
    sample = f"first {rows} of {M} tokens of every input group, all 7 projections, per step"
    print(json.dumps({
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * dt / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": WORKLOAD, "tokens": M, "eps": args.eps},
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
        res = measure.WORKLOADS[args.workload]()
    if args.workload == "llama_stack":
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
    args = parse()
    if args.impl == "reference":
        return run_reference(args)
    if args.workload != "llama_layer":
        return run_workload(args)
    import numpy as np
    import torch
    import torch.distributed as dist
    from paper_2609_15039_gb300 import spl, workloads as wl
    from paper_2609_15039_gb300.layer import MaskedLayer

    world, rank, local = dist_env()
    if world > 1:
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    model, M, mech, seed = wl.LLAMA_3_2_3B, args.tokens, "gaussian", 4242

    weights = {name: wl.weight(N, K, seed=200 + pi, device=dev) for pi, (name, K, N, g) in
               enumerate(model.projections())}
    layer = MaskedLayer.from_weights(model, weights, split=True, device=dev)
    layer.sensitivities()
    layer.allocate(M, DRAWS, args.path, stored_noise=args.stored_noise)
    inputs = {g: wl.activations(M, K, seed=100 + gi, device=dev) for gi, (g, K, _n) in
              enumerate(model.input_groups())}
    if args.path == "auto":
        layer.calibrate(inputs, args.eps, mech, seed)  # a8: bound-based path choice per group
    stream = torch.cuda.current_stream(dev)

    def step(s, x=inputs):
        """One eager step through the library calls (host-side Philox offsets)."""
        cycle, d = divmod(s, DRAWS)
        if d == 0:
            layer.refill(args.eps, mech, seed, cycle, path=args.path)
        return layer.online(x, args.eps, mech, seed, cycle, d, path=args.path)

    # One eager step sets up every library call (tensor maps, shared-memory attributes, occupancy
    # queries); then the steps of one bank cycle are captured as CUDA graphs, with CUDA events
    # around every product call (external event nodes, timestamped at each replay).
    step(0)
    torch.cuda.synchronize()
    gevents = {}  # (draw, kind, group) -> [begin, end] of the latest replay
    cur = {"d": 0}

    def gtimer(phase, kind, group):
        e = torch.cuda.Event(enable_timing=True, external=True)
        e.record()
        if phase == "begin":
            gevents[(cur["d"], kind, group)] = [e, None]
        else:
            gevents[(cur["d"], kind, group)][1] = e

    # the timed region replays graphs without event nodes (an event node between two kernels keeps
    # the second from launching early); a second pass over the same steps replays graphs with an
    # event pair around every product call, for the per-kernel times of the roofline
    graphs, graph_launches = layer.capture(inputs, args.eps, mech, seed, path=args.path)
    ev_graphs, _ = layer.capture(inputs, args.eps, mech, seed, path=args.path, timer=gtimer,
                                 before=lambda d: cur.update(d=d))
    # end to end: the same steps with every step's inputs copied in from pinned host memory and its
    # outputs copied back inside each graph, on a second stream.  Inputs are double-buffered: step s
    # computes on buffer s % 2 while its graph copies the next step's inputs into the other one; each
    # group's result starts back as soon as its product is done, while the next group computes, and
    # the last group's at the top of the next step.  The timed region holds one input copy and one
    # full result copy per step (the last step's last result is copied before the clock stops).
    host_in = {g: x.cpu().pin_memory() for g, x in inputs.items()}
    dev_in = [{g: torch.empty_like(x) for g, x in inputs.items()} for _ in range(2)]
    host_out = {g.name: torch.empty((M, g.N)).pin_memory() for g in layer.groups}
    h2d = sum(x.numel() * 4 for x in host_in.values())
    d2h = sum(o.numel() * 4 for o in host_out.values())
    copy_stream = torch.cuda.Stream()
    last = layer.groups[-1].name  # its result goes back at the top of the next step, which overwrites
                                  # it only at its own end

    last_back = {}

    def copy_in(d):
        copy_stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(copy_stream):
            host_out[last].copy_(layer.bank[last]["Y"], non_blocking=True)  # the previous step's
            last_back["ev"] = torch.cuda.Event()
            last_back["ev"].record(copy_stream)
            for g, x in dev_in[(d + 1) % 2].items():
                x.copy_(host_in[g], non_blocking=True)

    def group_in(gi, g):
        if g == last:  # its previous result has gone back
            torch.cuda.current_stream().wait_event(last_back["ev"])

    def group_out(gi, g):
        if g == last:
            return
        copy_stream.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(copy_stream):
            host_out[g].copy_(layer.bank[g]["Y"], non_blocking=True)

    def copy_out(d):
        torch.cuda.current_stream().wait_stream(copy_stream)

    e2e_graphs = None
    if not args.no_e2e:
        for buf in dev_in:  # the first replayed step finds its inputs in place
            for g, x in buf.items():
                x.copy_(host_in[g])
        e2e_graphs, _ = layer.capture(dev_in, args.eps, mech, seed, path=args.path, before=copy_in, after=copy_out,
                                      group_hooks=(group_in, group_out))

    # The corrections of the next bank cycle need nothing from this one: whole-cycle graphs compute
    # them during this cycle's steps, on streams of lower priority (MaskedLayer.capture_overlapped).
    # Used when every group takes the fused fp16 split and the step count is whole cycles.
    use_ov = (not args.no_overlap and args.steps % DRAWS == 0 and
              all(layer._fused_split(g, args.path, M) for g in layer.groups))
    if use_ov:
        ov_graphs, ov_launches = layer.capture_overlapped(inputs, args.eps, mech, seed, path=args.path)
        e2e_ov = None
        if e2e_graphs is not None:
            e2e_ov, _ = layer.capture_overlapped(dev_in, args.eps, mech, seed, path=args.path, before=copy_in,
                                                 after=copy_out, group_hooks=(group_in, group_out))

    def start_overlapped(cycle):
        """Bank buffer cycle % 2 holds the corrections of ``cycle``; the bases are at ``cycle``."""
        layer.set_cycle(cycle)
        layer.refill(args.eps, mech, seed, 0, path=args.path, device_base=True, parallel=True, parity=cycle % 2)

    s = DRAWS  # the graphs start at a bank cycle
    if use_ov:
        start_overlapped(s // DRAWS)
        for _ in range(-(-args.warmup // DRAWS)):  # warm-up: whole cycles, at least the W steps
            ov_graphs[(s // DRAWS) % 2].replay()
            s += DRAWS
    else:
        layer.set_cycle(s // DRAWS)
        for _ in range(args.warmup):
            graphs[s % DRAWS].replay()
            s += 1
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    s_timed = s
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    with ClockSampler(local) as clocks:
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_push("timed")
        t_start.record(stream)
        if use_ov:
            for _ in range(args.steps // DRAWS):
                ov_graphs[(s // DRAWS) % 2].replay()
                s += DRAWS
        else:
            for _ in range(args.steps):
                graphs[s % DRAWS].replay()
                s += 1
        t_end.record(stream)
        torch.cuda.synchronize()
        torch.cuda.nvtx.range_pop()
    if world > 1:
        dist.barrier()
    if use_ov:
        gpu_launches = sum(ov_launches[(s_timed // DRAWS + i) % 2] for i in range(args.steps // DRAWS))
    else:
        gpu_launches = sum(graph_launches[(s_timed + i) % DRAWS] for i in range(args.steps))
    ms = t_start.elapsed_time(t_end) / args.steps
    layer.set_cycle(s // DRAWS)  # the per-step graphs below start at a bank cycle
    # second pass: per-call events (the last replay of each draw's graph holds its times)
    p_start = torch.cuda.Event(enable_timing=True)
    p_end = torch.cuda.Event(enable_timing=True)
    p_start.record(stream)
    for _ in range(args.steps):
        ev_graphs[s % DRAWS].replay()
        s += 1
    p_end.record(stream)
    torch.cuda.synchronize()
    ms_with_events = p_start.elapsed_time(p_end) / args.steps
    ms = max_over_ranks(ms, dev)
    st = spl.spl_get_device_status()
    if st != spl.SPL_OK:
        raise RuntimeError("device status " + spl.status_string(st))

    flops_step = layer.flops_per_step()
    value = job_rate(world, flops_step, ms) / 1e12
    group_paths = {g.name: spl.PATH_NAMES[spl.spl_resolve_path(M, g.K, g.N, layer.path_of(g, args.path, M))]
                   for g in layer.groups}
    path_name = "+".join(sorted(set(group_paths.values())))

    # roofline of the dominant kernel: the product calls (tcgen05 GEMM + its row exponents / reductions)
    pk = peaks()
    # per product call: the latest replay of each graph (the last bank cycle of the timed region)
    by_kind, by_group = {}, {}
    for (d, kind, group), (b, e) in gevents.items():
        by_kind.setdefault(kind, []).append(b.elapsed_time(e))
        by_group.setdefault((kind, group), []).append(b.elapsed_time(e))
    path_peak = {  # algorithmic flops (one product per term) per second at each path's instruction peak
        "fp16x3": pk["bf16_tflops_sustained"] / 3.0,
        "tf32x3": pk["bf16_tflops_sustained"] * TF32_OVER_BF16 / 3.0,
        "fp32": 152 * 128 * 2 * 2.07e9 / 1e12,
    }
    per_kind = {}
    for kind, v in by_kind.items():
        rows = DRAWS * M if kind == "precompute" else M
        f = sum(2 * rows * g.K * g.N for g in layer.groups) * len(v) / len(layer.groups)
        per_kind[kind] = {"calls": len(v), "avg_ms": sum(v) / len(v), "tflops": f / (sum(v) * 1e-3) / 1e12,
                          "rows": rows}
        for g in layer.groups:
            t = by_group[(kind, g.name)]
            avg = sum(t) / len(t)
            per_kind[kind][g.name] = {"avg_us": 1e3 * avg, "tflops": 2 * rows * g.K * g.N / (avg * 1e-3) / 1e12,
                                      "path": group_paths[g.name]}
    # The dominant kernel: the online masked products (a5 + a6), four calls per step.  At 128 rows
    # they do 64 algorithmic flops per byte, below the FP16X3 ridge (~84), so HBM bounds them:
    # achieved = algorithmic bytes per step (weight split 4 B per weight or the path's format,
    # X~ in, C in, Y out) / their measured time per step.
    online_ms = sum(by_kind["masked_linear_unmask"]) / DRAWS
    wbytes = {"fp16x3": 4, "tf32x3": 8, "fp32": 4}
    online_bytes = sum(wbytes[group_paths[g.name]] * g.K * g.N + 4 * M * g.K + 8 * M * g.N for g in layer.groups)
    achieved = online_bytes / (online_ms * 1e-3) / 1e9
    bank_ms = sum(by_kind["precompute"])
    bank_flops = sum(2 * DRAWS * M * g.K * g.N for g in layer.groups)
    bank_peak = bank_flops / sum(2 * DRAWS * M * g.K * g.N / path_peak[group_paths[g.name]] for g in layer.groups)
    traffic, traffic_note = profiled_traffic()
    roofline = {"bound": "hbm", "achieved": achieved, "peak": pk["hbm_gbs"], "unit": "GB/s",
                "frac": achieved / pk["hbm_gbs"], "traffic": traffic,
                "kernel": "tc_gemm_kernel online masked products with fused unmask (4 calls per step, 128 rows)",
                "algorithmic_bytes_per_step": online_bytes, "ms_per_step": online_ms,
                "traffic_note": traffic_note, "group_paths": group_paths,
                "share_of_step": (online_ms + bank_ms / DRAWS) / ms_with_events,
                "bank": {"bound": "tensor", "kernel": "tc_gemm_kernel bank refill, 1024 rows, segmented K",
                         "achieved": bank_flops / (bank_ms * 1e-3) / 1e12, "peak": bank_peak, "unit": "TFLOP/s",
                         "frac": bank_flops / (bank_ms * 1e-3) / 1e12 / bank_peak, "ms_per_refill": bank_ms},
                "per_call": per_kind,
                "timing": "per-call CUDA events (external event nodes) in a second pass over the same steps; "
                          f"that pass ran at {ms_with_events:.4f} ms/step",
                "peak_source": pk["source"],
                "peak_note": "hbm: measured copy bandwidth; bank: per group fp16x3 = measured sustained bf16 "
                             "(fp16 runs at the bf16 rate) / 3 products per term, tf32x3 = that x nominal "
                             "tf32/bf16 (1.1/2.25), fp32 FMA = 152 SMs x 128 lanes x 2 flop x 2.07 GHz (derived)"}

    e2e = None
    if e2e_graphs is not None:
        if use_ov:
            s = -(-s // DRAWS) * DRAWS
            start_overlapped(s // DRAWS)
            e2e_ov[(s // DRAWS) % 2].replay()  # warm-up cycle
            s += DRAWS
        else:
            for _ in range(2):
                e2e_graphs[s % DRAWS].replay()
                s += 1
        torch.cuda.synchronize()
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        if use_ov:
            for _ in range(args.steps // DRAWS):
                e2e_ov[(s // DRAWS) % 2].replay()
                s += DRAWS
        else:
            for _ in range(args.steps):
                e2e_graphs[s % DRAWS].replay()
                s += 1
        host_out[last].copy_(layer.bank[last]["Y"], non_blocking=True)  # the last step's, in the region
        e1.record(stream)
        torch.cuda.synchronize()
        e2e_ms = e0.elapsed_time(e1) / args.steps
        e2e_ms = max_over_ranks(e2e_ms, dev)
        e2e = {"value": job_rate(world, flops_step, e2e_ms) / 1e12, "unit": UNIT, "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms,
               "copies": "pinned host memory, on a second stream inside each step's graph: the next "
                         "step's inputs copied in (double-buffered) while this one computes, each result "
                         "copied out after its product (the last group's at the top of the next step)"}

    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "path": path_name, "data": "synthetic",
        "config": {"workload": WORKLOAD, "tokens": M, "eps": args.eps, "mech": mech, "layers_per_step": 1,
                   "bank_draws": DRAWS, "flops_per_step": flops_step,
                   "bank_schedule": ("each cycle's corrections computed during the previous cycle's steps, on "
                                     "lower-priority streams (whole-cycle graphs)") if use_ov else
                                    "each cycle's corrections computed before its first step",
                   "online_noise": ("kept from the bank refill, read by each step's mask" if args.stored_noise
                                    else "drawn again in each step's mask"),
                   "l2": "weights 1.2 GB per step > 129 MB L2 (no flush needed)",
                   "parallelism": "replicas" if world > 1 else "single"},
        "ms_per_prefill_28_layers": 28 * ms,
        "roofline": roofline,
        "gpu_launches": gpu_launches,
        "clocks": clocks.summary(),
    }
    if e2e is not None:
        result["e2e"] = e2e
    if layer.calibration:
        result["path_choice"] = {g: {"path": c["path"],
                                     **{f"{p}_max_err_over_hard": c[p]["max_err_over_hard"]
                                        for p in ("fp32", "tf32x3", "fp16x3")},
                                     **{f"{p}_mean_err": c[p]["mean_err"] for p in ("fp32", "tf32x3", "fp16x3")}}
                                 for g, c in layer.calibration.items()}
    # the paper's bound over every output of one more online step, evaluated on the GPU in fp64
    cycle, d = divmod(s, DRAWS)
    outs = step(s)
    s += 1
    bc = layer.bound_check(inputs, outs, args.eps, mech, seed, cycle, d)
    result["bound_check"] = {g: {"max_err_over_hard": v["max_err_over_hard"], "log_violation_pct": v["violation_pct"],
                                 "mean_err": v["mean_err"], "mean_log_bound": v["mean_log_bound"],
                                 "max_rel_err": v["max_err"] / v["max_abs_ref"] if v["max_abs_ref"] else 0.0}
                             for g, v in bc.items()}

    # cpu baseline + oracle match on the first rows (rank 0, N = 1 only)
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from oracle import bounds, linear, philox
        rows = args.cpu_sample_rows
        cycle, d = divmod(s, DRAWS)
        outs = step(s)
        torch.cuda.synchronize()
        gpu_rows = {g: outs[g][:rows].double().cpu().numpy() for g in outs}
        w_cpu = {g.name: g.W.cpu().numpy() for g in layer.groups}
        x_cpu = {g: x.cpu().numpy() for g, x in inputs.items()}
        t0, flops, reps = time.perf_counter(), 0, 0
        worst = 0.0
        while True:
            for gi, g in enumerate(layer.groups):
                X = x_cpu[g.name][:rows]
                eta = philox.noise((M, g.K), layer.deltas[g.name], args.eps, mech, seed, stream_id=gi,
                                   offset=layer.block_offset(g, cycle, d))[:rows]
                Xt = linear.mask(X, eta)
                r = linear.masked_linear(Xt, w_cpu[g.name])
                C = linear.precompute_noise_product(eta, w_cpu[g.name])
                Y = linear.unmask(r.astype(np.float32), C.astype(np.float32))
                flops += 2 * 2 * rows * g.K * g.N
                if reps == 0:
                    S = linear.abs_products(X, Xt, eta, w_cpu[g.name])
                    err = np.abs(gpu_rows[g.name] - linear.reference_output(X, w_cpu[g.name]))
                    worst = max(worst, float(np.max(err / bounds.hard_bound(*S, g.K))))
                    del Y
            reps += 1
            if time.perf_counter() - t0 > 10.0 or reps >= 50:
                break
        dt = time.perf_counter() - t0
        result["cpu_baseline"] = {"value": flops / dt / 1e12, "unit": UNIT, "cores": os.cpu_count(),
                                  "kind": "oracle", "seconds": dt,
                                  "sample": f"first {rows} of {M} tokens of every input group, {reps} repetitions"}
        result["oracle_match"] = {"rows_checked": rows, "max_err_over_hard_bound": worst, "pass": worst <= 1.0}

    if rank == 0:
        print(json.dumps(result))
    if world > 1:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
