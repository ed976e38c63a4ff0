"""Measurements of the stack and sweep workloads (bench.py --workload ...).

Each function runs one workload on the current CUDA device through the library (MaskedStack /
MaskedLayer sequencing ABI calls, replayed as CUDA graphs) and returns a dict that bench.py
prints as its JSON line.  Times are CUDA events on the launching stream around graph replays;
inputs are resident in HBM.  The workloads:

* llama_stack -- 28 Llama-3.2-3B-shaped layers: prefill of 512 tokens (banks of 8 draws), then
  decode at one token per step for 256 steps (its own banks of 8 one-row draws); Laplace, eps = 1.
* qwen_stack  -- 36 Qwen3-4B-shaped layers, prefill of 2048 tokens at eps in {0.1, 1, 10} with
  the cancellation error of every output of the first and last layer checked against the bound.
* qwen_sweep  -- one Qwen3-4B-shaped layer at M in {1, 4, 16, 64, 256, 1024} tokens, and the
  noise + mask kernel alone on 10^9 elements.
* lm_head     -- the Llama LM head (3072 -> 128256) at 512 and 1 tokens with its bank.
"""

import torch

from . import spl, workloads as wl
from .layer import MaskedStack


def _peaks():
    import json
    import os
    p = {"hbm_gbs": 6800.0, "bf16_tflops_sustained": 1700.0, "source": "fallback"}
    path = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            m = json.load(f)
        p.update({k: float(m[k]) for k in ("hbm_gbs", "bf16_tflops_sustained") if k in m})
        p["source"] = "measured"
    except (OSError, ValueError, KeyError):
        pass
    return p


def _path_peak(path, pk):
    """Algorithmic TFLOP/s at each path's instruction peak (see bench.py)."""
    return {"fp16x3": pk["bf16_tflops_sustained"] / 3.0,
            "tf32x3": pk["bf16_tflops_sustained"] * (1.1 / 2.25) / 3.0,
            "fp32": 152 * 128 * 2 * 2.07e9 / 1e12}[path]


def _group_paths(stack_or_layer, M):
    layers = getattr(stack_or_layer, "layers", [stack_or_layer])
    out = {}
    for g in layers[0].groups:
        out[g.name] = spl.PATH_NAMES[spl.spl_resolve_path(M, g.K, g.N, layers[0].path_of(g, "auto", M))]
    return out


def _weight_bytes(layer, M, paths):
    """HBM bytes of one online step of a layer: the weight in the format its path reads, x~ in,
    C in, Y out (fp32)."""
    per_w = {"fp32": 4, "tf32x3": 8, "fp16x3": 4}
    total = 0
    for g in layer.groups:
        total += per_w[paths[g.name]] * g.K * g.N + 4 * M * g.K + 8 * M * g.N
    return total


def _time_replays(graphs, start, n, stream):
    """Replays graphs[(start + i) % D] for i < n; returns per-replay ms (events around each)."""
    D = len(graphs)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(n + 1)]
    ev[0].record(stream)
    for i in range(n):
        graphs[(start + i) % D].replay()
        ev[i + 1].record(stream)
    torch.cuda.synchronize()
    return [ev[i].elapsed_time(ev[i + 1]) for i in range(n)]


def _calibrate(stack, inputs, eps, mech):
    for layer, x, seed in zip(stack.layers, inputs, stack.seeds):
        layer.calibrate(x, eps, mech, seed)


def _bound(stack, inputs, eps, mech, s, layers):
    """The bound over every output of layers ``layers`` for eager step s (its bank cycle is
    refilled first, whatever the bank held before)."""
    cycle, d = divmod(s, stack.draws)
    res = {}
    for li in layers:
        layer, x, seed = stack.layers[li], inputs[li], stack.seeds[li]
        layer.refill(eps, mech, seed, cycle)
        outs = layer.online(x, eps, mech, seed, cycle, d)
        bc = layer.bound_check(x, outs, eps, mech, seed, cycle, d)
        res[f"layer{li}"] = {g: {"max_err_over_hard": v["max_err_over_hard"], "log_violation_pct": v["violation_pct"],
                                 "mean_err": v["mean_err"], "mean_log_bound": v["mean_log_bound"],
                                 "max_rel_err": v["max_err"] / v["max_abs_ref"] if v["max_abs_ref"] else 0.0}
                             for g, v in bc.items()}
    return res


def _prefill(stack, inputs, eps, mech, cycles=2, product_times=False):
    """Graph-replayed prefill: online-only steps (draws 1..D-1) and the draw-0 step that also
    refills every bank; returns ms per online pass and per refill.  product_times: also the ms per
    online pass spent in the masked products alone, from a second pass over the same steps whose
    graphs hold a CUDA event pair around every product call (an event node keeps the next kernel
    from starting early, so this slightly over-counts)."""
    stream = torch.cuda.current_stream()
    D = stack.draws
    stack.step(inputs, eps, mech, 0)  # sets up every library call before capture
    torch.cuda.synchronize()
    graphs, launches = stack.capture(inputs, eps, mech)
    stack.set_cycle(1)
    _time_replays(graphs, 0, D, stream)  # warm-up cycle
    times = _time_replays(graphs, 0, cycles * D, stream)
    online = [t for i, t in enumerate(times) if i % D != 0]
    with_refill = [t for i, t in enumerate(times) if i % D == 0]
    on = sum(online) / len(online) if online else float("nan")
    rf = sum(with_refill) / len(with_refill) - (on if online else 0.0)
    del graphs
    torch.cuda.synchronize()
    if not product_times:
        return on, rf, launches
    ev = {}

    def timer(d, li, phase, kind, group):
        if kind != "masked_linear_unmask":
            return
        e = torch.cuda.Event(enable_timing=True, external=True)
        e.record()
        ev.setdefault((d, li, group), [None, None])[0 if phase == "begin" else 1] = e

    ev_graphs, _ = stack.capture(inputs, eps, mech, timer=timer)
    stack.set_cycle(1)
    _time_replays(ev_graphs, 0, D, stream)  # one cycle: each graph's events hold its last replay
    prod = sum(b.elapsed_time(e) for (d, li, g), (b, e) in ev.items() if d != 0) / max(1, D - 1)
    del ev_graphs
    torch.cuda.synchronize()
    return on, rf, launches, prod


def llama_stack(layers=28, tokens=512, decode_steps=256, eps=1.0, mech="laplace", draws=8):
    model = wl.LLAMA_3_2_3B
    pk = _peaks()
    stack = MaskedStack.build(model, layers, tokens, draws, base_seed=7)
    inputs = stack.inputs(11)
    _calibrate(stack, inputs, eps, mech)
    paths = _group_paths(stack, tokens)
    on_ms, refill_ms, launches, prod_ms = _prefill(stack, inputs, eps, mech, product_times=True)
    flops = 2 * tokens * model.weights_per_layer() * layers
    peak = flops / sum(2 * tokens * g.K * g.N * layers / _path_peak(paths[g.name], pk) for g in stack.layers[0].groups)
    prefill = {"ms_per_prefill": on_ms, "tflops": flops / (on_ms * 1e-3) / 1e12, "tokens_per_s": tokens / (on_ms * 1e-3),
               "roofline_peak_tflops": peak, "frac": flops / (on_ms * 1e-3) / 1e12 / peak,
               "gemm": {"ms": prod_ms, "tflops": flops / (prod_ms * 1e-3) / 1e12,
                        "frac": flops / (prod_ms * 1e-3) / 1e12 / peak,
                        "timing": "the masked products alone (tensor-core kernels with fused unmask), CUDA event "
                                  "pairs around each product call in a second pass over the same graph-replayed "
                                  "steps; the mask + split kernels between them are the rest of ms_per_prefill"},
               "bank_refill_ms": refill_ms, "bank_refill_ms_per_draw": refill_ms / draws,
               "bank_refill_tflops": draws * flops / (refill_ms * 1e-3) / 1e12, "paths": paths,
               "kernels_per_online_step": launches[1] if len(launches) > 1 else launches[0]}
    bound = _bound(stack, inputs, eps, mech, 3 * draws + 1, [0, layers - 1])
    # decode: the same layers re-allocated for one token per step, banks of `draws` one-row draws
    ws = spl.workspace(max(l.workspace_bytes(1, draws) for l in stack.layers))
    for layer in stack.layers:
        layer.allocate(1, draws, workspace=ws)
    inputs1 = stack.inputs(13)
    stream = torch.cuda.current_stream()
    stack.step(inputs1, eps, mech, 0)
    torch.cuda.synchronize()
    # serial schedule: one graph per step, the draw-0 step refilling every bank first
    graphs, dl = stack.capture(inputs1, eps, mech)
    stack.set_cycle(1)
    _time_replays(graphs, 0, draws, stream)
    times = _time_replays(graphs, 0, decode_steps, stream)
    serial_ms = sum(times) / len(times)
    del graphs
    # overlapped schedule: whole-cycle graphs computing the next cycle's corrections on a stream of
    # lower priority while this cycle's steps run (MaskedStack.capture_overlapped)
    bank_ws = spl.workspace(max(l.workspace_bytes(1, draws) for l in stack.layers))
    ov_graphs, ol = stack.capture_overlapped(inputs1, eps, mech, bank_ws)
    cycles = -(-decode_steps // draws)
    stack.start_overlapped(1, eps, mech)
    _time_replays([ov_graphs[1], ov_graphs[0]], 0, 2, stream)  # warm-up: cycles 1 and 2
    times = _time_replays([ov_graphs[1], ov_graphs[0]], 0, cycles, stream)  # cycles 3, 4, ...
    step_ms = sum(times) / (cycles * draws)
    del ov_graphs
    dpaths = _group_paths(stack, 1)
    step_bytes = sum(_weight_bytes(l, 1, dpaths) for l in stack.layers) * (1 + 1.0 / draws)  # + the bank's share
    decode = {"steps": cycles * draws, "ms_per_token": step_ms, "tokens_per_s": 1e3 / step_ms,
              "gbs": step_bytes / (step_ms * 1e-3) / 1e9, "hbm_peak_gbs": pk["hbm_gbs"],
              "frac": step_bytes / (step_ms * 1e-3) / 1e9 / pk["hbm_gbs"], "bytes_per_step": step_bytes,
              "paths": dpaths, "kernels_per_step": sum(ol) / len(ol) / draws,
              "schedule": "each cycle's corrections computed during the previous cycle's steps, on a stream of "
                          "lower priority (whole-cycle graphs)",
              "serial": {"ms_per_token": serial_ms, "tokens_per_s": 1e3 / serial_ms,
                         "frac": step_bytes / (serial_ms * 1e-3) / 1e9 / pk["hbm_gbs"],
                         "kernels_per_step": sum(dl) / len(dl),
                         "schedule": "one graph per step, the first step of a cycle refilling every bank"}}
    return {"workload": f"llama-3.2-3b-shaped stack, {layers} layers, prefill {tokens} tokens + decode "
                        f"{decode_steps} steps at 1 token, {mech} eps={eps}, banks of {draws} draws",
            "prefill": prefill, "decode": decode, "bound_check": bound, "peak_source": pk["source"]}


def qwen_stack(layers=36, tokens=2048, eps_list=(0.1, 1.0, 10.0), mech="gaussian", draws=2):
    model = wl.QWEN3_4B
    pk = _peaks()
    stack = MaskedStack.build(model, layers, tokens, draws, base_seed=11)
    inputs = stack.inputs(17)
    res = {}
    flops = 2 * tokens * model.weights_per_layer() * layers
    for eps in eps_list:
        _calibrate(stack, inputs, eps, mech)
        paths = _group_paths(stack, tokens)
        on_ms, refill_ms, _, prod_ms = _prefill(stack, inputs, eps, mech, cycles=2, product_times=True)
        peak = flops / sum(2 * tokens * g.K * g.N * layers / _path_peak(paths[g.name], pk)
                           for g in stack.layers[0].groups)
        res[f"eps={eps}"] = {
            "ms_per_prefill": on_ms, "tflops": flops / (on_ms * 1e-3) / 1e12, "tokens_per_s": tokens / (on_ms * 1e-3),
            "roofline_peak_tflops": peak, "frac": flops / (on_ms * 1e-3) / 1e12 / peak,
            "gemm": {"ms": prod_ms, "tflops": flops / (prod_ms * 1e-3) / 1e12,
                     "frac": flops / (prod_ms * 1e-3) / 1e12 / peak},
            "bank_refill_ms_per_draw": refill_ms / draws, "paths": paths,
            "bound_check": _bound(stack, inputs, eps, mech, 5 * draws + 1, [0, layers - 1])}
    return {"workload": f"qwen3-4b-shaped stack, {layers} layers, prefill {tokens} tokens, {mech}, "
                        f"banks of {draws} draws", "prefill": res, "peak_source": pk["source"]}


def qwen_sweep(Ms=(1, 4, 16, 64, 256, 1024), eps=1.0, mech="gaussian", draws=8, mask_elements=10 ** 9):
    model = wl.QWEN3_4B
    pk = _peaks()
    stack = MaskedStack.build(model, 1, Ms[0], draws, base_seed=13)
    layer = stack.layers[0]
    out = {}
    for M in Ms:
        ws = spl.workspace(layer.workspace_bytes(M, draws))
        layer.allocate(M, draws, workspace=ws)
        inputs = stack.inputs(19)
        _calibrate(stack, inputs, eps, mech)
        paths = _group_paths(stack, M)
        on_ms, refill_ms, _ = _prefill(stack, inputs, eps, mech, cycles=4)
        flops = 2 * M * model.weights_per_layer()
        nbytes = _weight_bytes(layer, M, paths)
        peak_t = flops / sum(2 * M * g.K * g.N / _path_peak(paths[g.name], pk) for g in layer.groups)
        t_hbm = nbytes / (pk["hbm_gbs"] * 1e9)
        t_tc = flops / (peak_t * 1e12)
        out[f"M={M}"] = {"online_ms": on_ms, "tflops": flops / (on_ms * 1e-3) / 1e12,
                         "gbs": nbytes / (on_ms * 1e-3) / 1e9, "bound": "hbm" if t_hbm >= t_tc else "tensor",
                         "roofline_ms": max(t_hbm, t_tc) * 1e3, "frac": max(t_hbm, t_tc) * 1e3 / on_ms,
                         "bank_refill_ms_per_draw": refill_ms / draws, "paths": paths}
        del ws
    # the noise + mask kernel alone (eta regenerated, not stored): 8 bytes per element
    n = mask_elements
    X = torch.empty(n, device="cuda")
    X.normal_(generator=torch.Generator(device="cuda").manual_seed(3))
    Xt = torch.empty_like(X)
    stream = torch.cuda.current_stream()
    mask = {}
    for m in ("laplace", "gaussian"):
        for _ in range(2):
            spl.spl_noise_mask(Xt, None, X, 719.8, 1.0, m, 5)
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        reps = 10
        e0.record(stream)
        for r in range(reps):
            spl.spl_noise_mask(Xt, None, X, 719.8, 1.0, m, 5, offset=r * (n // 4))
        e1.record(stream)
        torch.cuda.synchronize()
        ms = e0.elapsed_time(e1) / reps
        mask[m] = {"ms": ms, "gbs": 8 * n / (ms * 1e-3) / 1e9, "frac": 8 * n / (ms * 1e-3) / 1e9 / pk["hbm_gbs"]}
    return {"workload": f"qwen3-4b-shaped layer, M sweep {list(Ms)}, {mech} eps={eps}, banks of {draws} draws; "
                        f"noise + mask alone on {n} elements", "sweep": out, "mask": mask,
            "hbm_peak_gbs": pk["hbm_gbs"], "peak_source": pk["source"]}


def down_fp64(tokens=(128, 1), eps=1.0, mech="laplace", draws=8, steps=8):
    """The Down projection of a Llama layer in binary32-family arithmetic (the calibrated path)
    and in binary64 (Sec. 5.5): time per online product call and the recovered error over every
    output of one step, against the exact product."""
    model = wl.LLAMA_3_2_3B
    out = {}
    for M in tokens:
        stack = MaskedStack.build(model, 1, M, draws, base_seed=23)
        layer = stack.layers[0]
        inputs = stack.inputs(29)
        _calibrate(stack, inputs, eps, mech)
        res = {}
        for mode in ("binary32", "binary64"):
            layer.fp64 = {"down"} if mode == "binary64" else set()
            ws = spl.workspace(layer.workspace_bytes(M, draws))
            layer.allocate(M, draws, workspace=ws)
            events = []

            def timer(phase, kind, group):
                if group != "down" or kind != "masked_linear_unmask":
                    return
                e = torch.cuda.Event(enable_timing=True)
                e.record()
                events.append(e)

            seed = stack.seeds[0]
            layer.refill(eps, mech, seed, 0)
            for d in range(min(steps, draws)):
                layer.online(inputs[0], eps, mech, seed, 0, d, timer=timer)
            torch.cuda.synchronize()
            times = [events[i].elapsed_time(events[i + 1]) for i in range(0, len(events), 2)]
            outs = layer.online(inputs[0], eps, mech, seed, 0, 0)
            bc = layer.bound_check(inputs[0], outs, eps, mech, seed, 0, 0)["down"]
            path = "fp64" if mode == "binary64" else _group_paths(layer, M)["down"]
            res[mode] = {"path": path, "us_per_call": 1e3 * sum(times[1:]) / max(1, len(times) - 1),
                         "mean_err": bc["mean_err"], "max_err": bc["max_err"], "max_abs_ref": bc["max_abs_ref"],
                         "max_err_over_hard_binary32": bc["max_err_over_hard"]}
        out[f"M={M}"] = res
        del stack, layer
        torch.cuda.empty_cache()
    return {"workload": f"llama-3.2-3b-shaped Down projection (8192 -> 3072) in binary32 and binary64, {mech} "
                        f"eps={eps}, M in {list(tokens)}", "down": out}


def slalom_compare(tokens=(128, 1), eps=1.0, mech="gaussian", reps=10):
    """Slalom's masking (Sec. 6.2: 8-bit fixed point, one-time pad over Z_q, exact integer product,
    modular unmask) beside this path on the outsourced projections of one Llama layer: time per
    product call and the error of the recovered output against the exact product."""
    model = wl.LLAMA_3_2_3B
    out = {}
    for M in tokens:
        stack = MaskedStack.build(model, 1, M, 2, base_seed=31)
        layer = stack.layers[0]
        inputs = stack.inputs(37)[0]
        _calibrate(stack, [inputs], eps, mech)
        seed = stack.seeds[0]
        layer.refill(eps, mech, seed, 0)
        outs = layer.online(inputs, eps, mech, seed, 0, 0)
        bc = layer.bound_check(inputs, outs, eps, mech, seed, 0, 0)
        res = {}
        for gi, g in enumerate(layer.groups):
            if g.name == "down":
                continue  # kept in the enclave by both systems (Sec. 5.5)
            X = inputs[g.name]
            Wq = torch.empty_like(g.W)
            spl.spl_slalom_quantize(Wq, g.W)
            Xt = torch.empty_like(X)
            eta = torch.empty_like(X)
            spl.spl_slalom_mask(Xt, eta, X, seed, stream_id=gi)
            ws = spl.workspace(spl.spl_f64_workspace_bytes(M, g.K, g.N))
            C = torch.empty((M, g.N), dtype=torch.float64, device=X.device)
            spl.spl_precompute_noise_product_f64(C, eta, Wq, workspace=ws)
            Y = torch.empty((M, g.N), device=X.device)
            call = lambda: spl.spl_slalom_linear_unmask(Y, Xt, Wq, C, workspace=ws)
            call()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            for _ in range(reps):
                call()
            e1.record()
            torch.cuda.synchronize()
            slalom_us = 1e3 * e0.elapsed_time(e1) / reps
            # error of each against the exact product (computed on the device in binary64)
            ref = X.double() @ g.W.double().T
            scale = float(ref.abs().max())
            ours_ev = []

            def timer(phase, kind, group, _g=g.name):
                if group == _g and kind == "masked_linear_unmask":
                    e = torch.cuda.Event(enable_timing=True)
                    e.record()
                    ours_ev.append(e)

            for d in range(reps + 1):
                layer.online(inputs, eps, mech, seed, 0, d % 2, timer=timer)
            torch.cuda.synchronize()
            ours_us = 1e3 * sum(ours_ev[i].elapsed_time(ours_ev[i + 1]) for i in range(2, len(ours_ev), 2)) / reps
            res[g.name] = {"slalom_us": slalom_us, "ours_us": ours_us,
                           "slalom_max_rel_err": float((Y.double() - ref).abs().max()) / scale,
                           "slalom_mean_abs_err": float((Y.double() - ref).abs().mean()),
                           "ours_max_rel_err": bc[g.name]["max_err"] / scale, "ours_mean_abs_err": bc[g.name]["mean_err"],
                           "ours_path": _group_paths(layer, M)[g.name]}
        out[f"M={M}"] = res
        del stack, layer
        torch.cuda.empty_cache()
    return {"workload": f"llama-3.2-3b-shaped layer, Q|K|V, O, Gate|Up: Slalom's one-time pad over Z_q (8-bit fixed "
                        f"point) vs this path ({mech} eps={eps}), M in {list(tokens)}", "compare": out}


def lm_head(tokens=(512, 1), eps=1.0, mech="gaussian", draws=8, cycles=3):
    """The Llama LM head (3072 -> 128256 after the final RMSNorm, Delta from Thm. 1) at prefill and
    decode sizes: per draw the noise + mask of X and the masked product with fused unmask, replayed
    as CUDA graphs of one bank cycle; the bank (8 draws, summed in the online order) timed apart."""
    model = wl.LLAMA_3_2_3B
    pk = _peaks()
    K, N = model.d_model, model.vocab
    W = wl.weight(N, K, seed=9001, device="cuda")
    Wt = spl.Weight.prepare(W)
    delta = spl.spl_delta_layernorm(torch.ones(K))
    stream = torch.cuda.current_stream()
    out = {}
    for M in tokens:
        path = spl.PATH_NAMES[spl.spl_resolve_path(M, K, N, "auto")]
        X = wl.activations(M, K, seed=9002, device="cuda")
        Xt = torch.empty_like(X)
        Y = torch.empty((M, N), device="cuda")
        eta = torch.empty((draws * M, K), device="cuda")
        C = torch.empty((draws * M, N), device="cuda")
        ws = spl.workspace(max(spl.spl_precompute_matched_workspace_bytes(draws * M, K, N, M),
                               spl.spl_linear_workspace_bytes(M, K, N)))
        base = torch.zeros(1, dtype=torch.int64, device="cuda")

        def refill():
            spl.spl_noise(eta, delta, eps, mech, seed=606, offset_dev=base)
            spl.spl_precompute_noise_product_matched(C, eta, Wt, M, workspace=ws)

        def online(d):
            spl.spl_noise_mask(Xt, None, X, delta, eps, mech, seed=606, offset=d * M * K // 4, offset_dev=base)
            spl.spl_masked_linear_unmask(Y, Xt, Wt, C[d * M:(d + 1) * M], workspace=ws)

        refill()
        for d in range(draws):
            online(d)
        torch.cuda.synchronize()
        g_on, g_rf = torch.cuda.CUDAGraph(), torch.cuda.CUDAGraph()
        with torch.cuda.graph(g_on):
            for d in range(draws):
                online(d)
        with torch.cuda.graph(g_rf):
            refill()
        on_t = _time_replays([g_on], 0, cycles + 1, stream)[1:]
        rf_t = _time_replays([g_rf], 0, cycles + 1, stream)[1:]
        step_ms = sum(on_t) / (cycles * draws)
        refill_ms = sum(rf_t) / cycles
        flops = 2 * M * K * N
        wbytes = 4 * K * N  # fp32 W (decode kernel) or its two fp16 halves: 4 bytes per weight either way
        byts = wbytes + 4 * M * K + 8 * M * N
        t_hbm = byts / (pk["hbm_gbs"] * 1e9)
        t_tc = flops / (_path_peak(path, pk) * 1e12)
        bound = "hbm" if t_hbm >= t_tc else "tensor"
        out[f"M={M}"] = {"path": path, "ms_per_step": step_ms, "tflops": flops / (step_ms * 1e-3) / 1e12,
                         "gbs": byts / (step_ms * 1e-3) / 1e9, "bound": bound,
                         "frac": max(t_hbm, t_tc) * 1e3 / step_ms,
                         "bank_refill_ms": refill_ms,
                         "bank_refill_tflops": draws * flops / (refill_ms * 1e-3) / 1e12}
        del g_on, g_rf, X, Xt, Y, eta, C, ws
        torch.cuda.empty_cache()
    return {"workload": f"llama-3.2-3b LM head (3072 -> 128256), {mech} eps={eps}, banks of {draws} draws, "
                        f"tokens {list(tokens)}", "lm_head": out, "peak_source": pk["source"]}


WORKLOADS = {"llama_stack_detail": llama_stack, "qwen_stack": qwen_stack, "qwen_sweep": qwen_sweep, "down_fp64": down_fp64,
             "slalom": slalom_compare, "lm_head": lm_head}
