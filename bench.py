#!/usr/bin/env python3
"""Benchmark of the BitsMoE quantized MoE-layer forward on GB300.

Default workload: the Qwen3-30B-A3B-shaped MoE layer (hidden 2048, 128 experts,
top-8, intermediate 768, shared-basis rank 2048, 2.0 mean unit bits, group 128),
batch-1 decode.  A step is one bitsmoe_moe_forward call (routing, shared-basis
projection, gate/up factors + SwiGLU, down factor + weighted expert sum, output
basis) on one synthetic token.

  value   tokens/s with inputs resident in HBM: K forwards replayed from CUDA
          graphs on one stream, timed with CUDA events; the layer rotates over
          `--copies` packed copies (each step touches ~36 MB; the rotation set is
          far larger than the 129 MB L2, so weights stream from HBM).
  e2e     the same metric through bitsmoe_moe_forward_host: pinned host input
          -> device, forward, y -> pinned host, synchronised, every step.
  roofline  dominant phase (from bitsmoe_profile_forward, phases serialised and
          timed with CUDA events), algorithmic bytes / its duration, against the
          measured HBM copy bandwidth.
  cpu_baseline  the fp64 oracle on the host cores, on a bounded sample.

`--task quantize` measures the per-unit quantiser instead (bitsmoe_quantize_units on a
Qwen3-shaped layer's 786,432 float units; roofline against the fp32 lanes, since the
MSE-optimal scale search is ALU-bound) and `--task allocate` the per-projection bit
allocation (bitsmoe_allocate_bits on the same layer's three projections under the paper's
budget; roofline of the dominant phase against HBM).  Both print the same kind of JSON line.

`--impl reference` times the oracle (the only reference for this path) on the
host cores instead and prints the same JSON line with "impl": "reference".
Multi-GPU: the forward does not shard, so `--gpus N` under torchrun runs N
independent replicas (weak scaling, no collective in the data path).
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import synth  # noqa: E402

METRIC = "MoE-layer decode tokens/s at 2.0 avg bits; achieved HBM GB/s vs ~8 TB/s peak"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
PHASES = ["route", "basis_proj_gate_up", "gate_up_factors", "down_factor_sum", "out_basis"]


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            return json.load(f), "measured"
    except Exception:
        return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


def measured_traffic(profile, sources):
    """DRAM bytes per launch of a kernel from a committed ncu summary, or None when
    the kernel's sources changed since that capture (the summary records their hash)."""
    import hashlib
    try:
        lines = open(os.path.join(ROOT, "profiles", profile)).read().splitlines()
        kv = dict(l.split(":", 1) for l in lines if ":" in l and not l.startswith("#"))
        h = hashlib.sha256()
        for src in sources:
            h.update(open(os.path.join(ROOT, "paper_2606_00079_gb300", "csrc", src), "rb").read())
        if kv.get("source_sha256", "").strip() != h.hexdigest():
            return None
        return int(kv["dram_bytes_per_launch"].strip())
    except Exception:
        return None


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def rank_barrier(world):
    """All ranks meet here (N > 1) before and after the timed region."""
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(ms, world, device):
    """The slowest rank's time: the job's time for the units all ranks processed."""
    if world <= 1:
        return float(ms)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(ms)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world, steps, tokens, ms):
    """Whole-job tokens/s: every rank processed steps x tokens in the slowest rank's time."""
    return world * steps * tokens / (ms / 1e3)


def host_route(logits, k):
    """Experts each token is routed to (k largest logits, ties to the lower index):
    used only to count the algorithmic bytes of a step."""
    out = []
    for row in logits:
        order = np.lexsort((np.arange(row.size), -row.astype(np.float64)))[:k]
        out.append(order)
    return np.array(out)


# --------------------------------------------------------------------------
# clocks sampled during the timed region
# --------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("timestamp,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.idx = gpu_index
        self.proc = None
        self.file = None
        self.t0 = self.t1 = None

    def start(self):
        try:
            self.file = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.idx), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "20"], stdout=self.file, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None

    def mark(self, which):
        setattr(self, which, time.time())

    def stop(self):
        if not self.proc:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"], "samples": 0}
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except Exception:
            self.proc.kill()
        self.file.flush()
        self.file.seek(0)
        rows = []
        for line in self.file.read().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                ts = time.mktime(time.strptime(parts[0].split(".")[0], "%Y/%m/%d %H:%M:%S"))
                frac = float("0." + parts[0].split(".")[1]) if "." in parts[0] else 0.0
                rows.append((ts + frac, float(parts[1]), float(parts[2]), parts[5:9]))
            except Exception:
                continue
        os.unlink(self.file.name)
        window = [r for r in rows if self.t0 and self.t1 and self.t0 - 0.05 <= r[0] <= self.t1 + 0.05]
        src = "timed_region"
        l0, l1 = getattr(self, "l0", None), getattr(self, "l1", None)
        if len(window) < 20 and l0 and l1:   # a short timed region: the same load around it as well
            window = [r for r in rows if l0 <= r[0] <= l1]
            src = "timed_region_and_the_same_load_around_it"
        if not window:
            window, src = rows, "whole_run"
        if not window:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no_samples"], "samples": 0}
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in window for i, v in enumerate(r[3]) if v.lower().startswith("active")})
        return {"sm_mhz": statistics.median(r[1] for r in window), "sm_max_mhz": max(r[2] for r in window),
                "reasons": reasons, "samples": len(window), "window": src}


# --------------------------------------------------------------------------
# CPU baseline: the oracle on the host cores
# --------------------------------------------------------------------------
def oracle_tokens_per_s(spec, layer, T, budget_s=12.0, max_steps=None, seed=0):
    import oracle
    times, toks, steps = [], 0, 0
    t_start = time.perf_counter()
    while True:
        x, logits = synth.make_inputs(spec, T, seed=seed, step=1000 + steps)
        t = time.perf_counter()
        oracle.moe_forward_factored(layer, x, logits, spec.top_k)
        times.append(time.perf_counter() - t)
        toks += T
        steps += 1
        if (max_steps and steps >= max_steps) or time.perf_counter() - t_start > budget_s:
            break
    return toks / sum(times), steps, sum(times)


def oracle_one_core(spec, T, budget_s=12.0):
    """The oracle's factored forward on one host core (BLAS threads limited to 1 in a child
    process), on a bounded sample: a layer of the workload's dims whose experts number the
    ones a T-token step routes to (at most T * top_k), so that a step's work is the same."""
    E = min(spec.E, T * spec.top_k)
    code = (
        "import sys, time, json\n"
        f"sys.path.insert(0, {ROOT!r})\n"
        "import synth, oracle\n"
        f"spec = synth.scaled_spec(synth.WORKLOADS[{spec.name!r}], E={E})\n"
        "layer = synth.make_layer(spec, seed=0)\n"
        "n, secs = 0, 0.0\n"
        f"while secs < {budget_s} and n < 64:\n"
        f"    x, lg = synth.make_inputs(spec, {T}, seed=0, step=1000 + n)\n"
        "    t0 = time.perf_counter()\n"
        "    oracle.moe_forward_factored(layer, x, lg, spec.top_k)\n"
        "    secs += time.perf_counter() - t0\n"
        "    n += 1\n"
        "print(json.dumps({'steps': n, 'secs': secs}))\n")
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    try:
        r = subprocess.run([sys.executable, "-c", code], capture_output=True, text=True, env=env, timeout=600)
        d = json.loads(r.stdout.strip().splitlines()[-1])
    except Exception as e:   # reported, not fatal: the GPU line stands without it
        return {"value": None, "unit": "tokens/s", "cores": 1, "kind": "oracle", "sample": f"failed: {e}"}
    layers = spec.layers
    v = d["steps"] * T / d["secs"] / layers
    return {"value": v, "unit": "tokens/s", "cores": 1, "kind": "oracle",
            "sample": f"{d['steps']} fp64 numpy factored forwards of {T} token(s) on a layer with the workload's "
                      f"dims and {E} experts (BLAS threads 1, {d['secs']:.1f} s)"
                      + (f", extrapolated to {layers} layers" if layers > 1 else "")}


def cpu_cores():
    try:
        from threadpoolctl import threadpool_info
        n = max((i.get("num_threads", 1) for i in threadpool_info()), default=None)
        if n:
            return int(n)
    except Exception:
        pass
    return os.cpu_count() or 1


# --------------------------------------------------------------------------
def run_reference(args, spec, T):
    rank, world, _ = dist_env()
    if rank != 0:
        return
    layer = synth.make_layer(spec, seed=0)
    # warmup steps (bounded), then K steps each a bounded sample: one oracle forward of T tokens
    oracle_tokens_per_s(spec, layer, T, budget_s=5.0, max_steps=max(1, min(args.warmup, 3)))
    budget = float(os.environ.get("BITSMOE_REF_BUDGET_S", "90"))
    v, steps, secs = oracle_tokens_per_s(spec, layer, T, budget_s=budget, max_steps=args.steps)
    cores = cpu_cores()
    line = {
        "impl": "reference", "metric": METRIC, "value": v, "unit": "tokens/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * secs / steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": config_of(spec, T, args),
        "cpu_baseline": {"value": v, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                         "sample": f"{steps} of {args.steps} steps timed ({secs:.1f} s), one fp64 numpy "
                                   f"factored forward of {T} token(s) per step"},
        "e2e": {"value": v, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def config_of(spec, T, args):
    return {"workload": f"{spec.name}: Qwen3-30B-A3B-shaped MoE layer" if spec.name.startswith("qw3") else spec.name,
            "hidden": spec.D, "experts": spec.E, "top_k": spec.top_k, "intermediate": spec.I,
            "rank": spec.n, "group": spec.group, "mean_unit_bits": spec.mean_bits, "tokens_per_step": T,
            "l2": f"rotating {args.copies} packed layer copies (>> 129 MB L2)", "seed": 0}


def run_stack(args, spec, T, torch, bm, dev, rank, world, local):
    """48-layer pre-norm MoE FFN stack: a step feeds one batch of hidden states
    through every block (RMSNorm + router + quantized MoE + residual)."""
    eps = 1e-6
    layers, routers, moved = [None] * spec.layers, [], []
    pend = []

    def pack(l, host):
        layers[l] = bm.bitsmoe_pack(host, device=local)

    for l in range(spec.layers):
        host = synth.make_layer(spec, seed=0, layer_index=l)
        th = threading.Thread(target=pack, args=(l, host))
        th.start()
        pend.append(th)
        routers.append(torch.from_numpy(synth.make_router_weight(spec, seed=0, layer_index=l).view(np.int16)).to(dev))
        if len(pend) > 1:
            pend.pop(0).join()
    for th in pend:
        th.join()
    for L in layers:
        moved.append(np.array([L.expert_moved_bytes(e) for e in range(spec.E)], dtype=np.float64))
    k = spec.top_k
    NI = 8
    h0 = [torch.from_numpy(synth.make_hidden(spec, T, seed=0, step=i)).to(dev) for i in range(NI)]
    h = torch.empty((T, spec.D), dtype=torch.float32, device=dev)
    ws = bm.Workspace(layers[0], T, k, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def step(i, st):
        h.copy_(h0[i % NI])
        for l in range(spec.layers):
            bm.bitsmoe_moe_block_forward(h.data_ptr(), routers[l].data_ptr(), eps, T, k, layers[l], ws.ptr,
                                         ws.nbytes, st.cuda_stream)

    # realised routing of step 0, layer by layer (outside the timed region): byte accounting
    x = torch.empty((T, spec.D), dtype=torch.int16, device=dev)
    lg = torch.empty((T, spec.E), dtype=torch.float32, device=dev)
    step_bytes = 0.0
    with torch.cuda.stream(stream):
        h.copy_(h0[0])
        for l in range(spec.layers):
            bm.bitsmoe_rmsnorm_router(h.data_ptr(), routers[l].data_ptr(), eps, T, spec.D, spec.E, x.data_ptr(),
                                      lg.data_ptr(), stream.cuda_stream)
            stream.synchronize()
            used = np.unique(host_route(lg.cpu().numpy(), k))
            # bases, routed experts' factors, router matrix, hidden state in and out
            step_bytes += (3.0 * spec.D * spec.n * 2 + moved[l][used].sum() + spec.E * spec.D * 2 +
                           2.0 * T * spec.D * 4)
            bm.bitsmoe_moe_block_forward(h.data_ptr(), routers[l].data_ptr(), eps, T, k, layers[l], ws.ptr,
                                         ws.nbytes, stream.cuda_stream)
    stream.synchronize()
    with torch.cuda.stream(stream):
        for i in range(min(args.warmup, 3)):
            step(i, stream)
    stream.synchronize()
    G = max(1, min(args.graph // spec.layers or 1, args.steps))

    def capture(n, off):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(n):
                step(off + i, stream)
        return g

    nfull, rem = divmod(args.steps, G)
    g_main = capture(G, 0)
    g_rem = capture(rem, 0) if rem else None
    with torch.cuda.stream(stream):
        for _ in range(max(1, args.warmup // G)):
            g_main.replay()
    stream.synchronize()
    clk = ClockSampler(local)
    clk.start()
    rank_barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk.mark("t0")
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(nfull):
            g_main.replay()
        if g_rem is not None:
            g_rem.replay()
    e1.record(stream)
    e1.synchronize()
    clk.mark("t1")
    torch.cuda.synchronize()
    rank_barrier(world)
    ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    clocks = clk.stop()
    value = job_throughput(world, args.steps, T, ms)
    gbs = step_bytes * args.steps / (ms / 1e3) / 1e9
    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    # e2e: host hidden state in, host hidden state out, every step
    hh = torch.from_numpy(synth.make_hidden(spec, T, seed=0, step=0)).pin_memory()
    ho = torch.empty((T, spec.D), dtype=torch.float32).pin_memory()
    ne = max(3, min(args.steps, 50))
    t0 = time.perf_counter()
    for i in range(ne):
        with torch.cuda.stream(stream):
            h.copy_(hh, non_blocking=True)
            for l in range(spec.layers):
                bm.bitsmoe_moe_block_forward(h.data_ptr(), routers[l].data_ptr(), eps, T, k, layers[l], ws.ptr,
                                             ws.nbytes, stream.cuda_stream)
            ho.copy_(h, non_blocking=True)
        stream.synchronize()
    e2e_s = time.perf_counter() - t0
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": dict(config_of(spec, T, args), layers=spec.layers, l2="48 distinct layers per step (>> L2)"),
        "hbm_gbs": gbs, "hbm_frac_of_8tbs": gbs / NOMINAL_HBM_GBS, "hbm_frac_of_measured": gbs / peak,
        "bytes_per_step": step_bytes,
        # the step is 48 block forwards back to back: its roofline is the step's, algorithmic bytes over
        # the timed region
        "roofline": {"bound": "hbm", "kernel": f"{spec.layers} pre-norm MoE blocks (the whole step)",
                     "achieved": gbs, "peak": peak, "peak_source": peak_src, "unit": "GB/s", "frac": gbs / peak,
                     "traffic": None, "bytes_per_launch": step_bytes / spec.layers,
                     "duration_us": ms / args.steps * 1e3 / spec.layers,
                     "duration_source": "CUDA events over the timed region / (steps x layers)",
                     "frac_of_8tbs": gbs / NOMINAL_HBM_GBS},
        "e2e": {"value": world * ne * T / e2e_s, "unit": "tokens/s", "steps": ne,
                "h2d_bytes_per_step": T * spec.D * 4, "d2h_bytes_per_step": T * spec.D * 4},
        "clocks": clocks,
        "gpu_launches": args.steps * spec.layers * bm.bitsmoe_block_forward_launches(layers[0], T, k),
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        # the oracle on one layer of the stack (RMSNorm, router, factored MoE forward), T tokens,
        # extrapolated to the 48 layers of a step
        import oracle
        host = synth.make_layer(spec, seed=0, layer_index=0)
        wr = synth.make_router_weight(spec, seed=0, layer_index=0)
        hs = synth.make_hidden(spec, T, seed=0, step=0).astype(np.float64)
        reps, secs = 0, 0.0
        while secs < 12.0 and reps < 8:
            t0 = time.perf_counter()
            xb = synth.f32_to_bf16_bits(oracle.rms_norm(hs, eps).astype(np.float32))
            lg = oracle.router_logits(wr, xb)
            oracle.moe_forward_factored(host, xb, lg, k)
            secs += time.perf_counter() - t0
            reps += 1
        per_layer = secs / reps
        line["cpu_baseline"] = {"value": T / (per_layer * spec.layers), "unit": "tokens/s", "cores": cpu_cores(),
                                "kind": "oracle",
                                "sample": f"{reps} forwards of one stacked layer ({T} token(s), fp64 numpy, "
                                          f"{per_layer * 1e3:.0f} ms each), extrapolated to {spec.layers} layers"}
        line["cpu_baseline_1core"] = oracle_one_core(spec, T)
    return line


QUANT_METRIC = "spectral units quantised/s (per-unit Q_b into the stored format, MSE-optimal group scales)"
# lane-instructions of the definition per (element, candidate) of the scale search: quotient as a
# product, two clamp bounds, one rounding, fused product-difference, square, accumulate
QUANT_OPS_PER_EVAL = 7
FP32_LANES_PER_SM = 128


def quant_inputs(torch, U, I, dist, seed, dev):
    """Unit-norm Gaussian directions (fp32, U x I) and i.i.d. bit-widths, drawn on the device
    from a seeded generator (the layer-sized input is 2.4 GB)."""
    g = torch.Generator(device=dev)
    g.manual_seed(seed)
    P = torch.empty((U, I), dtype=torch.float32, device=dev)
    for u0 in range(0, U, 65536):
        blk = torch.randn((min(65536, U - u0), I), generator=g, device=dev, dtype=torch.float32)
        P[u0:u0 + blk.shape[0]] = blk / blk.norm(dim=1, keepdim=True)
    vals = torch.tensor([b for b, _ in dist], dtype=torch.uint8, device=dev)
    probs = torch.tensor([p for _, p in dist], dtype=torch.float64, device=dev)
    bits = vals[torch.multinomial(probs, U, replacement=True, generator=g)]
    return P, bits.contiguous()


def quant_config(spec, U, I, group, grid):
    return {"workload": f"quantiser: {spec.name} layer's spectral units (3 x {spec.E} x {spec.n} units "
                        f"of {I}, group {group}, mean {spec.mean_bits} bits, {grid} scale candidates)",
            "units": U, "unit_length": I, "group": group, "grid": grid,
            "l2": f"input {U * I * 4 / 1e9:.2f} GB per step (129 MB L2)"}


def alloc_config(spec, U, I, budget, gamma):
    return {"workload": f"bit allocation: {spec.name} layer, 3 projections x {U} units of {I}, budget "
                        f"B_h = {budget} (b_eq {spec.mean_bits}), gamma {gamma}",
            "units": 3 * U, "unit_length": I, "budget_per_projection": budget,
            "l2": f"input {3 * U * I * 4 / 1e9:.2f} GB per step (129 MB L2)"}


def run_reference_task(args, spec):
    """Reference arm of --task quantize / allocate: the oracle of that step on the host cores,
    each step a bounded sample of the same workload (the units/s of the sample)."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    I = spec.I
    budget_s = float(os.environ.get("BITSMOE_REF_BUDGET_S", "90")) / max(1, args.steps)
    if args.task == "importance":
        cpu = imp_oracle_rate(spec, budget_s=min(60.0, float(os.environ.get("BITSMOE_REF_BUDGET_S", "90"))))
        line = {
            "impl": "reference", "metric": IMP_METRIC, "value": cpu["value"], "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * args.calib_tokens / cpu["value"], "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": imp_config(spec, args.calib_tokens),
            "cpu_baseline": cpu,
            "e2e": {"value": cpu["value"], "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }
        print(json.dumps(line), flush=True)
        return
    if args.task == "decompose":
        cpu = dec_oracle_rate(spec, budget_s=min(60.0, float(os.environ.get("BITSMOE_REF_BUDGET_S", "90"))))
        n = min(spec.D, spec.E * spec.I)
        line = {
            "impl": "reference", "metric": DEC_METRIC, "value": cpu["value"], "unit": "units/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1000.0 * spec.E * n / cpu["value"], "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "config": dec_config(spec),
            "cpu_baseline": cpu,
            "e2e": {"value": cpu["value"], "unit": "units/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
        }
        print(json.dumps(line), flush=True)
        return
    if args.task == "quantize":
        from oracle import quantizer as Q
        U = args.units or 3 * spec.E * spec.n
        config = quant_config(spec, U, I, spec.group, args.grid)
        chunk = 2048
        P, bits = synth.make_float_units(chunk, I, seed=0, bits_dist=dict(spec.bits_dist))
        run = lambda: Q.quantize_units(P, bits, spec.group, args.grid)
        metric, what = QUANT_METRIC, f"fp32 numpy quantiser on chunks of {chunk} units"
    else:
        from oracle import allocator as Aor
        U = args.units or spec.E * spec.n
        budget = Aor.projection_budget(U // spec.n, spec.n, I, spec.mean_bits) if U % spec.n == 0 else None
        if budget is None:
            from fractions import Fraction
            budget = int((Fraction(U) * Fraction(str(spec.mean_bits)) * I - 16 * spec.n * spec.n) // I)
        config = alloc_config(spec, U, I, budget, 0.5)
        chunk = 16384
        P, _ = synth.make_float_units(chunk, I, seed=0)
        an = (((np.arange(chunk) % spec.n) + 1.0) ** -0.5).astype(np.float32)
        bn = np.random.default_rng([0, 5]).lognormal(0.0, 1.0, chunk).astype(np.float32)
        kap = {2: KAPPA_TABLE[0], 3: KAPPA_TABLE[1], 4: KAPPA_TABLE[2]}
        run = lambda: Aor.allocate(Aor.costs(P, an, bn, 0.5, kap), int(budget * chunk / U))
        metric, what = ALLOC_METRIC, f"numpy allocation of chunks of {chunk} units (budget scaled)"
    for _ in range(max(1, min(args.warmup, 3))):
        run()
    done, secs = 0, 0.0
    for _ in range(args.steps):
        t0 = time.perf_counter()
        reps = 0
        while True:   # one step: at least one chunk, up to the per-step budget
            run()
            reps += 1
            if time.perf_counter() - t0 > min(budget_s, 10.0) or reps >= 64:
                break
        secs += time.perf_counter() - t0
        done += reps * chunk
    v = done / secs
    line = {
        "impl": "reference", "metric": metric, "value": v, "unit": "units/s", "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1000.0 * secs / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f32", "data": "synthetic",
        "config": config,
        "cpu_baseline": {"value": v, "unit": "units/s", "cores": cpu_cores(), "kind": "oracle",
                         "sample": f"{done} units in {args.steps} steps ({secs:.1f} s), {what}"},
        "e2e": {"value": v, "unit": "units/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def run_quantize(args, spec, rank, world, local):
    """Quantiser of one Qwen3-shaped layer's spectral units (U = 3 E n units of length I, group
    128, bits from the workload's distribution, 256 scale candidates): one
    bitsmoe_quantize_units launch per step; input 2.4 GB >> L2."""
    import torch
    import paper_2606_00079_gb300 as bm
    dev = torch.device("cuda", local)
    U, I, group, grid = args.units or 3 * spec.E * spec.n, spec.I, spec.group, args.grid
    P, bits = quant_inputs(torch, U, I, spec.bits_dist, 1000 + rank, dev)
    ng = I // group
    codes = torch.empty((U, I), dtype=torch.int16, device=dev)
    scale = torch.empty((U, ng), dtype=torch.int16, device=dev)
    zero = torch.empty((U, ng), dtype=torch.int16, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def step():
        bm.bitsmoe_quantize_units(P.data_ptr(), bits.data_ptr(), U, I, group, grid, codes.data_ptr(),
                                  scale.data_ptr(), zero.data_ptr(), status.data_ptr(), stream.cuda_stream)

    with torch.cuda.stream(stream):
        for _ in range(max(3, min(args.warmup, 5))):
            step()
    stream.synchronize()
    if int(status.item()) != 0:
        raise bm.BitsMoEError(int(status.item()), "bitsmoe_quantize_units")
    clk = ClockSampler(local)
    clk.start()
    rank_barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk.mark("t0")
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    e1.synchronize()
    clk.mark("t1")
    torch.cuda.synchronize()
    rank_barrier(world)
    ms_own = e0.elapsed_time(e1)
    ms = max_over_ranks(ms_own, world, dev)
    clocks = clk.stop()
    value = job_throughput(world, args.steps, U, ms)
    # roofline: the search's lane-instructions against the fp32 lanes at the clock seen under load
    low = ((bits >= 2) & (bits <= 4)).sum().item()
    evals = float(low) * ng * group * grid
    ops = evals * QUANT_OPS_PER_EVAL
    sec = ms_own / args.steps / 1e3
    peaks, _ = measured_peaks()
    sm_mhz = clocks.get("sm_mhz") or float(peaks.get("sm_max_mhz", 2070.0))
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    peak = sms * FP32_LANES_PER_SM * sm_mhz * 1e6 / 1e12
    peak_max = sms * FP32_LANES_PER_SM * float(peaks.get("sm_max_mhz", 2070.0)) * 1e6 / 1e12
    achieved = ops / sec / 1e12
    hbm_bytes = U * I * 4.0 + U * I * 2.0 + U + 2.0 * U * ng * 2
    roofline = {"bound": "alu", "kernel": "k_quantize (scale search of the 2-4 bit units)", "achieved": achieved,
                "peak": peak, "unit": "T lane-instr/s", "frac": achieved / peak,
                "peak_source": f"{sms} SMs x {FP32_LANES_PER_SM} fp32 lanes x {sm_mhz:.0f} MHz (median SM clock "
                               "under load)",
                "frac_at_max_clock": achieved / peak_max, "traffic": None,
                "ops_per_eval": QUANT_OPS_PER_EVAL, "evals_per_launch": evals,
                "hbm_gbs": hbm_bytes / sec / 1e9, "bytes_per_launch": hbm_bytes,
                "duration_us": sec * 1e6}
    # e2e: pinned host units in, codes / scales / zeros out, every step
    ne = 3
    Ph = P.cpu().pin_memory()
    ch = torch.empty_like(codes, device="cpu").pin_memory()
    sh = torch.empty_like(scale, device="cpu").pin_memory()
    zh = torch.empty_like(zero, device="cpu").pin_memory()
    t0 = time.perf_counter()
    for _ in range(ne):
        with torch.cuda.stream(stream):
            P.copy_(Ph, non_blocking=True)
            step()
            ch.copy_(codes, non_blocking=True)
            sh.copy_(scale, non_blocking=True)
            zh.copy_(zero, non_blocking=True)
        stream.synchronize()
    e2e_s = time.perf_counter() - t0
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from oracle import quantizer as Q
        n_done, secs, chunk = 0, 0.0, 0
        while secs < 12.0 and chunk < 64:   # chunks of 4096 units, about 12 s of CPU work
            Pn, bn = synth.make_float_units(4096, I, seed=chunk, bits_dist=dict(spec.bits_dist))
            t = time.perf_counter()
            Q.quantize_units(Pn, bn, group, grid)
            secs += time.perf_counter() - t
            n_done += 4096
            chunk += 1
        cpu = {"value": n_done / secs, "unit": "units/s", "cores": cpu_cores(), "kind": "oracle",
               "sample": f"{n_done} units of {I} (same bit distribution), fp32 numpy quantiser, {secs:.1f} s"}
    if rank == 0:
        line = {
            "metric": QUANT_METRIC, "value": value, "unit": "units/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": quant_config(spec, U, I, group, grid),
            "roofline": roofline, "cpu_baseline": cpu,
            "e2e": {"value": world * ne * U / e2e_s, "unit": "units/s", "steps": ne,
                    "h2d_bytes_per_step": U * I * 4, "d2h_bytes_per_step": U * I * 2 + 2 * U * ng * 2},
            "clocks": clocks, "gpu_launches": args.steps,
        }
        print(json.dumps(line), flush=True)


IMP_METRIC = "calibration tokens/s (importance beta of every unit of an MoE layer from calibration activations)"
FP32_FLOPS_PER_SM_CLK = 256   # 128 fp32 lanes x 2 flops per fused multiply-add


def imp_flops(spec, T):
    """FLOPs of one importance step: Z = Phi^T X for gate and up, the token contraction of z^2,
    the experts' gate/up factors on their tokens, the down factor's transposed product."""
    D, n, E, I, k = spec.D, spec.n, spec.E, spec.I, spec.top_k
    return 2.0 * 2 * n * D * T + 2.0 * 2 * n * T * E + 2.0 * 2 * I * n * T * k + 2.0 * n * I * T * k


def imp_config(spec, T):
    return {"workload": f"importance: {spec.name} layer's float factors (hidden {spec.D}, {spec.E} experts, top-"
                        f"{spec.top_k}, intermediate {spec.I}, rank {spec.n}), {T} calibration tokens",
            "tokens": T, "l2": f"float factors {3 * spec.E * spec.I * spec.n * 4 / 1e9:.2f} GB per step (129 MB L2)"}


def run_importance(args, spec, rank, world, local):
    """Importance beta of one Qwen3-shaped layer from T calibration tokens: one bitsmoe_importance
    call per step on float factors drawn on the device (orthonormal-scale bases, j^-1/2 energies,
    unit-norm spectral vectors), bf16 N(0, 1) activations, N(0, 1) router logits."""
    import torch
    import paper_2606_00079_gb300 as bm
    dev = torch.device("cuda", local)
    T, D, n, E, I, k = args.calib_tokens, spec.D, spec.n, spec.E, spec.I, spec.top_k
    g = torch.Generator(device=dev)
    g.manual_seed(4000 + rank)
    basis = [torch.randn((D, n), generator=g, device=dev) / float(np.sqrt(D)) for _ in range(2)]
    j = torch.arange(1, n + 1, device=dev, dtype=torch.float32)
    alpha = [j.pow(-0.5).repeat(E, 1).contiguous() for _ in range(2)]
    factor = []
    for _ in range(3):
        f = torch.randn((E, I, n), generator=g, device=dev)
        factor.append((f / f.norm(dim=1, keepdim=True)).contiguous())
    x = (torch.randn((T, D), generator=g, device=dev).to(torch.bfloat16)).view(torch.int16).contiguous()
    logits = torch.randn((T, E), generator=g, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def step():
        return bm.importance(x, logits, k, basis, alpha, factor, stream=stream)

    with torch.cuda.stream(stream):
        for _ in range(max(3, min(args.warmup, 5))):
            step()
    stream.synchronize()
    clk = ClockSampler(local)
    clk.start()
    rank_barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk.mark("t0")
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(args.steps):
            step()
    e1.record(stream)
    e1.synchronize()
    clk.mark("t1")
    torch.cuda.synchronize()
    rank_barrier(world)
    ms_own = e0.elapsed_time(e1)
    ms = max_over_ranks(ms_own, world, dev)
    clocks = clk.stop()
    value = job_throughput(world, args.steps, T, ms)
    flops = imp_flops(spec, T)
    sec = ms_own / args.steps / 1e3
    peaks, _ = measured_peaks()
    sm_mhz = clocks.get("sm_mhz") or float(peaks.get("sm_max_mhz", 2070.0))
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    peak = sms * FP32_FLOPS_PER_SM_CLK * sm_mhz * 1e6 / 1e12
    roofline = {"bound": "alu", "kernel": "bitsmoe_importance (fp32 contractions on the CUDA cores)",
                "achieved": flops / sec / 1e12, "peak": peak, "unit": "TFLOP/s", "frac": flops / sec / 1e12 / peak,
                "peak_source": f"{sms} SMs x 128 fp32 lanes x 2 flops x {sm_mhz:.0f} MHz (median SM clock under load)",
                "traffic": None, "flops_per_launch": flops, "duration_us": sec * 1e6}
    # e2e: pinned host activations and logits in, beta out, every step (the factors stay resident)
    ne = 3
    xh = x.cpu().pin_memory()
    lh = logits.cpu().pin_memory()
    bh = torch.empty((3, E, n), dtype=torch.float32).pin_memory()
    t0 = time.perf_counter()
    for _ in range(ne):
        with torch.cuda.stream(stream):
            x.copy_(xh, non_blocking=True)
            logits.copy_(lh, non_blocking=True)
            bh.copy_(step(), non_blocking=True)
        stream.synchronize()
    e2e_s = time.perf_counter() - t0
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = imp_oracle_rate(spec, budget_s=12.0)
    if rank == 0:
        line = {
            "metric": IMP_METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": imp_config(spec, T),
            "roofline": roofline, "cpu_baseline": cpu,
            "e2e": {"value": world * ne * T / e2e_s, "unit": "tokens/s", "steps": ne,
                    "h2d_bytes_per_step": T * D * 2 + T * E * 4, "d2h_bytes_per_step": 3 * E * n * 4},
            "clocks": clocks, "gpu_launches": args.steps * 7,
        }
        print(json.dumps(line), flush=True)


def imp_oracle_rate(spec, budget_s=12.0):
    """The calibration oracle (fp64 numpy) on the host cores, on a bounded sample: a layer with
    the workload's D, n and I and top_k + 1 experts, 32 tokens per call (calibration tokens/s)."""
    from oracle import calibration as Co
    rng = np.random.default_rng(5)
    E = spec.top_k + 1
    D, n, I, T = spec.D, spec.n, spec.I, 32
    Phi = [np.linalg.qr(rng.standard_normal((D, n)))[0] for _ in range(3)]
    al = [np.tile(np.arange(1, n + 1) ** -0.5, (E, 1)) for _ in range(3)]
    P = [[rng.standard_normal((I, n)) / np.sqrt(I) for _ in range(E)] for _ in range(3)]
    x = synth.f32_to_bf16_bits(rng.standard_normal((T, D)).astype(np.float32))
    lg = rng.standard_normal((T, E)).astype(np.float32)
    n_done, secs = 0, 0.0
    while secs < budget_s and n_done < 64 * T:
        t0 = time.perf_counter()
        Co.factor_importance(Phi, al, P, x, lg, spec.top_k)
        secs += time.perf_counter() - t0
        n_done += T
    return {"value": n_done / secs * (E / spec.E), "unit": "tokens/s", "cores": cpu_cores(), "kind": "oracle",
            "sample": f"{n_done} tokens through factor_importance on a layer with {E} experts of the workload's dims "
                      f"({secs:.1f} s), scaled to {spec.E} experts by the per-expert work"}


DEC_METRIC = ("spectral units/s (shared-basis decomposition of one projection: Gram, Jacobi eigensolver, "
              "basis, spectral energies and vectors)")


def dec_config(spec):
    return {"workload": f"shared-basis decomposition: the gate projection of a {spec.name} layer ({spec.E} experts "
                        f"of {spec.I} x {spec.D} fp32 weights, rank {min(spec.D, spec.E * spec.I)})",
            "experts": spec.E, "intermediate": spec.I, "hidden": spec.D, "side": "in",
            "l2": f"weights {spec.E * spec.I * spec.D * 4 / 1e9:.2f} GB per step (129 MB L2)"}


def dec_oracle_rate(spec, budget_s=20.0):
    """The decomposition oracle (fp64 numpy SVD) on the host cores, on a bounded sample: the
    workload's feature dimension with fewer experts (spectral units/s of the sample)."""
    import oracle
    rng = np.random.default_rng(6)
    E = 8
    W = [(rng.standard_normal((spec.I, spec.D)) / np.sqrt(spec.D)).astype(np.float32) for _ in range(E)]
    n_units, secs, calls = 0, 0.0, 0
    while secs < budget_s and calls < 4:
        t0 = time.perf_counter()
        oracle.shared_basis_decompose(W, "in")
        secs += time.perf_counter() - t0
        n_units += E * min(spec.D, E * spec.I)
        calls += 1
    return {"value": n_units / secs, "unit": "units/s", "cores": cpu_cores(), "kind": "oracle",
            "sample": f"{calls} decompositions of {E} experts of {spec.I} x {spec.D} (oracle.shared_basis_decompose, "
                      f"numpy SVD in fp64, {secs:.1f} s); the full workload has {spec.E} experts"}


def run_decompose(args, spec, rank, world, local):
    """Shared-basis decomposition of one Qwen3-shaped projection (gate: E experts of I x D fp32
    weights, N(0, 1/D)) per step: bitsmoe_shared_basis, all of its launches timed."""
    import torch
    import paper_2606_00079_gb300 as bm
    dev = torch.device("cuda", local)
    E, I, D = spec.E, spec.I, spec.D
    n = min(D, E * I)
    g = torch.Generator(device=dev)
    g.manual_seed(5000 + rank)
    W = (torch.randn((E, I, D), generator=g, device=dev) / float(np.sqrt(D))).contiguous()
    stream = torch.cuda.Stream(device=dev)
    phi = torch.empty((D, n), dtype=torch.float32, device=dev)
    sig = torch.empty((n,), dtype=torch.float32, device=dev)
    alpha = torch.empty((E, n), dtype=torch.float32, device=dev)
    P = torch.empty((E, n, I), dtype=torch.float32, device=dev)
    info = torch.zeros((2,), dtype=torch.int32, device=dev)
    nb = int(bm._lib().bitsmoe_decompose_workspace_bytes(0, E, I, D))
    ws = torch.empty(nb + 256, dtype=torch.uint8, device=dev)
    wsp = (ws.data_ptr() + 255) // 256 * 256

    def step():
        bm._check(bm._lib().bitsmoe_shared_basis(0, W.data_ptr(), E, I, D, phi.data_ptr(), sig.data_ptr(),
                                                alpha.data_ptr(), P.data_ptr(), wsp, nb, 30, info.data_ptr(),
                                                info.data_ptr() + 4, stream.cuda_stream), "bitsmoe_shared_basis")

    with torch.cuda.stream(stream):
        for _ in range(max(3, min(args.warmup, 3))):
            step()
    stream.synchronize()
    clk = ClockSampler(local)
    clk.start()
    rank_barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk.mark("t0")
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    e1.synchronize()
    clk.mark("t1")
    torch.cuda.synchronize()
    rank_barrier(world)
    ms_own = e0.elapsed_time(e1)
    ms = max_over_ranks(ms_own, world, dev)
    clocks = clk.stop()
    sweeps, status = int(info[0].item()), int(info[1].item())
    if status != 0:
        raise RuntimeError(f"bitsmoe_shared_basis device status {status}")
    value = world * args.steps * E * n / (ms / 1e3)
    sec = ms_own / args.steps / 1e3
    # the dominant kernel is the Jacobi solver (its share: the launch list under profiles/); its
    # arithmetic per round: 8 flops per element of G (row and column rotations) and 4 per element
    # of V^T, D^2 elements each, (D - 1) rounds a sweep, sweeps + 1 sweeps (the last one checks)
    m = D + (D & 1)
    jac_flops = 12.0 * D * D * (m - 1) * (sweeps + 1 if sweeps < 30 else 30)
    peaks, _ = measured_peaks()
    sm_mhz = clocks.get("sm_mhz") or float(peaks.get("sm_max_mhz", 2070.0))
    sms = torch.cuda.get_device_properties(dev).multi_processor_count
    peak = sms * FP32_FLOPS_PER_SM_CLK * sm_mhz * 1e6 / 1e12
    roofline = {"bound": "alu", "kernel": "k_jacobi (cyclic Jacobi eigensolver of the D x D Gram matrix, fp32)",
                "achieved": jac_flops / sec / 1e12, "peak": peak, "unit": "TFLOP/s",
                "frac": jac_flops / sec / 1e12 / peak,
                "peak_source": f"{sms} SMs x 128 fp32 lanes x 2 flops x {sm_mhz:.0f} MHz (median SM clock under load)",
                "note": "the whole call's time in the denominator; the solver is bound by its rounds (one grid "
                        "barrier and a pass over its rows of G and V^T each), not by arithmetic",
                "traffic": None, "flops_per_launch": jac_flops, "duration_us": sec * 1e6, "sweeps": sweeps}
    # e2e: weights in from pinned host memory, basis + energies + spectral vectors back, every step
    ne = 2
    Wh = W.cpu().pin_memory()
    Ph = torch.empty_like(P, device="cpu").pin_memory()
    phih = torch.empty_like(phi, device="cpu").pin_memory()
    ah = torch.empty_like(alpha, device="cpu").pin_memory()
    t0 = time.perf_counter()
    for _ in range(ne):
        with torch.cuda.stream(stream):
            W.copy_(Wh, non_blocking=True)
            step()
            Ph.copy_(P, non_blocking=True)
            phih.copy_(phi, non_blocking=True)
            ah.copy_(alpha, non_blocking=True)
        stream.synchronize()
    e2e_s = time.perf_counter() - t0
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = dec_oracle_rate(spec, budget_s=20.0)
    if rank == 0:
        line = {
            "metric": DEC_METRIC, "value": value, "unit": "units/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic", "config": dec_config(spec),
            "roofline": roofline, "cpu_baseline": cpu, "clocks": clocks, "gpu_launches": 6 * args.steps,
            "e2e": {"value": world * ne * E * n / e2e_s, "unit": "units/s", "steps": ne,
                    "h2d_bytes_per_step": E * I * D * 4, "d2h_bytes_per_step": (E * n * I + D * n + E * n) * 4},
        }
        print(json.dumps(line), flush=True)


ALLOC_METRIC = "spectral units allocated/s (per-projection bit allocation: costs, Lagrangian cut, greedy fill)"
KAPPA_TABLE = (0.14949200, 0.04067890, 0.01184786)   # kappa_2, kappa_3, kappa_4 (Table kappa_values)


def run_allocate(args, spec, rank, world, local):
    """Bit allocation of one Qwen3-shaped layer: three projections of U = E n units of length I,
    each under the paper's budget B_h = floor(E n b_eq - 16 n^2 / I) at b_eq = mean unit bits;
    alpha_j = j^-1/2, beta log-normal, gamma 1/2.  A step is three bitsmoe_allocate_bits calls."""
    import torch
    import paper_2606_00079_gb300 as bm
    dev = torch.device("cuda", local)
    U, I = args.units or spec.E * spec.n, spec.I
    P, _ = quant_inputs(torch, 3 * U, I, spec.bits_dist, 2000 + rank, dev)
    g = torch.Generator(device=dev)
    g.manual_seed(3000 + rank)
    j = (torch.arange(3 * U, device=dev) % spec.n + 1).to(torch.float32)
    alpha = j.pow(-0.5).contiguous()
    beta = torch.exp(torch.randn(3 * U, generator=g, device=dev, dtype=torch.float32)).contiguous()
    gamma = 0.5
    if U % spec.n == 0:   # the paper's budget for U / n experts (library helper, exact integers)
        budget = bm.bitsmoe_projection_budget(U // spec.n, spec.n, I, spec.mean_bits)
    else:
        from fractions import Fraction
        budget = int((Fraction(U) * Fraction(str(spec.mean_bits)) * I - 16 * spec.n * spec.n) // I)
    bits = torch.empty(3 * U, dtype=torch.uint8, device=dev)
    nb = bm.bitsmoe_allocate_workspace_bytes(U)
    wsb = torch.empty(nb + 256, dtype=torch.uint8, device=dev)
    ws = (wsb.data_ptr() + 255) // 256 * 256
    stream = torch.cuda.Stream(device=dev)

    def call(h, profile=False):
        o = h * U
        return bm.bitsmoe_allocate_bits(P[o].data_ptr(), alpha[o:].data_ptr(), beta[o:].data_ptr(), gamma, U, I,
                                        KAPPA_TABLE, budget, bits[o:].data_ptr(), ws, nb, stream.cuda_stream,
                                        profile=profile)

    def step():
        for h in range(3):
            call(h)

    with torch.cuda.stream(stream):
        for _ in range(max(3, min(args.warmup, 5))):
            step()
    stream.synchronize()
    used = [int(bits[h * U:(h + 1) * U].to(torch.int64).sum().item()) for h in range(3)]
    clk = ClockSampler(local)
    clk.start()
    rank_barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk.mark("t0")
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    e1.synchronize()
    clk.mark("t1")
    torch.cuda.synchronize()
    rank_barrier(world)
    ms_own = e0.elapsed_time(e1)
    ms = max_over_ranks(ms_own, world, dev)
    clocks = clk.stop()
    value = job_throughput(world, args.steps, 3 * U, ms)
    # roofline of the dominant phase (the profiling call times the three phases alone, with CUDA
    # events on the launching stream): algorithmic bytes of each phase
    #   costs_and_hull   k_alloc_cost: the unit rows, alpha, beta                       U (4 I + 8)
    #   cut_and_result   4 radix passes over the increments (key 8 B + reach 1 B, 7 a unit),
    #                    their 64 Ki-bin histograms read and cleared, the cut applied and
    #                    the bit-widths written                                         5 U 63 + U + 4 MB
    #   fill             16 rounds over every unit's next key and bit count             16 U 9
    nprof = 6
    ph = np.zeros(3)
    for i in range(nprof):
        ph += np.array(call(i % 3, profile=True))
    ph /= nprof
    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    names = ["costs_and_hull", "cut_and_result", "fill"]
    kernels = ["k_alloc_cost (distortions, costs and hull of every unit)",
               "radix select: k_alloc_hist + k_alloc_scan (4 passes), k_alloc_final",
               "fill: 16 rounds of k_fill_max + k_fill_take"]
    pbytes = [U * (4.0 * I + 8.0), 5.0 * U * 63 + U + 4 * 2 * 65536 * 8.0, 16.0 * U * 9]
    dom = int(np.argmax(ph))
    gbs = [pbytes[i] / (ph[i] / 1e3) / 1e9 for i in range(3)]
    roofline = {"bound": "hbm", "kernel": kernels[dom], "achieved": gbs[dom], "peak": peak,
                "peak_source": peak_src, "unit": "GB/s", "frac": gbs[dom] / peak, "traffic": None,
                "bytes_per_launch": pbytes[dom], "duration_us": ph[dom] * 1e3,
                "duration_source": "CUDA events around the phase (profiling call)",
                "phase_ms": {names[i]: ph[i] for i in range(3)},
                "phase_frac_of_measured": {names[i]: gbs[i] / peak for i in range(3)},
                "frac_of_8tbs": gbs[dom] / NOMINAL_HBM_GBS}
    # e2e: pinned host units in, bit-widths out, every step
    ne = 3
    Ph = P.cpu().pin_memory()
    bh = torch.empty_like(bits, device="cpu").pin_memory()
    t0 = time.perf_counter()
    for _ in range(ne):
        with torch.cuda.stream(stream):
            P.copy_(Ph, non_blocking=True)
            step()
            bh.copy_(bits, non_blocking=True)
        stream.synchronize()
    e2e_s = time.perf_counter() - t0
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        from oracle import allocator as Aor
        kap = {2: KAPPA_TABLE[0], 3: KAPPA_TABLE[1], 4: KAPPA_TABLE[2]}
        Pn, _ = synth.make_float_units(16384, I, seed=0)
        an = (((np.arange(16384) % spec.n) + 1.0) ** -0.5).astype(np.float32)
        n_done, secs, rep = 0, 0.0, 0
        while secs < 12.0 and rep < 400:   # one chunk of 16384 units, new betas each time, ~12 s of CPU work
            bn = np.random.default_rng([rep, 5]).lognormal(0.0, 1.0, 16384).astype(np.float32)
            t = time.perf_counter()
            Aor.allocate(Aor.costs(Pn, an, bn, gamma, kap), int(budget * 16384 / U))
            secs += time.perf_counter() - t
            n_done += 16384
            rep += 1
        cpu = {"value": n_done / secs, "unit": "units/s", "cores": cpu_cores(), "kind": "oracle",
               "sample": f"{rep} allocations of a 16384-unit chunk of {I} (budget scaled, new betas each), "
                         f"numpy, {secs:.1f} s"}
    if rank == 0:
        line = {
            "metric": ALLOC_METRIC, "value": value, "unit": "units/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32", "data": "synthetic",
            "config": alloc_config(spec, U, I, budget, gamma), "bits_used": used,
            "roofline": roofline, "cpu_baseline": cpu,
            "e2e": {"value": world * ne * 3 * U / e2e_s, "unit": "units/s", "steps": ne,
                    "h2d_bytes_per_step": 3 * U * I * 4, "d2h_bytes_per_step": 3 * U},
            "clocks": clocks, "gpu_launches": args.steps * 3 * 43,
        }
        print(json.dumps(line), flush=True)


def run_layer(args, spec, T, torch, bm, dev, rank, world, local):
    """One MoE layer: K forwards of T tokens from CUDA graphs over rotating packed copies; returns
    rank 0's JSON line (None on the other ranks)."""
    # ---- workload: one generated layer, packed once, uploaded as rotating copies
    layer = synth.make_layer(spec, seed=0)
    blob = bm.bitsmoe_pack_to_host(layer)
    copies = [bm.bitsmoe_load_blob(blob, device=local) for _ in range(args.copies)]
    L0 = copies[0]
    moved = np.array([L0.expert_moved_bytes(e) for e in range(spec.E)], dtype=np.float64)  # E x 3
    NI = args.inputs
    xs, lgs, routes = [], [], []
    for i in range(NI):
        x, lg = synth.make_inputs(spec, T, seed=0, step=i)
        xs.append(torch.from_numpy(x.view(np.int16)).to(dev))
        lgs.append(torch.from_numpy(lg).to(dev))
        routes.append(host_route(lg, spec.top_k))
    ws = bm.Workspace(L0, T, spec.top_k, device=dev)
    y = torch.empty((T, spec.D), dtype=torch.float32, device=dev)
    stream = torch.cuda.Stream(device=dev)

    def step_args(i):
        return xs[i % NI], lgs[i % NI], copies[i % args.copies]

    def fwd(i, st):
        x, lg, L = step_args(i)
        bm.bitsmoe_moe_forward(x.data_ptr(), lg.data_ptr(), T, spec.top_k, L, y.data_ptr(), ws.ptr, ws.nbytes,
                               st.cuda_stream)

    # algorithmic bytes per step (bases, routed experts' factors, x, logits, y)
    base_bytes = 3.0 * spec.D * spec.n * 2 + T * spec.D * 2 + T * spec.E * 4 + T * spec.D * 4

    def step_bytes(i):
        used = np.unique(routes[i % NI])
        return base_bytes + moved[used].sum()

    # ---- warmup (eager) then capture graphs of forwards
    with torch.cuda.stream(stream):
        for i in range(min(args.warmup, 8)):
            fwd(i, stream)
    stream.synchronize()
    G = max(1, min(args.graph, args.steps))

    def capture(n, offset):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            for i in range(n):
                fwd(offset + i, stream)
        return g

    nfull, rem = divmod(args.steps, G)
    g_main = capture(G, 0)
    g_rem = capture(rem, nfull * G) if rem else None
    w0, w1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    nwarm = max(1, args.warmup // G)
    w0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(nwarm):
            g_main.replay()
    w1.record(stream)
    stream.synchronize()
    # a timed region too short for the clock record (20 ms samples) gets the same load, untimed,
    # for about 0.2 s before and after it, and the record covers both
    per_replay_s = w0.elapsed_time(w1) / 1e3 / nwarm
    pad = int(0.2 / max(per_replay_s, 1e-6)) if per_replay_s * max(nfull, 1) < 0.4 else 0

    clk = ClockSampler(local)
    clk.start()
    rank_barrier(world)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clk.mark("l0")
    with torch.cuda.stream(stream):
        for _ in range(pad):
            g_main.replay()
    clk.mark("t0")
    e0.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(nfull):
            g_main.replay()
        if g_rem is not None:
            g_rem.replay()
    e1.record(stream)
    with torch.cuda.stream(stream):
        for _ in range(pad):
            g_main.replay()
    e1.synchronize()
    clk.mark("t1")
    torch.cuda.synchronize()
    clk.mark("l1")
    rank_barrier(world)
    ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    clocks = clk.stop()
    total_bytes = sum(step_bytes(i) for i in range(args.steps))
    value = job_throughput(world, args.steps, T, ms)
    fwd_gbs = total_bytes / (ms / 1e3) / 1e9

    # ---- roofline of the dominant kernel
    launches = bm.bitsmoe_forward_launches(L0, T, spec.top_k)
    peaks, peak_src = measured_peaks()
    peak = float(peaks.get("hbm_gbs", FALLBACK_HBM_GBS))
    phase_ms = np.zeros(5)
    nprof = 64
    for i in range(nprof):
        x, lg, L = step_args(i)
        phase_ms += bm.bitsmoe_profile_forward(x.data_ptr(), lg.data_ptr(), T, spec.top_k, L, y.data_ptr(),
                                               ws.ptr, ws.nbytes, stream.cuda_stream)
    phase_ms /= nprof
    if launches == 1:
        # one fused kernel does the whole step: its average duration is at most the timed region per
        # step (which also holds the gap between launches), so this is a lower bound
        achieved = (total_bytes / args.steps) / (ms / args.steps / 1e3) / 1e9
        traffic = measured_traffic("ncu_full_k_fused_qw3_T1.txt", ("fused.cu", "fused_common.cuh", "device.cuh", "format.h"))
        roofline = {"bound": "hbm", "kernel": "k_fused (whole single-token forward)", "achieved": achieved,
                    "peak": peak, "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak,
                    "traffic": traffic,
                    "bytes_per_launch": total_bytes / args.steps,
                    "duration_us": ms / args.steps * 1e3,
                    "duration_source": "CUDA events over the timed region / steps",
                    "isolated_us": float(phase_ms[0]) * 1e3,
                    "frac_of_8tbs": achieved / NOMINAL_HBM_GBS}
    else:
        mean_moved = np.mean([moved[np.unique(routes[i % NI])].sum(axis=0) for i in range(nprof)], axis=0)
        P = T * spec.top_k
        phase_bytes = [
            T * spec.E * 4,
            2.0 * spec.D * spec.n * 2 + T * spec.D * 2 + 2.0 * T * spec.n * 4,
            mean_moved[0] + mean_moved[1] + 2.0 * T * spec.n * 4 + 2.0 * P * spec.I * 4,
            mean_moved[2] + 2.0 * P * spec.I * 4 + T * spec.n * 4,
            1.0 * spec.D * spec.n * 2 + T * spec.n * 4 + T * spec.D * 4,
        ]
        dom = int(np.argmax(phase_ms))
        achieved = phase_bytes[dom] / (phase_ms[dom] / 1e3) / 1e9
        roofline = {"bound": "hbm", "kernel": PHASES[dom], "achieved": achieved, "peak": peak,
                    "peak_source": peak_src, "unit": "GB/s", "frac": achieved / peak, "traffic": None,
                    "phase_ms": {PHASES[i]: float(phase_ms[i]) for i in range(5)},
                    "phase_bytes": {PHASES[i]: float(phase_bytes[i]) for i in range(5)},
                    "forward_gbs": fwd_gbs, "forward_frac_of_measured": fwd_gbs / peak,
                    "forward_frac_of_8tbs": fwd_gbs / NOMINAL_HBM_GBS}

    # ---- e2e through the asynchronous host-buffer entry point: every step's inputs come from
    # its own pinned host buffers and its output lands in its own pinned host buffer (read in
    # place by the single-token kernel, copied otherwise); the steps are enqueued back to back
    # and the stream is synchronised once, as a serving loop keeps them in flight; the
    # synchronous entry point (one synchronisation a step) is timed beside it
    NB = 64
    xh = [torch.from_numpy(synth.make_inputs(spec, T, seed=0, step=i % 8)[0].view(np.int16).copy()).pin_memory()
          for i in range(NB)]
    lh = [torch.from_numpy(synth.make_inputs(spec, T, seed=0, step=i % 8)[1].copy()).pin_memory() for i in range(NB)]
    yh = [torch.empty((T, spec.D), dtype=torch.float32).pin_memory() for _ in range(NB)]
    ne2e = max(10, min(args.steps, 2000))

    def host_call(i, fn):
        L = copies[i % args.copies]
        rc = fn(xh[i % NB].data_ptr(), lh[i % NB].data_ptr(), T, spec.top_k, L.handle, yh[i % NB].data_ptr(),
                ws.ptr, ws.nbytes, stream.cuda_stream)
        if rc != 0:
            raise bm.BitsMoEError(rc, "host-buffer forward")

    fa, fs = bm._lib().bitsmoe_moe_forward_host_async, bm._lib().bitsmoe_moe_forward_host
    for i in range(5):
        host_call(i, fs)
    t0 = time.perf_counter()
    for i in range(ne2e):
        host_call(i, fa)
        if i % NB == NB - 1:   # an output buffer is written again only after its step was read
            stream.synchronize()
    stream.synchronize()
    e2e_s = time.perf_counter() - t0
    ns = max(10, ne2e // 4)
    t0 = time.perf_counter()
    for i in range(ns):
        host_call(i, fs)
    sync_s = time.perf_counter() - t0
    e2e = {"value": world * ne2e * T / e2e_s, "unit": "tokens/s", "steps": ne2e,
           "h2d_bytes_per_step": T * spec.D * 2 + T * spec.E * 4, "d2h_bytes_per_step": T * spec.D * 4,
           "api": "bitsmoe_moe_forward_host_async, steps in flight, one synchronisation per 64 steps",
           "synchronous_value": world * ns * T / sync_s}

    # ---- CPU baseline (rank 0, N = 1 only)
    cpu = cpu1 = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        v, steps, secs = oracle_tokens_per_s(spec, layer, T, budget_s=12.0)
        cpu = {"value": v, "unit": "tokens/s", "cores": cpu_cores(), "kind": "oracle",
               "sample": f"{steps} decode steps of {T} token(s), fp64 numpy factored forward ({secs:.1f} s)"}
        cpu1 = oracle_one_core(spec, T)

    line = None
    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f32",
            "arith": "bf16 basis x f32 (f32 accumulate); u8 codes x i16 activations (dp2a, i32 accumulate)",
            "data": "synthetic", "config": config_of(spec, T, args),
            "hbm_gbs": fwd_gbs, "hbm_frac_of_8tbs": fwd_gbs / NOMINAL_HBM_GBS, "hbm_frac_of_measured": fwd_gbs / peak,
            "bytes_per_step": total_bytes / args.steps,
            "roofline": roofline, "cpu_baseline": cpu, "cpu_baseline_1core": cpu1, "e2e": e2e, "clocks": clocks,
            "gpu_launches": args.steps * launches,
        }
    return line


ALL_CONFIGS = [("qw3", 1), ("qw3_skew", 1), ("qw3_skew", 8), ("qw3_skew", 32), ("qw3_skew", 128),
               ("mixtral", 1), ("mixtral", 16), ("qw3_stack", 1), ("qw3_stack", 32)]


def run_all(args, torch, bm, dev, rank, world, local):
    """Every workload configuration in turn, one JSON line each; the step count adapts so that
    each timed region is a fraction of a second to a few seconds."""
    import copy
    import gc
    for wl, T in ALL_CONFIGS:
        spec = synth.WORKLOADS[wl]
        a = copy.copy(args)
        a.workload, a.tokens = wl, T
        if spec.layers > 1:
            a.steps = args.steps or (200 if T == 1 else 20)
            line = run_stack(a, spec, T, torch, bm, dev, rank, world, local)
        else:
            a.steps = args.steps or (4000 if T <= 4 else 1000 if T <= 32 else 400)
            line = run_layer(a, spec, T, torch, bm, dev, rank, world, local)
        if rank == 0:
            print(json.dumps(line), flush=True)
        gc.collect()
        torch.cuda.empty_cache()


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=None,
                    help="default 20000 (one layer), 400 (layer stack), 20 (--task quantize)")
    ap.add_argument("--warmup", type=int, default=200)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default="qw3")
    ap.add_argument("--tokens", type=int, default=None)
    ap.add_argument("--copies", type=int, default=8)
    ap.add_argument("--inputs", type=int, default=64)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--graph", type=int, default=256, help="forwards per captured CUDA graph")
    ap.add_argument("--task", default="forward",
                    choices=["forward", "quantize", "allocate", "importance", "decompose"],
                    help="forward: the MoE-layer forward (default); quantize: the per-unit quantiser; "
                         "allocate: the per-projection bit allocation; importance: the importance beta of "
                         "every unit from calibration tokens; decompose: the shared-basis decomposition of "
                         "one projection")
    ap.add_argument("--calib-tokens", type=int, default=4096,
                    help="calibration tokens per step of --task importance")
    ap.add_argument("--grid", type=int, default=256, help="scale candidates of the quantiser (--task quantize)")
    ap.add_argument("--all", action="store_true",
                    help="one JSON line per workload configuration and token count (the single layers at "
                         "T = 1; qw3_skew at 1, 8, 32, 128; mixtral at 1, 16; the 48-layer stack at 1, 32)")
    ap.add_argument("--units", type=int, default=None,
                    help="units per quantiser step (default the whole layer, 3 E n) or per allocated "
                         "projection (default E n)")
    args = ap.parse_args()
    spec = synth.WORKLOADS[args.workload]
    T = args.tokens or spec.tokens[0]
    if args.steps is None and not args.all:
        args.steps = {"forward": 20000 if spec.layers == 1 else 400, "decompose": 3}.get(args.task, 20)
    if args.impl == "reference":
        if args.task == "forward":
            run_reference(args, spec, T)
        else:
            run_reference_task(args, spec)
        return

    import torch
    import paper_2606_00079_gb300 as bm
    from paper_2606_00079_gb300 import build as bmbuild
    bmbuild.build()
    rank, world, local = dist_env()
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl" if torch.cuda.is_available() else "gloo")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    if args.task != "forward":
        {"quantize": run_quantize, "allocate": run_allocate, "importance": run_importance,
         "decompose": run_decompose}[args.task](args, spec, rank, world, local)
        if world > 1:
            torch.distributed.barrier()
            torch.distributed.destroy_process_group()
        return
    if args.all:
        run_all(args, torch, bm, dev, rank, world, local)
    elif spec.layers > 1:
        line = run_stack(args, spec, T, torch, bm, dev, rank, world, local)
        if rank == 0:
            print(json.dumps(line), flush=True)
    else:
        line = run_layer(args, spec, T, torch, bm, dev, rank, world, local)
        if rank == 0:
            print(json.dumps(line), flush=True)
    if world > 1:
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()


if __name__ == "__main__":
    main()
