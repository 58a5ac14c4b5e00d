#!/usr/bin/env python3
"""Throughput of the layer-dropout decoder stack, forward + backward, on GB300.

One step = ld_forward + ld_backward of the whole stack (every layer: mask
draw, kept-row RMSNorm, QKV + RoPE, causal GQA attention, O projection with
the 1/(1-p) residual update, RMSNorm, SwiGLU, down projection, and the
mirrored backward) over one batch of synthetic activations, through the C ABI.

Default workload: the Llama-3-8B-shaped stack (32 layers, d 4096, 32 query /
8 key-value heads of 128, SwiGLU 14336, 4 x 4096 tokens, ILD p_max 0.4,
per-sequence masks).  Reported:
  value          effective tokens/s = B*S / step time (inputs resident in HBM)
  e2e            the same with the step's inputs copied host->device from
                 pinned memory and dX copied back, inside the timed region
  pct_bf16_peak  executed FLOPs / time / measured bf16 peak (sustained)
  skip_speedup   t(p=0) / t(p), next to the ideal 1/(1 - p_bar)
  roofline       the tcgen05 GEMM class (the dominant kernel), timed with CUDA
                 events around each of its launches over a second pass of the
                 same steps (the library then keeps the backward's weight-
                 gradient products on one stream, so no launch overlaps
                 another; in the headline pass they run on a side stream)
  cpu_baseline   the CPU oracle on a bounded sample of the same workload

--impl reference times the CPU oracle alone (this workload has no runnable
reference implementation; the oracle is the reference arm).
Multi-GPU (torchrun): replicas only, one batch per rank, no collective on
the data path (weak scaling).
"""

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

METRIC = "effective tokens/s (fwd+bwd) under layer dropout; % bf16 peak; skip-speedup vs ideal"

# DRAM read + write of the tcgen05 GEMM per kept row of a launch, from one
# ncu capture (dram__bytes_read.sum + dram__bytes_write.sum) of the 24 GEMM
# launches of a 2-layer stack with the Llama-3-8B shapes and 12288 kept rows
# per launch; command and per-launch table in
# profiles/gemm_tc_llama8b_traffic.md.  Scaled by the kept rows per launch.
GEMM_DRAM_BYTES_PER_ROW = 166811.0
PEAKS = os.path.join(ROOT, "MEASURED_PEAKS.json")


def load_peaks():
    try:
        with open(PEAKS) as f:
            p = json.load(f)
        return dict(bf16=p["bf16_tflops"], bf16_sustained=p["bf16_tflops_sustained"], hbm=p["hbm_gbs"],
                    source="measured")
    except Exception:
        return dict(bf16=1900.0, bf16_sustained=1700.0, hbm=6800.0, source="fallback")


def flops_per_token(cfg, split=False):
    """Forward FLOPs per token per layer (2 x MACs; causal attention counted
    as S/2 keys per query) and the part of it in the projections; with
    split=True the projections of the attention block and of the FFN block
    separately: (total, attention-block projections, FFN)."""
    d, H, Hkv, Dh, F, S = cfg["d"], cfg["H"], cfg["Hkv"], cfg["Dh"], cfg["F"], cfg["S"]
    ffn = 4 * d * F if cfg.get("act") == "relu2" else 6 * d * F  # up (+ gate) and down
    attn_proj = 2 * d * (H + 2 * Hkv) * Dh + 2 * d * H * Dh
    attn = 2 * H * Dh * S
    if split:
        return attn_proj + ffn + attn, attn_proj, ffn
    return attn_proj + ffn + attn, attn_proj + ffn


def replica_command(n, argv, port):
    """The command that runs this script as n replica processes, one per
    GPU of this node (torchrun; rendezvous on 127.0.0.1): what `--gpus N`
    does when no launcher has set WORLD_SIZE."""
    return [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={n}",
            "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.abspath(__file__)] + list(argv)


def free_port():
    import socket
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def tensor_peak_at_clock(sm_mhz, sms=152):
    """Dense bf16 tensor rate of the whole GPU at a given SM clock: 8192
    FLOP per clock per SM (one M = 128, N = 256, K = 16 tcgen05 MMA every 128
    clocks, measured on this GPU), in TFLOP/s."""
    return sms * 8192.0 * sm_mhz * 1e6 / 1e12


def result_line(world, B, S, ms, **extra):
    """The JSON line's job-level fields: whole-job throughput over every
    replica (each rank processes its own batch of B x S tokens) from the
    slowest rank's step time `ms`."""
    return dict({"value": world * B * S / (ms / 1e3), "unit": "tokens/s", "n_gpus": world, "ms_per_step": ms,
                 "scaling": "weak"}, **extra)


def config_of(args, cfg, sched, first_step, world):
    """The `config` object of the JSON line (the same for both arms)."""
    return {"workload": args.config, **{k: cfg[k] for k in ("L", "d", "H", "Hkv", "Dh", "F", "B", "S")},
            "schedule": sched, "granularity": args.granularity, "sublayer": args.sublayer,
            "first_step": first_step, "parallelism": f"replicas x{world}",
            "l2": "inputs and weights larger than L2 (no flush)"}


def max_over_ranks(ms, world, device="cuda"):
    """Step time of the whole job: the slowest rank's."""
    if world <= 1:
        return ms
    import torch
    import torch.distributed as dist
    t = torch.tensor([ms], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


class Clocks:
    """nvidia-smi clock/throttle sampling while the timed region runs."""

    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,clocks_event_reasons.hw_slowdown,"
         "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
         "clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
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
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                rows.append((float(f[1]), float(f[2]), f[5], f[6], f[7], f[8]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[2 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(r[0] for r in rows), "sm_max_mhz": max(r[1] for r in rows),
                "reasons": reasons, "samples": len(rows)}


SLOWDOWNS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown")


def clocks_rejected(clk, stuck_frac=0.75):
    """True when a clock record disqualifies its timing: a hardware or
    thermal slowdown was active, or the median SM clock sat below
    `stuck_frac` of the maximum with no reason given (a leftover clock
    lock).  sw_power_cap alone is normal under a dense load and is kept."""
    if not clk:
        return False
    if any(r in clk["reasons"] for r in SLOWDOWNS):
        return True
    return not clk["reasons"] and clk["sm_mhz"] < stuck_frac * clk["sm_max_mhz"]


def cpu_baseline(cfg, host_w0, x_seq, dy_seq, rows, kept_units_per_step, s_l0):
    """The oracle (float64 numpy) on a bounded sample: layer 0, sequence 0,
    its first `rows` rows, forward + backward.  Extrapolated to a step by the
    kept tokens of the step (every kept (layer, sequence) processes S rows)."""
    import numpy as np
    from oracle import stack as OK

    W = {n: v.double().numpy() for n, v in host_w0.items()}
    x = x_seq[:rows].double().numpy()
    dy = dy_seq[:rows].double().numpy()
    rope = OK._rope_cs(cfg, rows)
    t0 = time.perf_counter()
    out, cache = OK.layer_forward(x, W, cfg, s_l0, rope)
    G = {n: np.zeros(OK.shape_of(cfg, n)) for n in OK.WEIGHT_NAMES}
    OK.layer_backward(dy, W, cfg, s_l0, cache, G, rope)
    dt = time.perf_counter() - t0
    per_token = dt / rows
    step_time = per_token * kept_units_per_step * cfg["S"]
    note = ("the whole sequence, so the per-sequence cost is measured, not extrapolated" if rows >= cfg["S"] else
            "attention cost of later rows under-represented, so the CPU figure is optimistic")
    return {"value": cfg["B"] * cfg["S"] / step_time, "unit": "tokens/s", "cores": os.cpu_count(),
            "kind": "oracle", "sample": f"layer 0, sequence 0, rows 0..{rows - 1} of {cfg['S']}, fwd+bwd, float64 "
            f"numpy ({dt:.1f} s); scaled to a step by the step's kept (layer, sequence) pairs ({note})",
            "sample_seconds": dt}


def run_reference(args):
    import torch
    from paper_2609_05275_gb300 import synth
    from oracle import masks as OM, schedule as OS

    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    cfg, sched = synth.CONFIGS[args.config], synth.SCHEDULES[args.config]
    rows = min(args.cpu_rows or cfg["S"], cfg["S"])  # a whole sequence unless asked otherwise
    w0 = synth.layer_weights(cfg, 0, seed=0)
    x = synth.activations(cfg, seed=0, B=1)[0]
    dy = synth.upstream_grad(cfg, B=1)[0]
    osched = dict(dist=sched["dist"], p_max=sched.get("p_max", 0.0), p_explicit=sched.get("p_explicit"),
                  time=sched.get("time", "const"), T=sched.get("T"), ramp=sched.get("ramp"))
    # the oracle's cost of one kept (layer, sequence) is measured once, on
    # layer 0 and sequence 0 (one forward + backward of `rows` rows); each
    # step's time is that cost times the step's kept (layer, sequence) pairs
    # from the step's own masks, so the run stays within minutes
    step0 = args.step0 if args.step0 is not None else synth.STEPS[args.config][-1]
    rates0 = OS.layer_rates(osched, cfg["L"], step0)
    r = cpu_baseline(cfg, w0, x, dy, rows, 1, OS.residual_scale(rates0[0]))
    per_pair = cfg["B"] * cfg["S"] / r["value"]  # seconds per kept (layer, sequence)
    times = []
    for k in range(args.warmup, args.warmup + args.steps):
        t = step0 + k
        rates = OS.layer_rates(osched, cfg["L"], t)
        mk = OM.draw_masks(sched["seed"], t, [OS.drop_threshold(p) for p in rates], cfg["B"])
        times.append(per_pair * int(mk.sum()))
    step = sum(times) / len(times)
    value = cfg["B"] * cfg["S"] / step
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": step * 1e3, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_of(args, cfg, sched, step0 + args.warmup, args.gpus),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": os.cpu_count(), "kind": "oracle",
                             "sample": r["sample"].split(";")[0] + "; measured once, each step scaled by its own "
                                       "kept (layer, sequence) pairs", "sample_seconds": r["sample_seconds"]},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def run_sweep(args):
    """Throughput against the ideal 1/(1 - p_bar) over the sweep grid: for
    every (p_max, distribution, granularity) cell, one timed step per seed at
    step 0 (after one warm-up step), CUDA events around each step."""
    import torch

    import paper_2609_05275_gb300 as P
    from paper_2609_05275_gb300 import synth

    sw = synth.SWEEP
    cfg = dict(synth.CONFIGS[sw["base"]])
    L, B, S = cfg["L"], cfg["B"], cfg["S"]
    layers = synth.stack_weights(cfg, seed=0, device="cuda")
    wtab = P.weight_table(layers)
    grads = [{n: torch.empty(v.shape, device="cuda", dtype=torch.float32) for n, v in W.items()} for W in layers]
    gtab = P.grad_table(grads)
    x0 = synth.activations(cfg, seed=0, device="cuda")
    dy0 = synth.upstream_grad(cfg, device="cuda")
    x, dx = torch.empty_like(x0), torch.empty_like(dy0)
    f_tok, _ = flops_per_token(cfg)
    stacks = {g: P.LayerDropStack(cfg, dict(dist="uniform", p_max=0.0, seed=1), granularity=g)
              for g in sw["granularity"]}
    seeds = sw["seeds"][: args.steps] if args.steps < len(sw["seeds"]) else sw["seeds"]

    def step(st, t):
        x.copy_(x0)
        dx.copy_(dy0)
        st.forward(t, wtab, x)
        st.backward(wtab, dx, gtab)

    def time_cell(st, sched):
        ms, kept = [], []
        for seed in seeds:
            st.schedule = P.make_schedule(dict(sched, seed=seed))
            P.ld_set_schedule(st.h, st.schedule)
            step(st, 0)
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record()
            step(st, 0)
            e1.record()
            torch.cuda.synchronize()
            ms.append(e0.elapsed_time(e1))
            kept.append(int(st.masks()[2].sum()))  # kept (layer, sequence) pairs, or kept tokens per token
        return ms, kept

    dense_ms, _ = time_cell(stacks["per_sequence"], dict(dist="uniform", p_max=0.0, time="const"))
    t_dense = statistics.median(dense_ms)
    cells = []
    for gran in sw["granularity"]:
        for dist in sw["dist"]:
            for p_max in sw["p_max"]:
                sched = dict(dist=dist, p_max=p_max, time="const")
                ms, kept = time_cell(stacks[gran], sched)
                rows_per_unit = 1 if gran == "per_token" else S
                p_real = 1.0 - sum(kept) * rows_per_unit / (len(kept) * L * B * S)
                t = sum(ms) / len(ms)
                speed = t_dense / t
                ideal = 1.0 / (1.0 - p_real)
                cell = {"granularity": gran, "dist": dist, "p_max": p_max, "seeds": len(seeds),
                        "ms_per_step": t, "tokens_per_s": B * S / (t / 1e3),
                        # per token the attention term of f_tok (whole-length sequences) overstates the
                        # work of the shortened sequences slightly
                        "executed_tflops": 3.0 * f_tok * rows_per_unit * sum(kept) / len(kept) / (t / 1e3) / 1e12,
                        "p_bar_realized": p_real, "speedup": speed, "ideal_speedup": ideal,
                        "frac_of_ideal": speed / ideal}
                cells.append(cell)
                print(json.dumps({"sweep_cell": cell}), flush=True)
    for st in stacks.values():
        st.close()
    print(json.dumps({"sweep": sw["base"], "dense_ms_per_step": t_dense,
                      "min_frac_of_ideal": min(c["frac_of_ideal"] for c in cells if c["p_max"] > 0),
                      "mean_frac_of_ideal": statistics.mean(c["frac_of_ideal"] for c in cells if c["p_max"] > 0)}),
          flush=True)
    return 0


def run_eval(args):
    """Depth-elastic inference forward (ld_forward_eval) on the workload's
    weights: full depth, early exit at L/2 and alternate-layer skipping, at
    the workload's B x S and at batch-1 shapes with S = 128 and 512.  Each
    setting is timed eagerly and as a CUDA graph replay (CUDA events, median
    of --steps after --warmup); one JSON line per (shape, setting)."""
    import torch

    import paper_2609_05275_gb300 as P
    from paper_2609_05275_gb300 import synth

    base = dict(synth.CONFIGS[args.config])
    if args.layers:
        base["L"] = args.layers
    L = base["L"]
    layers = synth.stack_weights(base, seed=0, device="cuda")
    wtab = P.weight_table(layers)
    settings = [("full depth", [1] * L), ("early exit at L/2", [1] * (L // 2) + [0] * (L - L // 2)),
                ("alternate layers", [1 - (l % 2) for l in range(L)])]
    shapes = [(base["B"], base["S"]), (1, 512), (1, 128)]
    for B, S in shapes:
        cfg = dict(base, B=B, S=S)
        f_tok, _ = flops_per_token(cfg)
        st = P.LayerDropStack(cfg, dict(dist="uniform", p_max=0.0, seed=1))
        st.workspace = torch.empty(P.ld_eval_workspace_size(st.h), dtype=torch.uint8, device="cuda")
        x0 = synth.activations(cfg, seed=0, device="cuda")
        x = torch.empty_like(x0)
        full_ms = None
        for name, ex in settings:
            def step():
                x.copy_(x0)
                st.forward_eval(ex, wtab, x)

            res = {}
            for mode in ("eager", "graph"):
                run = step
                if mode == "graph":
                    stream = torch.cuda.Stream()
                    stream.wait_stream(torch.cuda.current_stream())
                    g = torch.cuda.CUDAGraph()
                    with torch.cuda.stream(stream):
                        step()  # first call outside the capture (one-time set-up)
                        with torch.cuda.graph(g, stream=stream):
                            step()
                    torch.cuda.current_stream().wait_stream(stream)
                    run = g.replay
                for _ in range(max(args.warmup, 3)):
                    run()
                torch.cuda.synchronize()
                times = []
                for _ in range(args.steps):
                    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
                    e0.record()
                    run()
                    e1.record()
                    e1.synchronize()
                    times.append(e0.elapsed_time(e1))
                res[mode] = statistics.median(times)
            st.sync()
            ms = min(res.values())
            if full_ms is None:
                full_ms = ms
            n_exec = sum(ex)
            print(json.dumps({"eval": {
                "workload": args.config, "B": B, "S": S, "setting": name, "layers_executed": n_exec, "L": L,
                "ms_eager": res["eager"], "ms_graph": res["graph"], "tokens_per_s": B * S / (ms / 1e3),
                "executed_tflops": f_tok * B * S * n_exec / (ms / 1e3) / 1e12,
                "speedup_vs_full_depth": full_ms / ms, "ideal_speedup": L / max(n_exec, 1),
                "r_eval": 1.0, "dtype": "bf16", "data": "synthetic"}}), flush=True)
        st.close()
    return 0


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--config", default="llama8b")
    ap.add_argument("--step0", type=int, default=None, help="first step index (default: the workload's)")
    ap.add_argument("--no-dense", action="store_true", help="skip the p=0 run (no skip_speedup)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-rows", type=int, default=0,
                    help="rows of the CPU oracle sample (default: a whole sequence for the cpu_baseline leg, "
                         "1024 per step for --impl reference)")
    ap.add_argument("--layers", type=int, default=None, help="override L (profiling captures only)")
    ap.add_argument("--granularity", default="per_sequence", choices=["per_sequence", "per_batch", "per_token"],
                    help="mask granularity of the timed steps (the headline is per sequence)")
    ap.add_argument("--sublayer", action="store_true",
                    help="independent attention and FFN masks (sub-layer granularity) in the timed steps")
    ap.add_argument("--sweep", action="store_true",
                    help="drop-rate / distribution / granularity / seed sweep on the 1.3B shape (one JSON line "
                         "per cell, then a summary line)")
    ap.add_argument("--eval", action="store_true",
                    help="depth-elastic inference forward (full depth, early exit, layer skipping) at the "
                         "workload shape and batch-1 shapes; one JSON line per setting")
    args = ap.parse_args()
    if args.gpus > 1 and "WORLD_SIZE" not in os.environ:
        # no outer launcher: start the N replicas here (each rank reads its
        # RANK / LOCAL_RANK / WORLD_SIZE from the environment torchrun sets)
        return subprocess.call(replica_command(args.gpus, sys.argv[1:], free_port()))
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    if args.eval:
        return run_eval(args)

    import torch
    import torch.distributed as dist

    import paper_2609_05275_gb300 as P
    from paper_2609_05275_gb300 import synth

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    if world > 1:
        dist.init_process_group("nccl")

    def barrier():
        if world > 1:
            dist.barrier()

    cfg, sched = dict(synth.CONFIGS[args.config]), dict(synth.SCHEDULES[args.config])
    if args.layers:
        cfg["L"] = args.layers
    L, B, S, d = cfg["L"], cfg["B"], cfg["S"], cfg["d"]
    step0 = args.step0 if args.step0 is not None else synth.STEPS[args.config][-1]
    peaks = load_peaks()

    tok = args.granularity == "per_token"
    sub = args.sublayer
    st = P.LayerDropStack(cfg, sched, granularity=args.granularity, sublayer=sub)
    layers = synth.stack_weights(cfg, seed=0, device="cuda")
    wtab = P.weight_table(layers)
    grads = [{n: torch.empty(v.shape, device="cuda", dtype=torch.float32) for n, v in W.items()} for W in layers]
    gtab = P.grad_table(grads)
    x0 = synth.activations(cfg, seed=rank, device="cuda")
    dy0 = synth.upstream_grad(cfg, seed=2 + 1000 * rank, device="cuda")
    x = torch.empty_like(x0)
    dx = torch.empty_like(dy0)
    stream = torch.cuda.current_stream()

    def step(t):
        x.copy_(x0)
        dx.copy_(dy0)
        st.forward(t, wtab, x)
        st.backward(wtab, dx, gtab)

    def timed(nsteps, first, fn, tail=None):
        barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for k in range(nsteps):
            fn(first + k)
        if tail is not None:
            tail()  # work of the last step on other streams joins before the end event
        e1.record(stream)
        torch.cuda.synchronize()
        barrier()
        return max_over_ranks(e0.elapsed_time(e1) / nsteps, world)

    # ---- main timed region (p as scheduled)
    for k in range(args.warmup):
        step(step0 + k)
    st.sync()
    def measured():
        clocks = Clocks(local)
        clocks.start()
        t = timed(args.steps, step0 + args.warmup, step)
        return t, clocks.stop()

    ms, clk = measured()
    # a run whose clocks show a slowdown (or a clock lock) is measured once
    # more, on every rank, and the second run is the one reported
    if max_over_ranks(1.0 if clocks_rejected(clk) else 0.0, world) > 0.0:
        first = clk
        ms, clk = measured()
        if clk is not None:
            clk["remeasured_after"] = first
    st.sync()
    # ---- device time by kernel class: the same steps again with the
    # library's per-launch events on, which keep the backward's
    # weight-gradient products on the one stream (no overlap), so each
    # launch is timed alone
    P.ld_set_timing(st.h, 1)
    clk_serial = Clocks(local)
    clk_serial.start()
    ms_serial = timed(args.steps, step0 + args.warmup, step)
    clk_serial = clk_serial.stop()
    gemm_ms, gemm_launches = P.ld_get_timing(st.h, P.LD_KCLASS_GEMM)
    attn_ms, attn_launches = P.ld_get_timing(st.h, P.LD_KCLASS_ATTN)
    row_ms, row_launches = P.ld_get_timing(st.h, P.LD_KCLASS_ROWWISE)
    P.ld_set_timing(st.h, 0)
    st.sync()

    # kept counts of the timed steps (masks redrawn through the library):
    # kept (layer, sequence) pairs, or per token the kept tokens (and the
    # kept length of every (layer, sequence) for the attention FLOPs)
    # (with sub-layer masks the attention and FFN blocks keep their own units)
    kept_a, kept_f, attn_len2 = 0, 0, 0.0
    for k in range(args.steps):
        mk, _, cnt = st.draw_masks(step0 + args.warmup + k)
        ka = int(cnt[0].sum()) if sub else int(cnt.sum())
        kept_a += ka
        kept_f += int(cnt[1].sum()) if sub else ka
        if tok:
            mka = mk[0] if sub else mk
            attn_len2 += float((mka.reshape(-1, B, S).sum(axis=2).astype("float64") ** 2).sum())
    f_tok, f_aproj, f_ffn = flops_per_token(cfg, split=True)
    f_attn = f_tok - f_aproj - f_ffn  # attention scores and weighted sum, per token at full length
    kept_units = 0.5 * (kept_a + kept_f)  # per branch on average (equal without sub-layer masks)
    rows_per_unit = 1 if tok else S
    proj_flops = f_aproj * kept_a + f_ffn * kept_f  # per kept unit row
    if tok:  # projections per kept token; attention 2 H Dh len^2 per kept sequence of length len (forward)
        exec_flops = 3.0 * (proj_flops + 2.0 * cfg["H"] * cfg["Dh"] * attn_len2) / args.steps
    else:
        exec_flops = 3.0 * S * (proj_flops + f_attn * kept_a) / args.steps  # per step, this rank
    gemm_flops = 3.0 * rows_per_unit * proj_flops / args.steps
    p_real = 1.0 - kept_units * rows_per_unit / (args.steps * L * B * S)
    _, thr, _ = st.rates(step0 + args.warmup)
    p_exp = sum(t / 2 ** 32 for t in thr) / L
    tflops = exec_flops / (ms / 1e3) / 1e12

    # ---- dense reference point (p = 0 everywhere, same shapes)
    dense_ms = None
    if not args.no_dense:
        st.schedule = P.make_schedule(dict(dist="uniform", p_max=0.0, time="const", seed=sched["seed"]))
        P.ld_set_schedule(st.h, st.schedule)
        step(0)
        dense_ms = timed(args.steps, 0, step)
        P.ld_set_schedule(st.h, P.make_schedule(sched))

    # ---- end to end: host inputs in pinned memory, dX read back every step.
    # X is copied in on the compute stream (the forward starts from it); dY
    # on a copy stream while the forward runs; dX is read back on the copy
    # stream while the next step's forward runs, so dX alternates between two
    # device buffers.  Every step's copies are inside the timed region (the
    # last read-back joins the compute stream before the end event).
    e2e = None
    if not args.no_e2e:
        xh = x0.cpu().pin_memory()
        dyh = dy0.cpu().pin_memory()
        dxh = torch.empty(dx.shape, dtype=dx.dtype).pin_memory()
        copy = torch.cuda.Stream()
        dxs = [dx, torch.empty_like(dx)]

        def step_e2e(t):
            d = dxs[t % 2]
            x.copy_(xh, non_blocking=True)
            copy.wait_stream(stream)  # d's read-back two steps ago was on this stream too
            with torch.cuda.stream(copy):
                d.copy_(dyh, non_blocking=True)
            st.forward(t, wtab, x)
            stream.wait_stream(copy)
            st.backward(wtab, d, gtab)
            copy.wait_stream(stream)
            with torch.cuda.stream(copy):
                dxh.copy_(d, non_blocking=True)

        step_e2e(step0)
        e2e_ms = timed(args.steps, step0 + args.warmup, step_e2e, tail=lambda: stream.wait_stream(copy))
        nb = x.numel() * x.element_size()
        e2e = {"value": world * B * S / (e2e_ms / 1e3), "unit": "tokens/s", "h2d_bytes_per_step": 2 * nb,
               "d2h_bytes_per_step": nb, "ms_per_step": e2e_ms}
    st.sync()

    # ---- CPU oracle on a bounded sample (rank 0, one GPU only)
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu:
        w0 = {n: v.cpu() for n, v in layers[0].items()}
        _, _, sc = st.rates(step0 + args.warmup)
        cpu = cpu_baseline(cfg, w0, x0[0].cpu(), dy0[0].cpu(), min(args.cpu_rows or S, S),
                           kept_units * rows_per_unit / S / args.steps, sc[0])

    gemm_achieved = gemm_flops * args.steps / (gemm_ms / 1e3) / 1e12 if gemm_ms > 0 else None
    # 12 GEMM launches per executed layer (4 forward, 8 backward)
    traffic = None
    if args.config == "llama8b" and gemm_launches > 0:
        rows_per_launch = kept_units * rows_per_unit / (gemm_launches / 12.0)
        traffic = GEMM_DRAM_BYTES_PER_ROW * rows_per_launch
    roof = {"kernel": "gemm_tc_kernel (tcgen05 projections, fwd dgrad wgrad)", "bound": "tensor",
            "achieved": gemm_achieved, "peak": peaks["bf16_sustained"], "unit": "TFLOP/s",
            "frac": gemm_achieved / peaks["bf16_sustained"] if gemm_achieved else None, "traffic": traffic,
            "traffic_source": "ncu DRAM bytes of a 2-layer capture per kept row, times kept rows per launch",
            "peak_kind": f"bf16 sustained ({peaks['source']})", "launches_per_step": gemm_launches / args.steps,
            "avg_launch_ms": gemm_ms / max(gemm_launches, 1)}
    # attention class (forward and backward kernels) on model FLOPs: 3 x the
    # forward's 4 (len^2 / 2) Dh per head and kept sequence (the backward's
    # recomputation of the scores gets no credit)
    attn_flops = exec_flops - gemm_flops  # per step
    attn_achieved = attn_flops * args.steps / (attn_ms / 1e3) / 1e12 if attn_ms > 0 else None
    attn_roof = {"kernel": "attn_fwd_pp_kernel / attn_fwd_tc_kernel + attn_bwd_tc_kernel", "bound": "tensor",
                 "achieved": attn_achieved, "peak": peaks["bf16_sustained"], "unit": "TFLOP/s",
                 "frac": attn_achieved / peaks["bf16_sustained"] if attn_achieved else None,
                 "launches_per_step": attn_launches / args.steps}
    if clk_serial and attn_achieved:
        attn_roof["frac_at_clock"] = attn_achieved / tensor_peak_at_clock(clk_serial["sm_mhz"])
    if clk_serial and gemm_achieved:
        # the same launches against the tensor rate at the SM clock sampled
        # while they ran: separates kernel efficiency from the clock
        pk = tensor_peak_at_clock(clk_serial["sm_mhz"])
        roof.update({"sm_mhz_timing_pass": clk_serial["sm_mhz"], "peak_at_clock": pk,
                     "frac_at_clock": gemm_achieved / pk})
    line = {
        "metric": METRIC, **result_line(world, B, S, ms),
        "steps": args.steps, "warmup": args.warmup, "higher_is_better": True,
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": config_of(args, cfg, sched, step0 + args.warmup, world),
        "executed_tflops": tflops, "pct_bf16_peak": 100.0 * tflops / peaks["bf16"],
        "pct_bf16_peak_sustained": 100.0 * tflops / peaks["bf16_sustained"],
        "p_bar_expected": p_exp, "p_bar_realized": p_real,
        "skip_speedup": (dense_ms / ms) if dense_ms else None,
        "ideal_speedup": 1.0 / (1.0 - p_real), "dense_ms_per_step": dense_ms,
        "attention_roofline": attn_roof,
        "kernel_ms_per_step": {"gemm": gemm_ms / args.steps, "attention": attn_ms / args.steps,
                               "rowwise": row_ms / args.steps,
                               "serialized_ms_per_step": ms_serial,
                               "note": "separate pass, weight-gradient products not overlapped"},
        "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "clocks": clk,
        "gpu_launches": None,
    }
    # kernels of this library launched in the timed region: per step the mask
    # kernel and the RoPE table, then per layer 4 GEMMs + attention + 4
    # row-wise kernels forward, 8 GEMMs + 3 attention kernels + 7 row-wise
    # kernels backward (RoPE kernels drop out when theta = 0)
    # (per token also 3 + 3 tail-zeroing launches per layer; with sub-layer
    # masks one more row-wise gather per layer in the backward)
    rope = 1 if cfg.get("rope_theta") else 0
    line["gpu_launches"] = args.steps * (1 + rope + L * (4 + 1 + 3 + rope + 8 + 3 + 6 + rope + (6 if tok else 0) +
                                                         (1 if sub else 0)))
    if rank == 0:
        print(json.dumps(line), flush=True)
    st.close()
    if world > 1:
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
