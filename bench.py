"""Benchmark: tokens/s of one adaptive-depth MoE forward on GB300, and % of roofline.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config mixtral] [--impl ours|reference]

A step is one full forward (all layers: router, decide, compact, gather,
grouped FFN, combine) over T tokens of the seeded synthetic workload, starting
from a prepared initial hidden state and token state (a device copy that is
part of the step).  Inputs are larger than L2 (Mixtral-shaped: 90 GB of expert
weights, 134 MB of hidden states), so no L2 flush is needed.

The line carries the dominant GEMM launch's roofline (against the measured
dense bf16 burst peak, the sustained peak beside it), the whole forward's
roofline (algorithmic FLOPs and bytes of the executed work), the end-to-end
figure through the host-buffer entry point, the oracle on the host cores, and
an extra_workloads block with the Qwen- and Switch-shaped forwards and the
Mixtral-shaped decode stress case.

--gpus N outside torchrun starts N ranks itself; each rank runs an independent
replica on its own GPU (weak scaling: the token batches are independent and the
method has no exchange step); rank 0 prints one JSON line with the max time
over ranks.

--impl reference times the CPU oracle on the host cores on a bounded sample
of the same workload (S tokens through L layers, projected to tokens/s of a
full forward).
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "tokens/s per adaptive-depth MoE forward on 1 GB300; % of roofline"
UNIT = "tokens/s"

# Oracle sample per configuration: (tokens, layers) -- about 10-30 s on 16 cores.
CPU_SAMPLE = {"switch_tiny": (64, 4), "switch": (512, 12), "qwen": (256, 2), "mixtral": (128, 2),
              "mixtral_decode": (128, 2)}


def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", str(rank)))
    return rank, world, local


def init_dist(world):
    if world <= 1:
        return None
    import torch.distributed as dist
    dist.init_process_group("gloo")
    return dist


def max_over_ranks(dist, v: float) -> float:
    if dist is None:
        return v
    import torch
    t = torch.tensor([v], dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def barrier(dist):
    if dist is not None:
        dist.barrier()


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as fh:
            j = json.load(fh)
        return dict(hbm=j["hbm_gbs"], bf16=j["bf16_tflops"], bf16_sus=j["bf16_tflops_sustained"],
                    source="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, source="fallback")


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=self.fh, stderr=subprocess.DEVNULL)
            # let the sampler come up (first line written) before the timed region starts
            t_end = time.time() + 5.0
            while time.time() < t_end and os.path.getsize(self.path) == 0 and self.proc.poll() is None:
                time.sleep(0.02)
            self.skip = 0
            with open(self.path) as fh:
                self.skip = sum(1 for _ in fh)          # lines from before the timed region
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
        self.fh.close()
        rows = []
        with open(self.path) as fh:
            for i, line in enumerate(fh):
                parts = [x.strip() for x in line.split(",")]
                if i >= self.skip and len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0,
                    "note": "timed region shorter than the 200 ms sampling interval"}
        def num(x):
            try:
                return float(x)
            except ValueError:
                return float("nan")
        sm = [num(r[1]) for r in rows]
        mx = [num(r[2]) for r in rows]
        reasons = set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for r in rows:
            for n, v in zip(names, r[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        loaded = [s for s in sm if not math.isnan(s)]
        return {"sm_mhz": statistics.median(loaded) if loaded else None,
                "sm_max_mhz": max(mx) if mx else None, "reasons": sorted(reasons), "samples": len(rows)}


def workload_config(args):
    """The named workload; --layers / --tokens shrink it for profiling runs."""
    from paper_2608_00573_gb300 import workload as W
    cfg = W.CONFIGS[args.config]
    if args.exit_prediction:
        cfg = cfg.replace(n_centroids=args.exit_prediction)
    if args.budget:
        cfg = cfg.replace(budget=args.budget)      # same calibrated thresholds, other Dbar
    if args.full_block:
        cfg = W.with_attention(cfg)                # attention sublayer in front of every MoE step
    if args.layers or args.tokens:
        over = {}
        if args.layers:
            over["N"] = args.layers
        if args.tokens:
            over["T"] = args.tokens
        calib = W.load_calibration(cfg.name)
        cfg = cfg.replace(**over)
        cfg._calib = None if calib is None else {k: (v[: cfg.N] if isinstance(v, list) else v)
                                                 for k, v in calib.items()}
        cfg.name = f"{cfg.name}[N={cfg.N},T={cfg.T}]"
    return cfg


def make_workload(cfg, device):
    from paper_2608_00573_gb300 import workload as W
    calib = getattr(cfg, "_calib", "auto")
    small = W.make_small_weights(cfg, calib=calib)
    tables = W.make_tables(cfg, small["W_r"], calib=calib)
    experts = W.make_expert_weights_device(cfg, device=device)
    tok = W.make_tokens(cfg)
    return small, tables, experts, tok


def cpu_model() -> str:
    """The host CPU's model string (x86 "model name", or the Arm implementer and
    part numbers), with the machine type; never raises."""
    import platform
    name = ""
    try:
        info = {}
        with open("/proc/cpuinfo") as fh:
            for line in fh:
                if ":" in line:
                    k, v = line.split(":", 1)
                    info.setdefault(k.strip(), v.strip())
        if info.get("model name"):
            name = info["model name"]
        elif info.get("CPU part"):
            name = f"implementer {info.get('CPU implementer', '?')} part {info['CPU part']}"
    except OSError:
        pass
    return f"{name} ({platform.machine()})" if name else platform.machine()


def config_dict(cfg, world):
    """The workload description both arms print (same keys, same values)."""
    return {"workload": cfg.name, "T": cfg.T, "N": cfg.N, "d": cfg.d, "E": cfg.E, "k": cfg.k, "F": cfg.F,
            "F_sh": cfg.F_sh, "H": cfg.H, "budget": cfg.budget, "exit_prediction_centroids": cfg.n_centroids,
            "parallelism": f"replicas{world}",
            "l2": "inputs larger than L2 (expert weights and hidden states)",
            "full_block": bool(cfg.attn_heads),
            **({"attn_heads": cfg.attn_heads, "attn_kv_heads": cfg.attn_kv_heads, "head_dim": cfg.head_dim,
                "attn_seq": cfg.attn_seq} if cfg.attn_heads else {})}


def _experts_per_layer_host(experts, n_layers):
    import numpy as np
    import torch
    out = []
    for l in range(n_layers):
        d = {}
        for k, v in experts.items():
            if v is None:
                continue
            x = v[l]
            if hasattr(x, "detach"):
                x = x.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
            d[k] = np.ascontiguousarray(x)
        out.append(d)
    return out


def cpu_sample(cfg, small, tables, ex_l, tok, n_tok, n_layers, steps=1, nthreads=0):
    """Time the oracle on n_tok tokens through layers 0..n_layers-1 (ex_l: the
    host expert weights of those layers; nthreads 0 = every host core).  Returns
    (tokens/s of a full forward per step, seconds per step, threads used,
    sample description)."""
    import numpy as np
    from oracle import oracle as O
    O.build()
    om = O.OracleModel(cfg, tables, small, None)
    n_layers = min(n_layers, cfg.N)
    sub = {k: np.ascontiguousarray(v[:n_tok]) for k, v in tok.items()}
    threads = O.max_threads() if nthreads == 0 else nthreads
    secs = []
    for _ in range(steps):
        h = sub["h"].copy()
        st = {k: v.copy() for k, v in sub.items() if k != "h"}
        t0 = time.perf_counter()
        for l in range(n_layers):
            h, st, _ = O.layer_step(om, l, h, st, experts_l=ex_l[l], nthreads=threads)
        secs.append(time.perf_counter() - t0)
    vals = [n_tok / (t * cfg.N / n_layers) for t in secs]
    return vals, secs, threads, (f"{n_tok} tokens x layers 0..{n_layers - 1} of the {cfg.name} workload, "
                                 f"time scaled by {cfg.N}/{n_layers} to a full forward")


def cpu_tiny_forward(nthreads=0):
    """The oracle's full forward (every layer, every row) on the tiny workload."""
    from oracle import oracle as O
    from paper_2608_00573_gb300 import workload as W
    cfg = W.CONFIGS["switch_tiny"]
    small = W.make_small_weights(cfg)
    tables = W.make_tables(cfg, small["W_r"])
    experts = W.make_expert_weights_host(cfg)
    om = O.OracleModel(cfg, tables, small, experts)
    tok = W.make_tokens(cfg)
    h = tok.pop("h")
    threads = O.max_threads() if nthreads == 0 else nthreads
    t0 = time.perf_counter()
    O.forward(om, h, tok, nthreads=threads)
    s = time.perf_counter() - t0
    return {"value": cfg.T / s, "unit": UNIT, "ms_per_forward": s * 1e3, "cores": threads,
            "sample": f"full {cfg.N}-layer forward of the {cfg.name} workload (T = {cfg.T})"}


def cpu_baseline(cfg, small, tables, ex_l, tok):
    """The oracle on the host cores: a bounded sample on every core (the
    headline), a smaller one on one thread, and the tiny workload's full
    forward both ways."""
    from oracle import oracle as O
    n_tok, n_layers = CPU_SAMPLE.get(cfg.name, (64, 2))
    cores = O.max_threads()          # before any single-thread run changes the OpenMP default
    vals, secs, threads, sample = cpu_sample(cfg, small, tables, ex_l, tok, n_tok, n_layers, nthreads=cores)
    tiny = cpu_tiny_forward(cores)
    n1 = max(1, n_tok // 32)
    v1, s1, _, sample1 = cpu_sample(cfg, small, tables, ex_l, tok, n1, n_layers, nthreads=1)
    return {"value": vals[0], "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample,
            "cpu": cpu_model(),
            "single_thread": {"value": v1[0], "unit": UNIT, "cores": 1, "sample": sample1},
            "tiny_forward": tiny, "tiny_forward_single_thread": cpu_tiny_forward(1)}


def run_reference(args):
    rank, world, local = dist_env()
    if rank != 0:
        return
    import torch
    cfg = workload_config(args)
    device = "cuda" if torch.cuda.is_available() else "cpu"
    small, tables, experts, tok = make_workload(cfg, device)
    n_tok, n_layers = CPU_SAMPLE.get(cfg.name, (64, 2))
    ex_l = _experts_per_layer_host(experts, min(n_layers, cfg.N))
    del experts
    vals, secs, threads, sample = cpu_sample(cfg, small, tables, ex_l, tok, n_tok, n_layers,
                                             steps=args.warmup + args.steps)
    vals, secs = vals[args.warmup:], secs[args.warmup:]
    v = statistics.median(vals)
    line = {"metric": METRIC, "value": v, "unit": UNIT, "impl": "reference", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": statistics.median(secs) * 1e3,
            "ms_per_step_kind": (f"measured time of one sample step ({sample}); value projects that sample "
                                 f"to tokens/s of a full forward"),
            "projected_ms_per_full_forward": cfg.T / v * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "config": config_dict(cfg, world),
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample,
                             "cpu": cpu_model()},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# Per live (token, layer): the hidden row read and written, and the per-token
# state read and written (s, Dhat, Dbar, pJ, alive, last_exec, xi_last in;
# s, Dhat, last_exec, xi_last, alive, exit_layer out).
STATE_BYTES_PER_TOKEN_LAYER = 19 + 13


def rooflines(cfg, st, steps, ms_step, peaks, traffic, st_k=None):
    """The dominant GEMM launch kind's roofline and the whole forward's.

    Forward: F_alg = executed expert GEMM FLOPs + router/exit-head/centroid dot
    products of the live tokens; B_alg = the weights of the experts that received
    work (once per layer), the router/exit-head/norm rows of every layer run,
    and per live token-layer its hidden row in and out plus its state.  Roofline
    time = max(F_alg / bf16 peak, B_alg / HBM peak); frac = roofline / measured,
    against the dense burst peak, with the sustained peak beside it.  st_k:
    the counters of the pass whose events timed the GEMM launches (default st)."""
    sk = st if st_k is None else st_k
    kinds = {"grouped_gemm_gate_up": (sk["ms_gemm_up"], sk["flops_gemm_up"], sk["n_gemm_up"], sk["bytes_gemm_up"]),
             "grouped_gemm_down": (sk["ms_gemm_down"], sk["flops_gemm_down"], sk["n_gemm_down"],
                                   sk["bytes_gemm_down"])}
    dom = max(kinds, key=lambda k: kinds[k][0])
    ms_k, fl_k, n_k, by_k = kinds[dom]
    achieved = fl_k / (ms_k / 1e3) / 1e12 if ms_k > 0 else 0.0
    achieved_bw = by_k / (ms_k / 1e3) / 1e9 if ms_k > 0 else 0.0
    tensor_bound = fl_k / (peaks["bf16"] * 1e12) >= by_k / (peaks["hbm"] * 1e9)
    if tensor_bound:
        roof = {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": peaks["bf16"], "unit": "TFLOP/s",
                "frac": achieved / peaks["bf16"], "traffic": traffic,
                "peak_source": f"{peaks['source']} dense bf16 (burst)",
                "peak_sustained": peaks["bf16_sus"], "frac_sustained": achieved / peaks["bf16_sus"]}
    else:
        roof = {"bound": "hbm", "kernel": dom, "achieved": achieved_bw, "peak": peaks["hbm"], "unit": "GB/s",
                "frac": achieved_bw / peaks["hbm"], "traffic": traffic, "peak_source": f"{peaks['source']} HBM copy"}
    roof.update(flops_per_launch=fl_k / max(n_k, 1), bytes_per_launch=by_k / max(n_k, 1),
                ms_per_launch=ms_k / max(n_k, 1), launches_per_step=n_k / max(steps, 1) if st_k is None else None)
    rows = cfg.E + cfg.C + cfg.n_centroids
    live = st["layer_tokens"] / steps
    layers_run = st["layer_calls"] / steps
    f_alg = st["gemm_flops"] / steps + live * 2.0 * cfg.d * rows
    b_alg = (st["bytes_expert_weights"] / steps + layers_run * 2.0 * cfg.d * (rows + 1)
             + live * (2.0 * 2 * cfg.d + STATE_BYTES_PER_TOKEN_LAYER))
    if cfg.attn_heads:
        # Attention sublayer for all T tokens of every layer: its FLOPs, the
        # projection weights once, and the rows it must read and write.
        hd = cfg.attn_heads * cfg.head_dim
        f_alg += (st["flops_attn_gemm"] + st["flops_attn"]) / steps
        b_alg += layers_run * (2.0 * (cfg.n_qkv * cfg.d + cfg.d * hd) + 2.0 * cfg.T * (
            2 * cfg.d + 2 * cfg.n_qkv + 2 * hd + 2 * cfg.d + cfg.d))
    t_f = f_alg / (peaks["bf16"] * 1e12) * 1e3
    t_b = b_alg / (peaks["hbm"] * 1e9) * 1e3
    t_fs = f_alg / (peaks["bf16_sus"] * 1e12) * 1e3
    fwd = {"flops_per_forward": f_alg, "bytes_per_forward": b_alg, "bound": "tensor" if t_f >= t_b else "hbm",
           "roofline_ms": max(t_f, t_b), "frac": max(t_f, t_b) / ms_step,
           "roofline_ms_sustained": max(t_fs, t_b), "frac_sustained": max(t_fs, t_b) / ms_step,
           "gemm_flops_per_forward": st["gemm_flops"] / steps,
           "expert_weight_bytes_per_forward": st["bytes_expert_weights"] / steps}
    return roof, fwd


def decisions_block(st, steps, T):
    pairs = (st["pairs_local_exact"] + st["pairs_local_sub"] + st["pairs_remote_exact"] + st["pairs_remote_sub"])
    return {"layer_tokens": st["layer_tokens"] // steps,
            "skip_share": st["skipped"] / max(st["layer_tokens"], 1),
            "exit_share_of_tokens": st["exited"] / steps / T,
            "remote_share_of_pairs": (st["pairs_remote_exact"] + st["pairs_remote_sub"]) / max(pairs, 1),
            "substitute_share_of_pairs": (st["pairs_local_sub"] + st["pairs_remote_sub"]) / max(pairs, 1)}


def stored_traffic(cfg, kernel):
    tp = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(tp):
        return None
    with open(tp) as fh:
        tj = json.load(fh)
    ent = tj.get(cfg.name, {}).get(kernel)
    if ent and ent.get("kernel_rev") == KERNEL_REV.get(kernel):
        return ent.get("bytes_per_launch")
    return None


class Timed:
    """One engine timing forwards of a workload: the forward replays as a CUDA
    graph on a stream of its own (the legacy default stream cannot be
    captured), CUDA events bracket the grouped GEMM launches only (every event
    pair inside a graph costs a few microseconds) and the whole timed region.
    A step copies one of the prepared initial token states into the working
    buffers (part of the step) and runs the forward."""

    def __init__(self, cfg, tables, small, experts, pool, device, T_max=None, profile=2, graphs=True):
        import torch
        from paper_2608_00573_gb300 import binding as B
        self.torch = torch
        self.cfg = cfg
        self.eng = B.Engine(cfg, tables, small, experts, T_max=T_max or cfg.T, device=device, profile=profile,
                            graphs=graphs)
        self.pool = [self.eng.tokens_to_device(t) for t in pool]
        self.work = {k: v.clone() for k, v in self.pool[0].items()}
        self.stream = torch.cuda.Stream(device)
        self.i = 0

    def step(self):
        src = self.pool[self.i % len(self.pool)]
        self.i += 1
        with self.torch.cuda.stream(self.stream):
            for k in self.work:
                self.work[k].copy_(src[k], non_blocking=True)
        self.eng.forward(self.work, stream=self.stream)

    def run(self, steps, warmup, dist=None, clock_index=None):
        torch = self.torch
        for _ in range(warmup):
            self.step()
        torch.cuda.synchronize()
        st0 = self.eng.stats()
        if st0["status"] != 0:
            raise RuntimeError(f"{self.cfg.name}: warm-up failed: {st0}")
        self.eng.reset_stats()
        clocks = ClockSampler(clock_index) if clock_index is not None else None
        barrier(dist)
        torch.cuda.synchronize()
        if clocks:
            clocks.start()
        ev0 = torch.cuda.Event(enable_timing=True)
        ev1 = torch.cuda.Event(enable_timing=True)
        ev0.record(self.stream)
        for _ in range(steps):
            self.step()
        ev1.record(self.stream)
        torch.cuda.synchronize()
        barrier(dist)
        ms_total = ev0.elapsed_time(ev1)
        clk = clocks.stop() if clocks else None
        st = self.eng.stats()
        if st["status"] != 0 or st["device_error"]:
            raise RuntimeError(f"{self.cfg.name}: timed run failed: {st}")
        return ms_total / steps, clk, st

    def close(self):
        self.eng.close()


def extra_workloads(args, device, local, peaks, mixtral_experts):
    """Timed lines for the other workloads: the Qwen- and Switch-shaped
    forwards and the Mixtral-shaped decode stress case (T in {1, 8, 64, 256} at
    budget 0.02, and T = 64 at budgets 0.005 and 0.05), each step on a fresh
    initial state drawn from a pool of 16.  The decode case reuses the resident
    Mixtral-shaped expert weights.  The step time comes from a pass without
    per-kernel events (at these sizes the event nodes inside the graph cost a
    noticeable share of the step); the dominant GEMM's launch time from a
    second pass of the same steps with events around the GEMM launches."""
    import torch
    from paper_2608_00573_gb300 import workload as W
    out = {}

    def record(name, cfg, tables, small, experts, pool, steps, warmup):
        timed = Timed(cfg, tables, small, experts, pool, device, profile=0)
        ms, clk, st = timed.run(steps, warmup, clock_index=local)
        timed.close()
        ksteps = min(steps, 200)
        timed = Timed(cfg, tables, small, experts, pool, device, profile=2)
        _, _, st_k = timed.run(ksteps, warmup)
        timed.close()
        roof, fwd = rooflines(cfg, st, steps, ms, peaks, stored_traffic(cfg, "grouped_gemm_gate_up"), st_k=st_k)
        roof["timing"] = f"events around the GEMM launches in a second pass of {ksteps} steps"
        out[name] = {"workload": cfg.name, "T": cfg.T, "N": cfg.N, "budget": cfg.budget, "steps": steps,
                     "warmup": warmup, "ms_per_step": ms, "tokens_per_s": cfg.T / (ms / 1e3),
                     "roofline": roof, "forward_roofline": fwd, "decisions": decisions_block(st, steps, cfg.T),
                     "gpu_launches": st["launches"], "clocks": clk}

    dec = W.CONFIGS["mixtral_decode"]
    runs = [(T, dec.budget) for T in (1, 8, 64, 256)] + [(64, 0.005), (64, 0.05)]
    for T, budget in runs:
        cfg = dec.replace(T=T, budget=budget)
        small = W.make_small_weights(cfg)
        tables = W.make_tables(cfg, small["W_r"])
        pool = [W.make_tokens(cfg, T=T, seed_offset=1000 * T + i) for i in range(16)]
        name = f"mixtral_decode_T{T}" + ("" if budget == dec.budget else f"_budget{budget:g}")
        record(name, cfg, tables, small, mixtral_experts, pool, args.decode_steps, max(args.warmup, 3))
    for wl, steps in (("qwen", max(args.steps, 50)), ("switch", max(args.steps, 400))):
        cfg = W.CONFIGS[wl]
        small, tables, experts, tok = make_workload(cfg, device)
        record(wl, cfg, tables, small, experts, [tok], steps, max(args.warmup, 3))
        del experts
        torch.cuda.empty_cache()
    return out


def run_ours(args):
    import torch
    from paper_2608_00573_gb300 import binding as B

    rank, world, local = dist_env()
    dist = init_dist(world)
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    B.lib()
    cfg = workload_config(args)
    T = cfg.T
    small, tables, experts, tok = make_workload(cfg, device)
    peaks = load_peaks()

    timed = Timed(cfg, tables, small, experts, [tok], device)
    ms_step, clk, st = timed.run(args.steps, args.warmup, dist=dist, clock_index=local)
    ms_step = max_over_ranks(dist, ms_step)
    value = T * world / (ms_step / 1e3)

    # End to end through the public host-buffer entry point (pinned host memory,
    # copies in both directions inside the timed region).
    eng, stream = timed.eng, timed.stream
    host = {k: v.cpu().pin_memory() for k, v in timed.pool[0].items()}
    host_src = {k: v.clone().pin_memory() for k, v in host.items()}
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    eng.forward_host(host, stream=stream)
    barrier(dist)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        for k in host:
            host[k].copy_(host_src[k])
        eng.forward_host(host, stream=stream)
    e2e_s = max_over_ranks(dist, (time.perf_counter() - t0) / args.steps)
    e2e = {"value": T * world / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": h2d}
    timed.close()

    roof, fwd = rooflines(cfg, st, args.steps, ms_step, peaks, stored_traffic(cfg, "grouped_gemm_gate_up"))
    dom = roof["kernel"]
    roof["traffic"] = stored_traffic(cfg, dom)

    # Per-kernel split: a separate pass of plain launches with events around
    # every kernel, after the timed region (informational).
    kinds_ms = ("router", "decide", "compact", "gather", "gemm_up", "gemm_down", "combine")
    if cfg.attn_heads:
        kinds_ms = kinds_ms + ("attn", "attn_gemm")
    split = Timed(cfg, tables, small, experts, [tok], device, profile=1, graphs=False)
    _, _, st_split = split.run(args.steps, args.warmup)
    split.close()
    kernel_ms = {k: st_split[f"ms_{k}"] / args.steps for k in kinds_ms}

    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": config_dict(cfg, world),
        "roofline": roof,
        "forward_roofline": fwd,
        "kernel_ms_per_step": kernel_ms,
        "kernel_split_pass": "plain launches with events around every kernel, after the timed region",
        "decisions": decisions_block(st, args.steps, T),
        "e2e": e2e,
        "gpu_launches": st["launches"],
        "clocks": clk,
    }
    cpu_ex = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu_ex = _experts_per_layer_host(experts, min(CPU_SAMPLE.get(cfg.name, (64, 2))[1], cfg.N))
    if (world == 1 and not args.no_extra and cfg.name == "mixtral" and not cfg.attn_heads
            and not (args.layers or args.tokens or args.budget or args.exit_prediction)):
        line["extra_workloads"] = extra_workloads(args, device, local, peaks, experts)
    del experts
    torch.cuda.empty_cache()
    if cpu_ex is not None:
        line["cpu_baseline"] = cpu_baseline(cfg, small, tables, cpu_ex, tok)
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


# Revision tag of each timed GEMM launch kind; a stored ncu traffic figure is
# used only when it was taken on that revision.
KERNEL_REV = {"grouped_gemm_gate_up": "gemm-v10", "grouped_gemm_down": "gemm-v12"}


def launch_ranks(args, argv):
    """--gpus N outside torchrun: start N ranks on this node through
    torch.distributed.run (127.0.0.1 rendezvous) and return their exit code.
    Under torchrun, N must equal WORLD_SIZE."""
    world = os.environ.get("WORLD_SIZE")
    if world is not None:
        if int(world) != args.gpus:
            print(f"bench.py: --gpus {args.gpus} but WORLD_SIZE={world}", file=sys.stderr)
            return 2
        return None
    if args.gpus == 1:
        return None
    import socket
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", f"--nproc-per-node={args.gpus}",
           "--master-addr", "127.0.0.1", "--master-port", str(port), os.path.abspath(__file__), *argv]
    return subprocess.call(cmd)


def main(argv=None):
    argv = sys.argv[1:] if argv is None else argv
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default="mixtral")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-extra", action="store_true",
                    help="skip the extra_workloads block (Qwen-, Switch-shaped and decode lines)")
    ap.add_argument("--decode-steps", type=int, default=2000,
                    help="timed steps per decode batch size in extra_workloads (the decode stress case: 2000)")
    ap.add_argument("--budget", type=float, default=0.0, help="per-token quality budget Dbar (default: the workload's)")
    ap.add_argument("--full-block", action="store_true",
                    help="the full transformer block: the model family's attention sublayer in front of every MoE step")
    ap.add_argument("--layers", type=int, default=0, help="profiling only: first N layers of the workload")
    ap.add_argument("--tokens", type=int, default=0, help="profiling only: T tokens instead of the workload's")
    ap.add_argument("--exit-prediction", type=int, default=0,
                    help="K_c centroids per layer for the token-similarity exit prediction (Eq. 36); 0 = off")
    args = ap.parse_args(argv)
    rc = launch_ranks(args, argv)
    if rc is not None:
        return rc
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)
    return 0


if __name__ == "__main__":
    sys.exit(main())
