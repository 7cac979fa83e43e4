"""Benchmark: tokens/s of one adaptive-depth MoE forward on GB300, and % of roofline.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config mixtral] [--impl ours|reference]

A step is one full forward (all layers: decide, compact, gather, grouped FFN,
combine) over T tokens of the seeded synthetic workload, starting from the
same initial hidden states and token state each step (a 134 MB device copy
that is part of the step).  Inputs are larger than L2 (Mixtral-shaped: 90 GB
of expert weights, 134 MB of hidden states), so no L2 flush is needed.

Under torchrun each rank runs an independent replica on its own GPU (weak
scaling: the token batches are independent and the method has no exchange
step); rank 0 prints one JSON line with the max time over ranks.

--impl reference times the CPU oracle on the host cores on a bounded sample
of the same workload (S tokens through L layers, scaled to tokens/s of a full
forward).
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
import threading
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


def cpu_baseline(cfg, small, tables, experts, tok, n_tok, n_layers, steps=1):
    """Time the oracle (all host cores) on n_tok tokens through layers 0..n_layers-1."""
    import numpy as np
    import torch
    from oracle import oracle as O
    O.build()
    om = O.OracleModel(cfg, tables, small, None)
    n_layers = min(n_layers, cfg.N)
    ex_l = []
    for l in range(n_layers):
        d = {}
        for k, v in experts.items():
            if v is None:
                continue
            x = v[l]
            if hasattr(x, "detach"):
                x = x.detach().contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
            d[k] = np.ascontiguousarray(x)
        ex_l.append(d)
    sub = {k: np.ascontiguousarray(v[:n_tok]) for k, v in tok.items()}
    threads = O.max_threads()
    times = []
    for _ in range(steps):
        h = sub["h"].copy()
        st = {k: v.copy() for k, v in sub.items() if k != "h"}
        t0 = time.perf_counter()
        for l in range(n_layers):
            h, st, _ = O.layer_step(om, l, h, st, experts_l=ex_l[l], nthreads=threads)
        times.append(time.perf_counter() - t0)
    per_forward = [t * cfg.N / n_layers for t in times]
    vals = [n_tok / t for t in per_forward]
    return vals, threads, f"{n_tok} tokens x layers 0..{n_layers - 1} of the {cfg.name} workload, " \
                          f"time scaled by {cfg.N}/{n_layers} to a full forward"


def run_reference(args):
    rank, world, local = dist_env()
    if rank != 0:
        return
    import torch
    cfg = workload_config(args)
    device = "cuda" if torch.cuda.is_available() else "cpu"
    small, tables, experts, tok = make_workload(cfg, device)
    n_tok, n_layers = CPU_SAMPLE.get(cfg.name, (64, 2))
    vals, threads, sample = cpu_baseline(cfg, small, tables, experts, tok, n_tok, n_layers,
                                         steps=args.warmup + args.steps)
    vals = vals[args.warmup:]
    v = statistics.median(vals)
    ms = cfg.T / v * 1e3
    line = {"metric": METRIC, "value": v, "unit": UNIT, "impl": "reference", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": {"workload": cfg.name, "T": cfg.T, "N": cfg.N, "d": cfg.d, "E": cfg.E, "k": cfg.k,
                       "F": cfg.F, "F_sh": cfg.F_sh, "H": cfg.H, "budget": cfg.budget},
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": threads, "kind": "oracle", "sample": sample,
                             "cpu": cpu_model()},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def run_ours(args):
    import torch
    from paper_2608_00573_gb300 import binding as B
    from paper_2608_00573_gb300 import workload as W

    rank, world, local = dist_env()
    dist = init_dist(world)
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)
    B.lib()
    cfg = workload_config(args)
    T = cfg.T
    small, tables, experts, tok = make_workload(cfg, device)
    # Timed engine: the forward replays as a CUDA graph; CUDA events bracket the
    # grouped GEMM launches only (the roofline's kernel), since every event pair
    # inside a graph costs a few microseconds.
    eng = B.Engine(cfg, tables, small, experts, T_max=T, device=device, profile=2, graphs=True)
    tok0 = eng.tokens_to_device(tok)
    work = {k: v.clone() for k, v in tok0.items()}
    torch.cuda.synchronize()
    # A stream of our own: the library replays the forward as a CUDA graph,
    # which the legacy default stream cannot capture.
    stream = torch.cuda.Stream(device)
    torch.cuda.set_stream(stream)

    def step():
        for k in work:
            work[k].copy_(tok0[k], non_blocking=True)
        eng.forward(work, stream=stream)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    st0 = eng.stats()
    if st0["status"] != 0:
        raise RuntimeError(f"warm-up failed: {st0}")
    eng.reset_stats()
    clocks = ClockSampler(local)
    barrier(dist)
    torch.cuda.synchronize()
    clocks.start()
    ev0 = torch.cuda.Event(enable_timing=True)
    ev1 = torch.cuda.Event(enable_timing=True)
    ev0.record(stream)
    for _ in range(args.steps):
        step()
    ev1.record(stream)
    torch.cuda.synchronize()
    barrier(dist)
    ms_total = ev0.elapsed_time(ev1)
    clk = clocks.stop()
    st = eng.stats()
    if st["status"] != 0 or st["device_error"]:
        raise RuntimeError(f"timed run failed: {st}")
    ms_step = max_over_ranks(dist, ms_total / args.steps)
    value = T * world / (ms_step / 1e3)

    # End to end through the public host-buffer entry point (pinned host memory).
    host = {k: v.cpu().pin_memory() for k, v in tok0.items()}
    host_src = {k: v.clone().pin_memory() for k, v in host.items()}
    h2d = sum(v.numel() * v.element_size() for v in host.values())
    for _ in range(1):
        eng.forward_host(host, stream=stream)
    barrier(dist)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        for k in host:
            host[k].copy_(host_src[k])
        eng.forward_host(host, stream=stream)
    e2e_s = max_over_ranks(dist, (time.perf_counter() - t0) / args.steps)
    e2e = {"value": T * world / e2e_s, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": h2d}

    # Roofline of the dominant kernel (grouped FFN GEMM) from events recorded
    # around each launch on the launching stream during the timed region.
    peaks = load_peaks()
    kinds = {"grouped_gemm_gate_up": (st["ms_gemm_up"], st["flops_gemm_up"], st["n_gemm_up"], st["bytes_gemm_up"]),
             "grouped_gemm_down": (st["ms_gemm_down"], st["flops_gemm_down"], st["n_gemm_down"],
                                   st["bytes_gemm_down"])}
    dom = max(kinds, key=lambda k: kinds[k][0])
    ms_k, fl_k, n_k, by_k = kinds[dom]
    achieved = fl_k / (ms_k / 1e3) / 1e12 if ms_k > 0 else 0.0
    achieved_bw = by_k / (ms_k / 1e3) / 1e9 if ms_k > 0 else 0.0
    traffic = None
    tp = os.path.join(ROOT, "profiles", "traffic.json")
    if os.path.exists(tp):
        with open(tp) as fh:
            tj = json.load(fh)
        ent = tj.get(cfg.name, {}).get(dom)
        if ent and ent.get("kernel_rev") == KERNEL_REV[dom]:
            traffic = ent.get("bytes_per_launch")
    # The GEMM is tensor-bound when its FLOPs take longer at peak than its bytes.
    tensor_bound = fl_k / (peaks["bf16_sus"] * 1e12) >= by_k / (peaks["hbm"] * 1e9)
    if tensor_bound:
        roof = {"bound": "tensor", "kernel": dom, "achieved": achieved, "peak": peaks["bf16_sus"],
                "unit": "TFLOP/s", "frac": achieved / peaks["bf16_sus"], "traffic": traffic,
                "peak_source": f"{peaks['source']} bf16 sustained"}
    else:
        roof = {"bound": "hbm", "kernel": dom, "achieved": achieved_bw, "peak": peaks["hbm"],
                "unit": "GB/s", "frac": achieved_bw / peaks["hbm"], "traffic": traffic,
                "peak_source": f"{peaks['source']} HBM copy"}
    roof.update(flops_per_launch=fl_k / max(n_k, 1), bytes_per_launch=by_k / max(n_k, 1),
                ms_per_launch=ms_k / max(n_k, 1))
    # Whole-forward roofline: executed GEMM FLOPs at the bf16 peak vs the GEMMs'
    # bytes at HBM, whichever is slower.
    per_fwd_flops = st["gemm_flops"] / args.steps
    per_fwd_bytes = (st["bytes_gemm_up"] + st["bytes_gemm_down"]) / args.steps
    kinds_ms = ("router", "decide", "compact", "gather", "gemm_up", "gemm_down", "combine")
    if cfg.attn_heads:
        # Attention sublayer: its projections and attention FLOPs, and per layer the
        # projection weights once plus the activations it must read and write.
        hd = cfg.attn_heads * cfg.head_dim
        per_fwd_flops += (st["flops_attn_gemm"] + st["flops_attn"]) / args.steps
        per_layer = 2.0 * (cfg.n_qkv * cfg.d + cfg.d * hd) + 2.0 * T * (
            2 * cfg.d + 2 * cfg.n_qkv + 2 * hd + 2 * cfg.d + cfg.d)
        per_fwd_bytes += per_layer * cfg.N
        kinds_ms = kinds_ms + ("attn", "attn_gemm")
    fwd_roof_ms = max(per_fwd_flops / (peaks["bf16_sus"] * 1e12), per_fwd_bytes / (peaks["hbm"] * 1e9)) * 1e3
    # Per-kernel split: a separate pass of plain launches with events around
    # every kernel, after the timed region (informational).
    eng.close()
    eng = B.Engine(cfg, tables, small, experts, T_max=T, device=device, profile=1, graphs=False)
    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()
    eng.reset_stats()
    for _ in range(args.steps):
        step()
    torch.cuda.synchronize()
    st_split = eng.stats()
    kernel_ms = {k: st_split[f"ms_{k}"] / args.steps for k in kinds_ms}
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": cfg.name, "T": T, "N": cfg.N, "d": cfg.d, "E": cfg.E, "k": cfg.k, "F": cfg.F,
                   "F_sh": cfg.F_sh, "H": cfg.H, "budget": cfg.budget, "exit_prediction_centroids": cfg.n_centroids,
                   "parallelism": f"replicas{world}",
                   "l2": "inputs larger than L2 (expert weights and hidden states)",
                   "full_block": bool(cfg.attn_heads),
                   **({"attn_heads": cfg.attn_heads, "attn_kv_heads": cfg.attn_kv_heads, "head_dim": cfg.head_dim,
                       "attn_seq": cfg.attn_seq} if cfg.attn_heads else {})},
        "roofline": roof,
        "forward_roofline": {"gemm_flops_per_forward": per_fwd_flops, "gemm_bytes_per_forward": per_fwd_bytes,
                             "roofline_ms": fwd_roof_ms, "frac": fwd_roof_ms / ms_step},
        "kernel_ms_per_step": kernel_ms,
        "kernel_split_pass": "plain launches with events around every kernel, after the timed region",
        "decisions": {"layer_tokens": st["layer_tokens"] // args.steps,
                      "skip_share": st["skipped"] / max(st["layer_tokens"], 1),
                      "exit_share_of_tokens": st["exited"] / args.steps / T,
                      "remote_share_of_pairs": (st["pairs_remote_exact"] + st["pairs_remote_sub"]) /
                      max(st["pairs_local_exact"] + st["pairs_local_sub"] + st["pairs_remote_exact"] +
                          st["pairs_remote_sub"], 1)},
        "e2e": e2e,
        "gpu_launches": st["launches"],
        "clocks": clk,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        n_tok, n_layers = CPU_SAMPLE.get(cfg.name, (64, 2))
        vals, threads, sample = cpu_baseline(cfg, small, tables, experts, tok, n_tok, n_layers)
        line["cpu_baseline"] = {"value": vals[0], "unit": UNIT, "cores": threads, "kind": "oracle",
                                "sample": sample, "cpu": cpu_model()}
    eng.close()
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


# Revision tag of each timed GEMM launch kind; a stored ncu traffic figure is
# used only when it was taken on that revision.
KERNEL_REV = {"grouped_gemm_gate_up": "gemm-v7", "grouped_gemm_down": "gemm-v8"}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=5)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--config", default="mixtral")
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--budget", type=float, default=0.0, help="per-token quality budget Dbar (default: the workload's)")
    ap.add_argument("--full-block", action="store_true",
                    help="the full transformer block: the model family's attention sublayer in front of every MoE step")
    ap.add_argument("--layers", type=int, default=0, help="profiling only: first N layers of the workload")
    ap.add_argument("--tokens", type=int, default=0, help="profiling only: T tokens instead of the workload's")
    ap.add_argument("--exit-prediction", type=int, default=0,
                    help="K_c centroids per layer for the token-similarity exit prediction (Eq. 36); 0 = off")
    args = ap.parse_args()
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
