"""Benchmark: NOBLE linear fwd+bwd on the 1.5B-decoder-scale layer shapes.

One step = forward + backward (dx and every parameter gradient) of the three
CosNet-augmented layers of a 1.5B-scale decoder block at T = 16384 tokens
(batch 8 x seq 2048), r = 128: FFN up 2048->8192, FFN down 8192->2048 and QKV
2048->6144, bf16 operands with fp32 accumulation, all through the C ABI.

Reported: whole-job TFLOP/s over algorithmic FLOPs 6 T (d_in d_out +
r (d_in + d_out) + r^2) per layer, the overhead against the same library's
plain (r = 0) layer of the same shapes, a roofline entry for the dominant
kernel, and the fp64 oracle's throughput on a bounded sample of the same work
(host cores).  ``--impl reference`` times only the oracle (see below).

Launch: ``python bench.py --gpus N --steps K --warmup W``; for N > 1 under
torchrun each rank runs the same per-GPU workload (replicas: the layer needs no
exchange in this benchmark), timing is max over ranks and ``value`` the sum.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import threading
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

from paper_2603_06492_gb300.inputs import (CONFIGS, PAPER_WORKLOAD_SEED, PAPER_WORKLOADS, make_cos3_inputs,  # noqa: E402
                                           layer_seed, make_layer_inputs)

CONFIG_INDEX = 3
WORKLOADS = {
    0: "tiny correctness case, T=256, 128->128, r=16, fp32, fwd+bwd",
    1: "250M-scale attention QKV + output, T=8192, d=1024, r=64, CosNet, fwd+bwd",
    2: "250M-scale FFN up + down, T=8192, d=1024, r=64, CosNet, fwd+bwd",
    3: "1.5B-scale FFN up/down + QKV, T=16384, d=2048, r=128, CosNet, fwd+bwd",
    4: "ViT-Base-shaped QKV + FFN up/down, T=50432, d=768, r in {16..256}, CosNet, fwd+bwd",
    "geglu-base": "paper Base model GeGLU FFN (gate, up 1024->2752, down 2752->1024), T=8192, r=64, CosNet, fwd+bwd",
    "geglu-large": "paper Large model GeGLU FFN (gate, up 2048->5504, down 5504->2048), T=16384, r=128, CosNet, "
                   "fwd+bwd",
}

# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) per launch of the
# dominant kernel class, mean over the three layers of the 1.5B-scale workload,
# from one ncu capture.  "sources" is the hash (kernel_sources_hash) of the
# CUDA sources the capture ran on: when the sources differ, the figure no
# longer describes the kernels and the bench line reports traffic as null.
TRAFFIC_PER_LAUNCH = {3: {"sources": "ca3feec6b354dac5",
                          "capture": "ncu --metrics dram__bytes_read.sum,dram__bytes_write.sum on the weight-gradient "
                                     "launches of the three layers (python bench.py --profile-run --steps 1 "
                                     "--warmup 0), mean per launch",
                          "bytes": {"tc_wgrad": 870.5e6}}}
METRIC = "NOBLE linear fwd+bwd TFLOP/s"
# dense BF16 tensor-core rate of one sm_100-family SM: 8192 FLOP per clock
BF16_FLOP_PER_CLK_SM = 8192


def kernel_sources_hash() -> str:
    """sha256 (first 16 hex digits) over the CUDA sources and the C header."""
    import hashlib
    h = hashlib.sha256()
    csrc = os.path.join(ROOT, "paper_2603_06492_gb300", "csrc")
    files = sorted(os.path.join(csrc, f) for f in os.listdir(csrc) if f.endswith((".cu", ".cuh")))
    files.append(os.path.join(ROOT, "include", "noble.h"))
    for f in files:
        h.update(os.path.basename(f).encode())
        with open(f, "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def config_of(cfg, layers, world, sigma):
    """The bench line's ``config`` (the same object for both arms)."""
    return {"workload": WORKLOADS[cfg], "config_index": cfg, "sigma": sigma, "layers": [
        {"name": l.name, "T": l.T, "d_in": l.d_in, "d_out": l.d_out, "r": l.r} for l in layers],
        "l2": "inputs larger than L2: each step streams ~1.8 GB of activations",
        "parallelism": f"replicas x{world}"}


def peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            p = json.load(f)
        return {"bf16": p["bf16_tflops"], "bf16_sustained": p["bf16_tflops_sustained"],
                "hbm": p["hbm_gbs"], "sm_max_mhz": p.get("sm_max_mhz", 2070.0), "src": "measured"}
    return {"bf16": 1900.0, "bf16_sustained": 1700.0, "hbm": 6800.0, "sm_max_mhz": 2070.0,
            "src": "fallback"}


# ------------------------------------------------------------------ clocks
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "10"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            # the timed region starts only once the sampler is producing lines
            t0 = time.time()
            while not self.lines and self.proc.poll() is None and time.time() - t0 < 5.0:
                time.sleep(0.005)
        except OSError:
            self.proc = None
        self.start = len(self.lines)
        return self

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append(line.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=2)

    def mark(self) -> int:
        """Index of the next sample: brackets a window for summary()."""
        return len(self.lines)

    def summary(self, begin=None, end=None):
        sm, mx, pw, reasons = [], [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        # samples taken inside the timed region (or the window [begin, end));
        # if it was shorter than the sampling interval, the last sample before it
        b = self.start if begin is None else begin
        e = len(self.lines) if end is None else end
        region = self.lines[b:e] or self.lines[max(b - 1, 0):b] or self.lines[-1:]
        for ln in region:
            f = [x.strip() for x in ln.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            try:
                pw.append(float(f[3]))
            except ValueError:
                pass
            for n, v in zip(names, f[5:9]):
                if v.lower() in ("active", "1", "0x1"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
                "power_w": statistics.median(pw) if pw else None,
                "samples": len(sm), "samples_in_timed_region": len(self.lines[b:e])}


# ------------------------------------------------------------------ oracle arm
def oracle_sample(layers, tokens: int, seed: int = 0, sigma: str = "cosnet"):
    """The fp64 oracle's fwd+bwd, with the bottleneck variant ``sigma``, on the
    first ``tokens`` tokens of each layer (same shapes and distributions).
    Returns (seconds, flops)."""
    import oracle
    from paper_2603_06492_gb300.inputs import Layer, to_paper_orientation
    t_total, flops = 0.0, 0.0
    for li, layer in enumerate(layers):
        sl = Layer(layer.name, tokens, layer.d_in, layer.d_out, layer.r, layer.dtype)
        p = to_paper_orientation(make_layer_inputs(sl, seed + li))
        if sigma == "cos3":
            p.update(make_cos3_inputs(sl.r, seed + li + 1))
        t0 = time.perf_counter()
        if sigma == "cos3":
            oracle.fwd3(p["x"], p["W"], p["bias"], p)
            oracle.bwd3(p["x"], p["W"], p, p["dy"])
        else:
            mode = oracle.MODES[sigma]
            oracle.fwd(p["x"], p["W"], p["bias"], p["W_down"], p["omega1"], p["phi1"], p["M"],
                       p["omega2"], p["phi2"], p["W_up"], mode=mode)
            oracle.bwd(p["x"], p["W"], p["W_down"], p["omega1"], p["phi1"], p["M"], p["omega2"],
                       p["phi2"], p["W_up"], p["dy"], mode=mode)
        t_total += time.perf_counter() - t0
        flops += sl.flops()
    return t_total, flops


def host_cores():
    n = os.environ.get("OMP_NUM_THREADS")
    return int(n) if n else len(os.sched_getaffinity(0))


def select_workload(args):
    """(key, seed key, layers) of the workload the flags name: a numbered
    configuration, or one of the paper's GeGLU FFN shapes (--workload)."""
    if args.workload:
        return args.workload, PAPER_WORKLOAD_SEED[args.workload], PAPER_WORKLOADS[args.workload]
    return args.config, args.config, CONFIGS[args.config]


def run_reference(args, rank):
    """--impl reference: the oracle as it stands, on host cores, rank 0 only."""
    if rank != 0:
        return
    cfg, _, layers = select_workload(args)
    import oracle
    oracle.build()
    for _ in range(args.warmup):
        oracle_sample(layers, args.ref_tokens, sigma=args.sigma)
    secs, flops = 0.0, 0.0
    for s in range(args.steps):
        t, f = oracle_sample(layers, args.ref_tokens, seed=100 + s, sigma=args.sigma)
        secs += t
        flops += f
    v = flops / secs / 1e12
    sample = (f"first {args.ref_tokens} of {layers[0].T} tokens of each of the {len(layers)} layers "
              f"per step (fwd+bwd, fp64)")
    line = {"impl": "reference", "metric": METRIC, "value": v, "unit": "TFLOP/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": secs / args.steps * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_of(cfg, layers, args.gpus, args.sigma),
            "cpu_baseline": {"value": v, "unit": "TFLOP/s", "cores": host_cores(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": "TFLOP/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ------------------------------------------------------------------ ranks
def max_over_ranks(ms: float, dist, device: str = "cuda") -> float:
    """The job's time for a timed region: the slowest rank's (each rank's
    region ends at its own last event).  ``dist`` is torch.distributed or
    None for one process."""
    if dist is None:
        return ms
    import torch
    t = torch.tensor([ms], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, flops_per_rank_step: float, ms_per_step: float) -> float:
    """Whole-job TFLOP/s: every rank processes its own batch of the same
    shape (weak scaling, replicas), so the work is world times one rank's."""
    return world * flops_per_rank_step / (ms_per_step * 1e-3) / 1e12


# ------------------------------------------------------------------ GPU arm
def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=20)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="own", choices=["own", "reference"])
    ap.add_argument("--cpu-tokens", type=int, default=768,
                    help="tokens per layer in the oracle's bounded sample (cpu_baseline)")
    ap.add_argument("--ref-tokens", type=int, default=64,
                    help="tokens per layer in each step of --impl reference")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--profile-run", action="store_true",
                    help="fwd+bwd of the selected layers only, for ncu; prints no bench line")
    ap.add_argument("--profile-optimizer", action="store_true",
                    help="with --profile-run: also one optimizer step over the layers' parameters")
    ap.add_argument("--layers", default="", help="comma-separated layer names (default: all)")
    ap.add_argument("--config", type=int, default=CONFIG_INDEX,
                    help="workload: configuration 0-4 (default 3, the headline)")
    ap.add_argument("--workload", default="", choices=["", "geglu-base", "geglu-large"],
                    help="the paper's GeGLU FFN shapes instead of a numbered configuration")
    ap.add_argument("--sigma", default="cosnet",
                    choices=["cosnet", "cos1", "identity", "tanh1", "tanh2", "leaky1", "leaky2", "gelu1", "gelu2",
                             "cos3"],
                    help="bottleneck activation (the others: variants of the ablation, Section 4.4)")
    ap.add_argument("--fused-branch", action="store_true",
                    help="run the bottleneck inside the output GEMMs (NOBLE_FLAG_FUSED_BRANCH)")
    ap.add_argument("--per-layer", action="store_true",
                    help="also time every layer alone (NOBLE and plain) and report each")
    args = ap.parse_args()

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))
    if args.impl == "reference":
        return run_reference(args, rank)

    import torch
    from paper_2603_06492_gb300 import binding
    from paper_2603_06492_gb300.build import build

    torch.cuda.set_device(local_rank)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local_rank))
    if rank == 0 or world == 1:
        build()
    if dist is not None:
        dist.barrier()
    binding.load()
    assert args.profile_run or args.warmup >= 3, "at least 3 warm-up steps"

    cfg, seed_cfg, all_layers = select_workload(args)
    layers = all_layers
    if args.layers:
        keep = set(args.layers.split(","))
        layers = [l for l in layers if l.name in keep]
    dev_inputs, bufs, plain_bufs = [], [], []
    for layer in layers:
        li = [l.name for l in all_layers].index(layer.name)
        inp = make_layer_inputs(layer, layer_seed(seed_cfg, li))
        dev_inputs.append(binding.params_to_device(inp, layer.dtype))
        del inp
        sig_flags = binding.SIGMA_FLAGS[args.sigma] if args.sigma != "cos3" else binding.NOBLE_FLAG_SIGMA_COS3
        if args.sigma == "cos3":
            # the three-layer cosine's second mixing matrix and third frequency / phase
            dev_inputs[-1].update(binding.params_to_device(make_cos3_inputs(layer.r, layer_seed(seed_cfg, li) + 1),
                                                           layer.dtype))
        if args.fused_branch:
            sig_flags |= binding.NOBLE_FLAG_FUSED_BRANCH
        bufs.append(binding.NobleLinearBuffers(layer.T, layer.d_in, layer.d_out, layer.r, layer.dtype,
                                               flags=sig_flags))
        plain_bufs.append(binding.NobleLinearBuffers(layer.T, layer.d_in, layer.d_out, 0, layer.dtype))
    flops_step = sum(l.flops() for l in layers)
    flops_plain = sum(l.plain().flops() for l in layers)
    stream = torch.cuda.current_stream()

    def step(bset, plain=False):
        for d, b in zip(dev_inputs, bset):
            p = {k: d[k] for k in ("W", "bias")} if plain else d
            binding.forward(b, d["x"], p, stream)
            binding.backward(b, d["x"], d["dy"], p, stream)

    def timed(fn, k):
        if dist is not None:
            dist.barrier()
        torch.cuda.synchronize()
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(k):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return max_over_ranks(e0.elapsed_time(e1), dist)

    # optimizer step over the layers' parameters (fused AdamW with NOBLE's
    # per-group learning rates; fp32 masters and moments, bf16 operand copies
    # of W, W_down and W_up): HBM-bound, reported against the copy bandwidth
    def optimizer_tensors():
        opt_tensors, opt_bytes = [], 0.0
        for layer, d, b in zip(layers, dev_inputs, bufs):
            mult = binding.noble_linear_lr_multipliers(b.desc) if layer.r > 0 else [1.0] * 5
            groups = [("W", "dW", mult[0], True, True), ("bias", "dbias", mult[0], False, False)]
            if layer.r > 0:
                groups += [("W_down", "dW_down", mult[0], True, True), ("W_up", "dW_up", mult[1], True, True),
                           ("M", "dM", mult[2], True, False), ("omega1", "domega1", mult[3], False, False),
                           ("omega2", "domega2", mult[3], False, False), ("phi1", "dphi1", mult[4], False, False),
                           ("phi2", "dphi2", mult[4], False, False)]
            for name, gname, k, decay, lowp in groups:
                g = b.grads[gname].reshape(-1)
                n = g.numel()
                opt_tensors.append({"param": d[name].float().reshape(-1).clone(), "grad": g,
                                    "exp_avg": torch.zeros(n, device="cuda"), "exp_avg_sq": torch.zeros(n, device="cuda"),
                                    "param_bf16": torch.empty(n, dtype=torch.bfloat16, device="cuda") if lowp else None,
                                    "lr_mult": k, "decay": decay})
                opt_bytes += (28.0 + (2.0 if lowp else 0.0)) * n
        return opt_tensors, opt_bytes

    if args.profile_run:
        for _ in range(args.warmup + args.steps):
            step(bufs)
        if args.profile_optimizer:
            ts, _ = optimizer_tensors()
            binding.noble_adamw_step(ts, lr=3e-4, weight_decay=0.01, step=1)
        torch.cuda.synchronize()
        binding.noble_get_device_status(None)
        print("profile run done", flush=True)
        return

    # warm-up (NOBLE and plain)
    for _ in range(args.warmup):
        step(bufs)
        step(plain_bufs, plain=True)
    torch.cuda.synchronize()
    binding.noble_get_device_status(None)

    # timed: NOBLE steps back to back (the headline), then the same steps
    # again with per-kernel CUDA events around every launch (kernel breakdown
    # and roofline entry; the events separate the launches, so this second
    # run is not the headline)
    lib = binding.load()
    n0 = binding.noble_kernel_launch_count()
    with ClockSampler(local_rank) as clk:
        ms = timed(lambda: step(bufs), args.steps)
    launches = binding.noble_kernel_launch_count() - n0
    lib.noble_profile_reset()
    lib.noble_profile_enable(1)
    ms_profiled = timed(lambda: step(bufs), args.steps)
    lib.noble_profile_enable(0)
    prof = binding.profile_read()

    # overhead against the plain (r = 0) layer of this library, in the two
    # clock regimes of a GB300 under this load:
    #  * burst (the reported overhead): NOBLE and plain runs of the timed steps
    #    alternate five times, each after an idle second, so that both arms run
    #    at the maximum SM clock as the headline steps do (a run that follows
    #    another at once starts under the power cap the first one raised);
    #    medians compared, each run's clock sampled, and a clock-normalised
    #    overhead (time x median SM clock, i.e. SM cycles) given beside it;
    #  * sustained: blocks of back-to-back runs per arm (NOBLE, plain, NOBLE,
    #    plain) long enough to settle under the power cap, the median of each
    #    block's later runs, with that block's clock
    reps_n, reps_p, clk_n, clk_p = [], [], [], []
    sustained = {"noble": [], "plain": [], "noble_mhz": [], "plain_mhz": []}
    with ClockSampler(local_rank) as clk_ovh:
        for _ in range(5):
            for arm, reps, clks in ((False, reps_n, clk_n), (True, reps_p, clk_p)):
                time.sleep(1.0)
                m0 = clk_ovh.mark()
                reps.append(timed(lambda: step(plain_bufs if arm else bufs, plain=arm), args.steps))
                clks.append(clk_ovh.summary(m0, clk_ovh.mark()))
        sus_k = max(1, args.steps // 2)
        for _ in range(2):
            for arm in (False, True):
                key = "plain" if arm else "noble"
                ts, m_begin = [], None
                for i in range(40):
                    if i == 25:
                        m_begin = clk_ovh.mark()
                    t = timed(lambda: step(plain_bufs if arm else bufs, plain=arm), sus_k) / sus_k
                    if i >= 25:
                        ts.append(t)
                sustained[key].append(statistics.median(ts))
                sustained[key + "_mhz"].append(clk_ovh.summary(m_begin, clk_ovh.mark()).get("sm_mhz"))
    ms_noble_med, ms_plain = statistics.median(reps_n), statistics.median(reps_p)
    sus_n, sus_p = statistics.median(sustained["noble"]), statistics.median(sustained["plain"])
    mhz_n = [m for m in sustained["noble_mhz"] if m]
    mhz_p = [m for m in sustained["plain_mhz"] if m]
    overhead_sustained = {
        "noble_ms_per_step": sus_n, "plain_ms_per_step": sus_p, "overhead": sus_n / sus_p - 1.0,
        "noble_sm_mhz": statistics.median(mhz_n) if mhz_n else None,
        "plain_sm_mhz": statistics.median(mhz_p) if mhz_p else None,
        "overhead_clock_normalised": (sus_n * statistics.median(mhz_n) / (sus_p * statistics.median(mhz_p)) - 1.0)
        if mhz_n and mhz_p else None,
        "method": "2 blocks per arm of 40 back-to-back runs of steps/2 steps; median of runs 26-40"}

    def med_mhz(clks):
        v = [c["sm_mhz"] for c in clks if c.get("sm_mhz")]
        return statistics.median(v) if v else None

    def cycles(reps, clks):
        v = [t * c["sm_mhz"] for t, c in zip(reps, clks) if c.get("sm_mhz")]
        return statistics.median(v) if v else None

    cyc_n, cyc_p = cycles(reps_n, clk_n), cycles(reps_p, clk_p)

    # forward and backward passes timed apart
    def fwd_only(bset, plain=False):
        for d, b in zip(dev_inputs, bset):
            binding.forward(b, d["x"], {k: d[k] for k in ("W", "bias")} if plain else d, stream)

    def bwd_only(bset, plain=False):
        for d, b in zip(dev_inputs, bset):
            binding.backward(b, d["x"], d["dy"], {k: d[k] for k in ("W", "bias")} if plain else d, stream)

    # inference forward (NOBLE_FLAG_INFERENCE: h and b not saved)
    inf_bufs = [binding.NobleLinearBuffers(l.T, l.d_in, l.d_out, l.r, l.dtype, with_grads=False,
                                           flags=binding.NOBLE_FLAG_INFERENCE | b.desc.flags)
                for l, b in zip(layers, bufs)]
    fwd_only(inf_bufs)
    # each run after an idle second, so that every run starts at the maximum
    # clock like the headline (back to back, the later runs would meet the
    # power cap and the NOBLE / plain ratios would compare two clocks);
    # NOBLE and plain alternate, three runs each, medians
    passes = {"fwd": lambda: fwd_only(bufs), "fwd_p": lambda: fwd_only(plain_bufs, True),
              "bwd": lambda: bwd_only(bufs), "bwd_p": lambda: bwd_only(plain_bufs, True),
              "fwd_inf": lambda: fwd_only(inf_bufs)}
    sep = {k: [] for k in passes}
    for _ in range(3):
        for k, fn in passes.items():
            time.sleep(1.0)
            sep[k].append(timed(fn, args.steps))
    del inf_bufs
    ms_fwd, ms_bwd, ms_fwd_p, ms_bwd_p, ms_fwd_inf = (statistics.median(sep[k])
                                                      for k in ("fwd", "bwd", "fwd_p", "bwd_p", "fwd_inf"))
    binding.noble_get_device_status(None)

    ms_step = ms / args.steps
    value = job_throughput(world, flops_step, ms_step)
    pk = peaks()
    clk_main = clk.summary()
    n_sm = torch.cuda.get_device_properties(local_rank).multi_processor_count

    def hw_peak(mhz):
        return n_sm * BF16_FLOP_PER_CLK_SM * mhz * 1e6 / 1e12

    # dominant kernel: largest share of summed kernel time (profiled run)
    roof = None
    if prof:
        top = max(prof.values(), key=lambda e: e["ms"])
        achieved = top["flops"] / (top["ms"] / top["launches"] * 1e-3) / top["launches"] / 1e12 \
            if top["bound"] == "tensor" else top["bytes"] / (top["ms"] / top["launches"] * 1e-3) / top["launches"] / 1e9
        if top["bound"] == "tensor":
            # the timed region is tens of milliseconds at full clock (see
            # "clocks"), so the burst figure is the denominator
            peak, unit = pk["bf16"], "TFLOP/s"
        elif top["bound"] == "hbm":
            peak, unit = pk["hbm"], "GB/s"
        else:  # fp32 FMA pipe: 152 SMs x 128 lanes x 2 FLOP x max SM clock
            peak, unit = 152 * 128 * 2 * pk["sm_max_mhz"] * 1e6 / 1e12, "TFLOP/s"
        cap = TRAFFIC_PER_LAUNCH.get(cfg, {})
        fresh = bool(cap.get("sources")) and cap.get("sources") == kernel_sources_hash() and not args.layers
        traffic = cap.get("bytes", {}).get(top["name"]) if fresh else None
        roof = {"bound": top["bound"], "kernel": top["name"], "achieved": achieved, "peak": peak,
                "unit": unit, "frac": achieved / peak,
                "traffic": traffic,
                "traffic_src": (cap.get("capture") if traffic is not None else
                                "no ncu capture of the kernels as built (sources hash " + kernel_sources_hash() + ")"),
                "algorithmic_bytes": top["bytes"] / top["launches"],
                "peak_src": ("measured burst" if top["bound"] == "tensor" else
                             "measured" if top["bound"] == "hbm" else "derived from unit counts"),
                "frac_of_sustained": (achieved / pk["bf16_sustained"]) if top["bound"] == "tensor" else None,
                "share_of_step": top["ms"] / ms_profiled, "launches_per_step": top["launches"] / args.steps}

    # end to end through the C ABI: every step copies x, dy of each layer from
    # pinned host memory and y, dx back, inside the timed region.  Copies run
    # on their own streams and overlap the compute of other layers and of the
    # neighbouring step (device inputs and outputs are double-buffered).
    e2e = None
    if not args.no_e2e and args.sigma == "cos3":
        e2e = {"value": None, "note": "not measured for the three-layer cosine (its own entry points)"}
    elif not args.no_e2e:
        h2d_s, d2h_s = torch.cuda.Stream(), torch.cuda.Stream()
        host, sets, h2d, d2h = [], [], 0, 0
        for d, b in zip(dev_inputs, bufs):
            hx, hdy = d["x"].cpu().pin_memory(), d["dy"].cpu().pin_memory()
            hy = torch.empty(tuple(b.y.shape), dtype=b.y.dtype).pin_memory()
            hdx = torch.empty(tuple(b.dx.shape), dtype=b.dx.dtype).pin_memory()
            host.append((hx, hdy, hy, hdx))
            h2d += hx.numel() * hx.element_size() + hdy.numel() * hdy.element_size()
            d2h += hy.numel() * hy.element_size() + hdx.numel() * hdx.element_size()
        for _ in range(2):
            sets.append([{"x": torch.empty_like(d["x"]), "dy": torch.empty_like(d["dy"]),
                          "y": torch.empty_like(b.y), "dx": torch.empty_like(b.dx)}
                         for d, b in zip(dev_inputs, bufs)])
        free_in = [[None] * len(bufs) for _ in range(2)]   # compute done with inputs
        free_out = [[None] * len(bufs) for _ in range(2)]  # host read done with outputs
        counter = [0]
        sh = stream.cuda_stream

        def e2e_step():
            k = counter[0]
            counter[0] += 1
            for li, (d, b) in enumerate(zip(dev_inputs, bufs)):
                io, (hx, hdy, hy, hdx) = sets[k % 2][li], host[li]
                if free_in[k % 2][li] is not None:
                    h2d_s.wait_event(free_in[k % 2][li])
                with torch.cuda.stream(h2d_s):
                    io["x"].copy_(hx, non_blocking=True)
                    io["dy"].copy_(hdy, non_blocking=True)
                ev_in = torch.cuda.Event()
                ev_in.record(h2d_s)
                stream.wait_event(ev_in)
                if free_out[k % 2][li] is not None:
                    stream.wait_event(free_out[k % 2][li])
                p, g = d, b.grads
                binding.noble_linear_fwd(b.desc, io["x"], p["W"], p.get("bias"), p.get("W_down"),
                                         p.get("omega1"), p.get("phi1"), p.get("M"), p.get("omega2"),
                                         p.get("phi2"), p.get("W_up"), io["y"], b.saved, b.saved_bytes, sh)
                binding.noble_linear_bwd(b.desc, io["dy"], io["x"], p["W"], p.get("W_down"),
                                         p.get("omega1"), p.get("phi1"), p.get("M"), p.get("omega2"),
                                         p.get("phi2"), p.get("W_up"), b.saved, b.saved_bytes, io["dx"],
                                         g["dW"], g["dbias"], g.get("dW_down"), g.get("dM"),
                                         g.get("domega1"), g.get("dphi1"), g.get("domega2"),
                                         g.get("dphi2"), g.get("dW_up"), b.workspace,
                                         b.workspace_bytes, sh)
                ev_c = torch.cuda.Event()
                ev_c.record(stream)
                free_in[k % 2][li] = ev_c
                d2h_s.wait_event(ev_c)
                with torch.cuda.stream(d2h_s):
                    hy.copy_(io["y"], non_blocking=True)
                    hdx.copy_(io["dx"], non_blocking=True)
                ev_o = torch.cuda.Event()
                ev_o.record(d2h_s)
                free_out[k % 2][li] = ev_o

        def timed_e2e(k):
            if dist is not None:
                dist.barrier()
            torch.cuda.synchronize()
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            h2d_s.wait_event(e0)
            for _ in range(k):
                e2e_step()
            stream.wait_stream(d2h_s)
            e1.record(stream)
            torch.cuda.synchronize()
            return max_over_ranks(e0.elapsed_time(e1), dist)

        for _ in range(2):
            e2e_step()
        ms_e2e = timed_e2e(args.steps) / args.steps
        e2e = {"value": world * flops_step / (ms_e2e * 1e-3) / 1e12, "unit": "TFLOP/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "ms_per_step": ms_e2e,
               "copies": "pinned host buffers, copy streams overlapping compute"}

    adamw = None
    opt_tensors, opt_bytes = optimizer_tensors()
    opt_step = [0]

    def adamw_step():
        opt_step[0] += 1
        binding.noble_adamw_step(opt_tensors, lr=3e-4, weight_decay=0.01, step=opt_step[0])

    for _ in range(args.warmup):
        adamw_step()
    ms_adamw = timed(adamw_step, args.steps) / args.steps
    binding.noble_get_device_status(None)
    adamw = {"ms_per_step": ms_adamw, "bytes_per_step": opt_bytes,
             "achieved_gbs": opt_bytes / (ms_adamw * 1e-3) / 1e9, "peak_gbs": pk["hbm"],
             "frac": opt_bytes / (ms_adamw * 1e-3) / 1e9 / pk["hbm"],
             "params": sum(t["param"].numel() for t in opt_tensors),
             "note": "not part of the fwd+bwd step; lr 3e-4, betas (0.9, 0.98), weight decay 0.01"}
    del opt_tensors

    per_layer = None
    if args.per_layer:
        per_layer = {}
        for li, layer in enumerate(layers):
            d, b, bp = dev_inputs[li], bufs[li], plain_bufs[li]

            def one(plain=False, d=d, b=b, bp=bp):
                p = {k: d[k] for k in ("W", "bias")} if plain else d
                bb = bp if plain else b
                binding.forward(bb, d["x"], p, stream)
                binding.backward(bb, d["x"], d["dy"], p, stream)

            for _ in range(2):
                one()
                one(True)
            t_n = timed(one, args.steps) / args.steps
            t_p = timed(lambda: one(True), args.steps) / args.steps
            per_layer[layer.name] = {
                "ms": t_n, "tflops": world * layer.flops() / (t_n * 1e-3) / 1e12,
                "plain_ms": t_p, "plain_tflops": world * layer.plain().flops() / (t_p * 1e-3) / 1e12,
                "overhead_vs_plain": t_n / t_p - 1.0}

    # data parallel over N ranks (only under torchrun with N > 1): the same step
    # followed by the sum-all-reduce of every layer's gradient bucket, each
    # started as soon as that layer's backward is enqueued (NCCL overlaps it
    # with the next layer); and the all-reduces alone.  The headline above is
    # the replica step; these two report what the exchange adds.
    dp = None
    if dist is not None:
        from paper_2603_06492_gb300.dp import GradAllReduce
        ar = GradAllReduce()

        def dp_step():
            for d, b in zip(dev_inputs, bufs):
                binding.forward(b, d["x"], d, stream)
                binding.backward(b, d["x"], d["dy"], d, stream)
                ar.launch(b.bucket)
            ar.wait()

        def allreduce_only():
            for b in bufs:
                ar.launch(b.bucket)
            ar.wait()

        dp_step()
        ms_dp = timed(dp_step, args.steps) / args.steps
        ms_ar = timed(allreduce_only, args.steps) / args.steps
        dp = {"step_ms": ms_dp, "allreduce_ms_per_step": ms_ar,
              "bucket_bytes_per_step": sum(b.layout["total_bytes"] for b in bufs),
              "tflops": job_throughput(world, flops_step, ms_dp),
              "note": "tokens sharded over ranks; one sum-all-reduce per layer's gradient bucket (NCCL)"}

    # cuBLAS reference timing of the plain layer (torch.matmul x3), context only
    def cublas_step():
        for d in dev_inputs:
            y = torch.matmul(d["x"], d["W"].t())
            torch.matmul(d["dy"], d["W"])
            torch.matmul(d["dy"].t(), d["x"])
            del y
    for _ in range(3):
        cublas_step()
    ms_cublas = timed(cublas_step, args.steps) / args.steps

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        secs, fl = oracle_sample(layers, args.cpu_tokens, sigma=args.sigma)
        cpu = {"value": fl / secs / 1e12, "unit": "TFLOP/s", "cores": host_cores(), "kind": "oracle",
               "sample": f"fwd+bwd of the first {args.cpu_tokens} of {layers[0].T} tokens of each layer, fp64",
               "seconds": secs}

    if rank == 0:
        line = {
            "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms_step,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None,
            "dtype": "bf16" if layers[0].dtype == "bf16" else "f32",
            "data": "synthetic",
            "config": config_of(cfg, layers, world, args.sigma),
            # dense BF16 tensor peak of the GPU: SMs x 8192 FLOP/clk x SM clock,
            # at the median clock sampled in the timed region and at the maximum
            "pct_peak_bf16": value / world / hw_peak(clk_main.get("sm_mhz") or pk["sm_max_mhz"]),
            "pct_peak_bf16_at_max_clock": value / world / hw_peak(pk["sm_max_mhz"]),
            "peak_bf16_tflops": {"at_sampled_clock": hw_peak(clk_main.get("sm_mhz") or pk["sm_max_mhz"]),
                                 "at_max_clock": hw_peak(pk["sm_max_mhz"]), "sms": n_sm,
                                 "flop_per_clk_sm": BF16_FLOP_PER_CLK_SM},
            # against the best measured cuBLAS bf16 GEMM rate (8192^3), burst and sustained
            "vs_cublas_best": value / world / pk["bf16"],
            "vs_cublas_best_sustained": value / world / pk["bf16_sustained"],
            "peak_src": pk["src"],
            "plain_ms_per_step": ms_plain / args.steps,
            "plain_tflops": world * flops_plain / (ms_plain / args.steps * 1e-3) / 1e12,
            "overhead_vs_plain": ms_noble_med / ms_plain - 1.0,
            "overhead_method": "median of 5 alternating NOBLE / plain runs of the timed steps, each after an "
                               "idle second (both arms at the maximum SM clock, as the headline)",
            "overhead_sustained": overhead_sustained,
            "overhead_reps_ms_per_step": {"noble": [round(v / args.steps, 4) for v in reps_n],
                                          "plain": [round(v / args.steps, 4) for v in reps_p]},
            "overhead_clock_normalised": (cyc_n / cyc_p - 1.0) if cyc_n and cyc_p else None,
            "overhead_clock_method": "median over runs of time x median SM clock of the run (SM cycles)",
            "overhead_clocks": {"noble": {"sm_mhz_median": med_mhz(clk_n),
                                          "reasons": sorted({x for c in clk_n for x in c["reasons"]})},
                                "plain": {"sm_mhz_median": med_mhz(clk_p),
                                          "reasons": sorted({x for c in clk_p for x in c["reasons"]})},
                                "all": clk_ovh.summary()},
            "fwd_ms_per_step": ms_fwd / args.steps, "bwd_ms_per_step": ms_bwd / args.steps,
            "plain_fwd_ms_per_step": ms_fwd_p / args.steps, "plain_bwd_ms_per_step": ms_bwd_p / args.steps,
            "overhead_fwd": ms_fwd / ms_fwd_p - 1.0, "overhead_bwd": ms_bwd / ms_bwd_p - 1.0,
            "fwd_inference_ms_per_step": ms_fwd_inf / args.steps,
            "overhead_fwd_inference": ms_fwd_inf / ms_fwd_p - 1.0,
            "cublas_plain_ms_per_step": ms_cublas,
            "overhead_vs_cublas_plain": ms_noble_med / args.steps / ms_cublas - 1.0,
            "roofline": roof, "cpu_baseline": cpu, "e2e": e2e, "per_layer": per_layer,
            "gpu_launches": launches,
            "data_parallel": dp,
            "profiled_ms_per_step": ms_profiled / args.steps,
            "optimizer_step": adamw,
            "kernel_breakdown": {k: {"ms_per_step": v["ms"] / args.steps,
                                     "launches_per_step": v["launches"] / args.steps}
                                 for k, v in sorted(prof.items(), key=lambda kv: -kv[1]["ms"])},
            "clocks": clk_main,
        }
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.barrier()
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
