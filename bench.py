"""Throughput of the fused log-prob forward + MirrorPop filter + backward.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

One step = one pass of the whole hot path over one batch of the 9B-class
fused forward+backward workload (32 sequences of U[512, 8192] tokens, d = 4096,
V = 248320, bf16; seeded synthetic inputs, see paper_2606_04847_gb300/workloads.py):
  1. mc_token_logprobs      policy log-probs, entropies, log-sum-exp
  2. mc_seq_ratio_filter    per-sequence ratio statistics + MirrorPop keep-mask
  3. mc_token_logprobs_bwd  grad_hidden, grad_w for advantage weights on the
                            kept tokens (row_keep = the filter's token_keep)
The behaviour log-probs are the policy's plus a per-sequence N(0, 0.2^2) gap,
formed once before timing (the rollout engine's job, not part of the step).

Rank 0 prints one JSON line. ``value`` = tokens/s over all ranks with inputs
resident in HBM; ``e2e`` = the same through the C ABI with the step's inputs
copied from pinned host memory and its per-token / per-sequence results read
back inside the timed region (the gradients stay on the device for the rest of
the backward and the optimizer). Inputs (hidden 1.1 GB, W 2.0 GB) exceed the
129 MB L2, so no flush is needed between steps. ``--impl reference`` times the
CPU fp64 oracle instead, on a bounded sample of the same workload.

Multi-GPU (torchrun): one rank per GPU, each on its own batch (weak scaling).
Forward, filter and grad_hidden need no exchange; for the forward + backward
step, grad_w (each rank's gradient over its own batch) is all-reduced over
the ranks with NCCL inside the timed step, as data parallelism requires.
"""

from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import torch  # noqa: E402

METRIC = "rollout tokens/sec for fused logprob fwd+bwd at 1 GB300; % of bf16 tensor peak"
METRIC_FWD = "rollout tokens/sec for fused logprob fwd + MirrorPop filter at 1 GB300; % of bf16 tensor peak"
CONFIG_ID = 5  # the fused forward+backward workload the metric names (the default of --config)
FWD_TRAFFIC_FILE = os.path.join(ROOT, "profiles", "fwd_kernel_traffic.json")
BWD_TRAFFIC_FILE = os.path.join(ROOT, "profiles", "bwd_kernels_traffic.json")


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return {"hbm_gbs": d["hbm_gbs"], "bf16": d["bf16_tflops"], "bf16_sustained": d["bf16_tflops_sustained"],
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16": 1900.0, "bf16_sustained": 1700.0, "source": "fallback"}


FWD_SOURCES = ("mc_gemm.cuh", "mc_ptx.cuh", "mc_fwd.cu", "mc_schedule.h")  # the forward kernel and its schedule
BWD_SOURCES = ("mc_gemm.cuh", "mc_ptx.cuh", "mc_bwd.cu", "mc_schedule.h")  # the backward's kernels and schedule


def _kernel_source_hash(files=FWD_SOURCES):
    """Hash of a kernel's and its schedule's code, comments and whitespace
    removed (so that edits to comments keep a capture valid)."""
    import re

    h = hashlib.sha256()
    for f in files:
        src = open(os.path.join(ROOT, "paper_2606_04847_gb300", "csrc", f)).read()
        src = re.sub(r"/\*.*?\*/", " ", src, flags=re.S)
        src = re.sub(r"//[^\n]*", " ", src)
        h.update(" ".join(src.split()).encode())
    return h.hexdigest()[:16]


class ClockSampler:
    """nvidia-smi clocks/throttle reasons sampled every 200 ms while running."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = os.path.join("/tmp", f"mc_clocks_{os.getpid()}.csv")

    def start(self):
        try:
            self.fh = open(self.path, "w")
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=self.fh, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        sm, smax, power, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [x.strip() for x in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                smax.append(float(parts[2]))
                power.append(float(parts[3]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None, "sm_max_mhz": max(smax) if smax else None,
                "power_w_max": max(power) if power else None, "samples": len(sm), "reasons": sorted(reasons)}


def _dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist

        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    else:
        torch.cuda.set_device(0)
    return world, rank, local


def _barrier(world):
    if world > 1:
        import torch.distributed as dist

        dist.barrier()


def _reduce(x, world, op, device="cuda"):
    """x reduced over ranks (op = "max" | "sum"); identity for one rank."""
    if world == 1:
        return float(x)
    import torch.distributed as dist

    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX if op == "max" else dist.ReduceOp.SUM)
    return float(t.item())


def aggregate(tokens_local, ms_local, world, device="cuda"):
    """Whole-job throughput of independent replicas: tokens summed over ranks
    divided by the slowest rank's time (weak scaling). Returns
    (tokens_total, ms_max, tokens_per_second)."""
    tokens_total = _reduce(tokens_local, world, "sum", device)
    ms_max = _reduce(ms_local, world, "max", device)
    return tokens_total, ms_max, tokens_total / (ms_max / 1e3)


def _max_over_ranks(x, world):
    return _reduce(x, world, "max")


def dp_grad_w_allreduce(grad_w, world):
    """The backward's one data-parallel exchange: each rank's grad_w [V, d] is
    the gradient of its own batch; a DP trainer needs their sum before the
    optimizer step, so every rank ends with the sum over ranks (NCCL on GPUs).
    Forward, filter, loss and grad_hidden are per-sequence / per-row and need
    no exchange. One rank: nothing to do."""
    if world > 1:
        import torch.distributed as dist

        dist.all_reduce(grad_w, op=dist.ReduceOp.SUM)
    return grad_w


# --------------------------------------------------------------------------- CPU oracle leg


def oracle_sample_step(wl, rows, delta):
    """The fp64 oracle over the first `rows` packed tokens of the workload:
    forward, filter (those tokens as one sequence), backward with the kept
    advantage weights. Returns elapsed seconds."""
    import numpy as np

    import oracle

    h = wl.hidden[:rows].cpu()
    w = wl.w_vocab.cpu() if wl.w_vocab.is_cuda else wl.w_vocab
    y = wl.targets[:rows].cpu()
    adv = None if wl.advantages is None else wl.advantages[:rows].cpu().double().numpy()
    gap = wl.gap[:rows].cpu().double().numpy()
    t0 = time.perf_counter()
    fw = oracle.token_logprobs(h, w, y, 1.0)
    flt = oracle.seq_ratio_filter(fw["logp"], fw["logp"] + gap, None, np.array([0, rows]), delta, delta)
    if adv is not None:  # the forward-only configurations have no backward
        g = adv * flt["token_keep"]
        oracle.token_logprobs_bwd(h, w, y, g, None, 1.0)
    return time.perf_counter() - t0


def _l2_persisting_limit():
    """Read-only: the L2 set-aside for persisting accesses that this context
    sees (cudaDeviceGetLimit; None when the runtime cannot be found). Part of
    the L2 is then unavailable to ordinary accesses, which changes the
    forward's DRAM traffic (W re-reads per wave) though not its speed."""
    import ctypes
    import glob

    for path in (glob.glob(os.path.join(os.path.dirname(torch.__file__), "lib", "libcudart.so*")) +
                 glob.glob("/usr/local/cuda/lib64/libcudart.so*")):
        try:
            rt = ctypes.CDLL(path)
            v = ctypes.c_size_t(0)
            if rt.cudaDeviceGetLimit(ctypes.byref(v), 6) == 0:  # cudaLimitPersistingL2CacheSize
                return int(v.value)
        except OSError:
            continue
    return None


def _blas():
    """BLAS library NumPy was built against, and its thread count (the oracle's matmuls)."""
    import numpy as np

    name = "unknown"
    try:
        name = np.__config__.CONFIG["Build Dependencies"]["blas"]["name"]
    except (AttributeError, KeyError, TypeError):
        pass
    threads = os.environ.get("OPENBLAS_NUM_THREADS") or os.environ.get("OMP_NUM_THREADS") or str(_cores())
    return f"{name}, {threads} threads"


def _cores():
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


# --------------------------------------------------------------------------- main


def run_ours(args):
    from paper_2606_04847_gb300 import build as mcbuild
    from paper_2606_04847_gb300 import mc, workloads

    world, rank, local = _dist_setup(args)
    if not os.path.exists(mc.lib_path()):
        mcbuild.build()
    spec = workloads.spec_for(args.config)
    if world > 1:
        spec = workloads.spec_for(args.config, seed=spec.seed + 1000 * rank)  # each replica its own batch
    wl = workloads.build(spec, "cuda")
    dev = torch.device("cuda")
    N, d, V, B = wl.N, spec.d, spec.V, wl.B
    delta = spec.delta
    h, w, y = wl.hidden, wl.w_vocab, wl.targets
    cu, mask, adv = wl.cu_seqlens, wl.loss_mask, wl.advantages
    has_bwd = adv is not None  # the forward-only configurations time forward + filter

    # Behaviour log-probs: policy log-probs + the per-sequence gap (untimed).
    pre = mc.token_logprobs(h, w, y)
    logp_b = (pre["logp"] + wl.gap).contiguous()
    del pre

    fw_out = {k: torch.empty(N, dtype=torch.float32, device=dev) for k in ("logp", "entropy", "lse")}
    fw_ws = torch.empty(mc.forward_workspace_size(N, d, V), dtype=torch.uint8, device=dev)
    if has_bwd:
        bw_ws = torch.empty(mc.backward_workspace_size(N, d, V), dtype=torch.uint8, device=dev)
        gh = torch.empty((N, d), dtype=torch.bfloat16, device=dev)
        gw = torch.empty((V, d), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()
    ev = {k: [] for k in ("fwd", "filter", "bwd")}
    resident = (h, y, logp_b, mask, cu, adv)

    # The three calls of a step on stream `s`; returns the filter's outputs.
    def call(part, inputs, s, flt=None):
        hh, yy, lb, mm, cc, aa = inputs
        if part == "fwd":
            mc.token_logprobs(hh, w, yy, out=fw_out, workspace=fw_ws, stream=s)
        elif part == "filter":
            return mc.seq_ratio_filter(fw_out["logp"], lb, mm, cc, delta, delta, stream=s)
        elif has_bwd:
            mc.token_logprobs_bwd(hh, w, yy, fw_out["lse"], fw_out["entropy"], aa, None,
                                  row_keep=flt["token_keep"], grad_hidden=gh, grad_w=gw, workspace=bw_ws,
                                  stream=s)
        return None

    # Launch-bound steps replay each call as a CUDA graph (one set per input
    # buffer set); the kernels are the same, the host launch gaps go away.
    graphs = {}

    def capture(key, inputs):
        gs = {}
        flt = None
        for part in ("fwd", "filter", "bwd"):
            if part == "bwd" and not has_bwd:
                break
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, capture_error_mode="thread_local"):
                r = call(part, inputs, torch.cuda.current_stream(), flt)
            flt = r if part == "filter" else flt
            gs[part] = g
        graphs[key] = (gs, flt)

    def step(record=False, inputs=None, key="resident"):
        inputs = inputs if inputs is not None else resident
        e = [torch.cuda.Event(enable_timing=True) for _ in range(4)] if record else None
        flt = None
        for i, part in enumerate(("fwd", "filter", "bwd")):
            if record:
                e[i].record(stream)
            if key in graphs:
                gs, gflt = graphs[key]
                if part in gs:
                    gs[part].replay()
                flt = gflt
            else:
                r = call(part, inputs, stream, flt)
                flt = r if part == "filter" else flt
        if has_bwd:
            dp_grad_w_allreduce(gw, world)  # never captured: replayed graphs end at the backward
        if record:
            e[3].record(stream)
            ev["fwd"].append((e[0], e[1]))
            ev["filter"].append((e[1], e[2]))
            ev["bwd"].append((e[2], e[3]))
        return flt

    for _ in range(args.warmup):
        flt = step()
    torch.cuda.synchronize()
    # Graphs when a step is launch-bound (auto: under 2 ms of GPU time eagerly).
    probe = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    probe[0].record(stream)
    step()
    probe[1].record(stream)
    torch.cuda.synchronize()
    eager_ms = probe[0].elapsed_time(probe[1])
    use_graph = args.graph == "on" or (args.graph == "auto" and eager_ms < 2.0)
    graph_launches = 0
    if use_graph:
        l_cap = mc.kernel_launches()
        capture("resident", resident)
        graph_launches = mc.kernel_launches() - l_cap  # kernels in one step's graphs (counted at capture)
        for _ in range(args.warmup):
            flt = step()
        torch.cuda.synchronize()
    # Inputs that fit in L2 are evicted before every timed step by a 256 MB
    # write outside the step's events; the step times are then summed.
    flush_buf = torch.empty(256 << 20, dtype=torch.uint8, device=dev) if (N + V) * d * 2 <= 129e6 else None
    kept_rows = int(flt["token_keep"].sum().item())
    n_keep_seq = int(flt["keep"].sum().item())

    clocks = ClockSampler(local)
    clocks.start()
    time.sleep(0.3)
    _barrier(world)
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    l_timed = mc.kernel_launches()
    t_start.record(stream)
    for i in range(args.steps):
        if flush_buf is not None:
            flush_buf.fill_(i & 0xFF)
        step(record=True)
    t_end.record(stream)
    # libmc's own count of the kernels it enqueued in the timed steps; graph
    # replays bypass the library's host code, so there it is the kernels
    # captured into one step's graphs times the steps.
    gpu_launches = graph_launches * args.steps if use_graph else mc.kernel_launches() - l_timed
    torch.cuda.synchronize()
    _barrier(world)
    clk = clocks.stop()
    ms = t_start.elapsed_time(t_end)
    if flush_buf is not None:  # the flushes lie between the steps' events
        ms = sum(a.elapsed_time(b) for (a, _), (_, b) in zip(ev["fwd"], ev["bwd"]))
    tokens_total, ms_max, value = aggregate(float(N) * args.steps, ms, world)

    def avg(k):
        return sum(a.elapsed_time(b) for a, b in ev[k]) / len(ev[k])

    t_fwd, t_flt, t_bwd = avg("fwd"), avg("filter"), avg("bwd") if has_bwd else 0.0
    flop_fwd = 2.0 * N * d * V
    flop_bwd = 4.0 * kept_rows * d * V if has_bwd else 0.0  # algorithmic: rows with a nonzero upstream gradient
    peaks = _peaks()
    # The sustained (power-capped) figure for a kernel whose clocks the power
    # cap held down during the timed region, the burst figure otherwise.
    capped = clk.get("sm_mhz") is None or clk.get("sm_max_mhz") is None or \
        clk["sm_mhz"] < 0.97 * clk["sm_max_mhz"]
    peak_tf = peaks["bf16_sustained"] if capped else peaks["bf16"]
    peak_kind = "sustained" if capped else "burst"
    achieved = flop_fwd / (t_fwd / 1e3) / 1e12
    traffic = None
    if os.path.exists(FWD_TRAFFIC_FILE):
        tj = json.load(open(FWD_TRAFFIC_FILE))
        if tj.get("kernel_source_hash") == _kernel_source_hash() and tj.get("config", 5) == args.config:
            traffic = tj["bytes_per_full_launch"] * (N / tj["full_launch_rows"])
    traffic_bwd = None
    if has_bwd and os.path.exists(BWD_TRAFFIC_FILE):
        tj = json.load(open(BWD_TRAFFIC_FILE))
        if tj.get("kernel_source_hash") == _kernel_source_hash(BWD_SOURCES) and tj.get("config", 5) == args.config:
            traffic_bwd = tj["bytes_per_call"] * (kept_rows / tj["rows"])
    step_tflops = (flop_fwd + flop_bwd) * args.steps / (ms / 1e3) / 1e12

    # ---------------------------------------------------------------- e2e through the C ABI, host buffers
    e2e = None
    if not args.no_e2e:
        # Each step's inputs come from pinned host memory into one of two
        # device buffer sets on a copy stream, so the copy for step i+1
        # overlaps the kernels of step i; the per-token and per-sequence
        # results of every step are read back to pinned host memory. The
        # gradients (grad_hidden bf16 [N, d], grad_w fp32 [V, d]) stay on the
        # device, where the rest of the model's backward and the optimizer
        # take them. All of it, including the first copy, lies inside the
        # timed region.
        host = [t.cpu().pin_memory() for t in (h, y, logp_b, mask, cu, adv if has_bwd else logp_b[:1])]
        dev_in = [[torch.empty_like(t, device=dev) for t in host] for _ in range(2)]
        h2d = sum(t.numel() * t.element_size() for t in host)
        copy_stream = torch.cuda.Stream()
        copied = [torch.cuda.Event() for _ in range(2)]
        freed = [torch.cuda.Event() for _ in range(2)]
        host_out = None

        def e2e_steps(n, a_ev=None):
            nonlocal host_out
            for i in range(n):
                buf = i % 2
                with torch.cuda.stream(copy_stream):
                    if i >= 2:
                        copy_stream.wait_event(freed[buf])
                    if i == 0 and a_ev is not None:
                        a_ev.record(copy_stream)
                    for dst, src in zip(dev_in[buf], host):
                        dst.copy_(src, non_blocking=True)
                    copied[buf].record(copy_stream)
                stream.wait_event(copied[buf])
                f = step(inputs=dev_in[buf], key=buf if use_graph else "eager")
                freed[buf].record(stream)
                outs = [fw_out["logp"], fw_out["entropy"], f["signed_mean"], f["abs_mean"], f["n_tokens"],
                        f["keep"], f["token_keep"]]
                if host_out is None:
                    host_out = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in outs]
                for dst, src in zip(host_out, outs):
                    dst.copy_(src, non_blocking=True)

        on_device = ("; grad_hidden (bf16 [N, d]) and grad_w (fp32 [V, d]) stay on the device for the rest "
                     "of the backward and the optimizer" if has_bwd else "")
        copies = ("double-buffered H2D on a copy stream, overlapped; D2H of the per-token and per-sequence "
                  "outputs" + on_device)
        if use_graph:
            # A launch-bound step replays, per buffer set, one graph holding
            # its H2D copies, the step's calls and the D2H copies (serialised:
            # the copies are small next to the launch overhead they replace).
            gflt = graphs["resident"][1]
            outs0 = [fw_out["logp"], fw_out["entropy"], gflt["signed_mean"], gflt["abs_mean"], gflt["n_tokens"],
                     gflt["keep"], gflt["token_keep"]]
            host_out = [torch.empty(t.shape, dtype=t.dtype, pin_memory=True) for t in outs0]
            e2e_graphs = []
            for buf in range(2):
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, capture_error_mode="thread_local"):
                    cs = torch.cuda.current_stream()
                    for dst, src in zip(dev_in[buf], host):
                        dst.copy_(src, non_blocking=True)
                    fb = None
                    for part in ("fwd", "filter", "bwd"):
                        if part == "bwd" and not has_bwd:
                            break
                        r = call(part, dev_in[buf], cs, fb)
                        fb = r if part == "filter" else fb
                    outs = [fw_out["logp"], fw_out["entropy"], fb["signed_mean"], fb["abs_mean"], fb["n_tokens"],
                            fb["keep"], fb["token_keep"]]
                    for dst, src in zip(host_out, outs):
                        dst.copy_(src, non_blocking=True)
                e2e_graphs.append(g)

            def e2e_steps(n, a_ev=None):  # noqa: F811 (the graph form of the loop above)
                for i in range(n):
                    if i == 0 and a_ev is not None:
                        a_ev.record(stream)
                    e2e_graphs[i % 2].replay()
                    if has_bwd:
                        dp_grad_w_allreduce(gw, world)

            copies = "H2D copies, the step and D2H copies replayed as one CUDA graph per buffer set" + on_device
        e2e_steps(2)  # warm
        torch.cuda.synchronize()
        d2h = sum(t.numel() * t.element_size() for t in host_out)
        _barrier(world)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        e2e_steps(args.steps, a_ev=a)
        b.record(stream)
        torch.cuda.synchronize()
        _barrier(world)
        e2e_ms = _max_over_ranks(a.elapsed_time(b), world)
        e2e = {"value": tokens_total / (e2e_ms / 1e3), "unit": "tokens/s", "h2d_bytes_per_step": h2d,
               "d2h_bytes_per_step": d2h, "copies": copies}

    # ---------------------------------------------------------------- CPU oracle baseline (rank 0, N = 1)
    cpu = None
    if world == 1 and not args.no_cpu:
        rows = min(args.cpu_rows, N)  # the tiny configuration has fewer tokens than the sample
        secs = oracle_sample_step(wl, rows, delta)
        cpu = {"value": rows / secs, "unit": "tokens/s", "cores": _cores(), "kind": "oracle", "blas": _blas(),
               "sample": f"first {rows} packed tokens of the workload (one sequence slice): fp64 forward over "
                         f"V={V}, filter, backward; {secs:.1f} s"}

    if rank == 0:
        line = {
            "metric": METRIC if has_bwd else METRIC_FWD,
            "value": value,
            "unit": "tokens/s",
            "n_gpus": world,
            "steps": args.steps,
            "warmup": args.warmup,
            "ms_per_step": ms_max / args.steps,
            "higher_is_better": True,
            "scaling": "weak",
            "vs_baseline": None,
            "dtype": "bf16",
            "data": "synthetic",
            "config": {"workload": spec.name, "tokens_per_step": N, "sequences": B, "d": d, "V": V,
                       "delta": delta, "kept_sequences": n_keep_seq, "kept_tokens": kept_rows,
                       "l2": (f"inputs larger than L2 (hidden {N * d * 2 / 1e9:.2f} GB, W {V * d * 2 / 1e9:.2f} GB); "
                              "no flush") if flush_buf is None else
                             "inputs fit in L2: a 256 MB write flushes it before every timed step, outside the "
                             "step's CUDA events (value = summed step times; e2e not flushed)",
                       "cuda_graph": use_graph,
                       "l2_persisting_limit_bytes": _l2_persisting_limit(),
                       "parallelism": (f"dp x{world}: grad_w all-reduced over ranks every step (NCCL)"
                                       if has_bwd and world > 1 else f"replicas x{world}")},
            "pct_of_bf16_peak": step_tflops / peak_tf,
            "step_tflops_algorithmic": step_tflops,
            "ms_by_call": {"forward": t_fwd, "filter": t_flt, "backward": t_bwd},
            "clocks": clk,
            "e2e": e2e,
            "gpu_launches": gpu_launches,
            "gpu_launches_source": "libmc launch counter (mc_kernel_launches) over the timed steps" +
                                   (" (graph replays: kernels captured per step x steps)" if use_graph else ""),
            "roofline": {"bound": "tensor", "kernel": "forward (tcgen05 projection + online log-softmax)",
                         "achieved": achieved, "peak": peak_tf, "unit": "TFLOP/s", "frac": achieved / peak_tf,
                         "peak_source": f"{peaks['source']} bf16 {peak_kind}", "traffic": traffic,
                         "traffic_source": "ncu single-pass capture of the full launch (profiles/fwd_kernel_traffic.json)"
                         if traffic is not None else None},
            "roofline_backward": None if not has_bwd else {
                "bound": "tensor", "achieved": flop_bwd / (t_bwd / 1e3) / 1e12, "peak": peak_tf, "unit": "TFLOP/s",
                "frac": flop_bwd / (t_bwd / 1e3) / 1e12 / peak_tf,
                "note": "achieved = algorithmic 4*N_g*d*V; executed adds the 2*N_g*d*V logit recompute the "
                        "configuration requires",
                "executed": 1.5 * flop_bwd / (t_bwd / 1e3) / 1e12,
                "executed_frac": 1.5 * flop_bwd / (t_bwd / 1e3) / 1e12 / peak_tf,
                "traffic": traffic_bwd,
                "traffic_source": "ncu single-pass capture of the three backward GEMMs of one call, scaled by kept "
                                  "rows (profiles/bwd_kernels_traffic.json)" if traffic_bwd is not None else None},
            "cpu_baseline": cpu,
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        import torch.distributed as dist

        dist.destroy_process_group()


def run_stream(args):
    """HBM bandwidth of the two token-streaming kernels (MirrorPop filter and
    masked GRPO loss) on a large synthetic batch: 64M tokens in 16,384
    sequences of 4,096 (or --rows tokens), CUDA events over --launches calls.
    Algorithmic bytes per token: filter 4 + 4 + 1 read, 4 + 1 written;
    loss 4 + 4 + 1 read, 4 written (per-sequence arrays are negligible)."""
    from paper_2606_04847_gb300 import build as mcbuild
    from paper_2606_04847_gb300 import mc

    torch.cuda.set_device(0)
    if not os.path.exists(mc.lib_path()):
        mcbuild.build()
    N = args.rows if args.rows > 0 else 64 * 1024 * 1024
    B = 16384
    g = torch.Generator(device="cuda").manual_seed(0)
    lp = -torch.rand(N, generator=g, device="cuda") * 8
    lb = lp + torch.randn(N, generator=g, device="cuda") * 0.2
    mask = (torch.rand(N, generator=g, device="cuda") < 0.9).to(torch.uint8)
    cu = torch.linspace(0, N, B + 1, device="cuda").round().to(torch.int64)
    adv = torch.randn(B, generator=g, device="cuda")
    flt = mc.seq_ratio_filter(lp, lb, mask, cu, 0.2, 0.2)
    loss = mc.grpo_masked_loss(lp, lb, mask, cu, adv, flt["keep"], flt["n_tokens"], 0.2, 0.28)
    peaks = _peaks()
    res = {"case": "stream", "tokens": N, "sequences": B, "launches": args.launches,
           "hbm_peak_gbs": peaks["hbm_gbs"], "peak_source": peaks["source"]}
    for name, fn, bpt in (("filter", lambda: mc.seq_ratio_filter(lp, lb, mask, cu, 0.2, 0.2, out=flt), 14),
                          ("loss", lambda: mc.grpo_masked_loss(lp, lb, mask, cu, adv, flt["keep"], flt["n_tokens"],
                                                               0.2, 0.28, out=loss), 13)):
        fn()
        torch.cuda.synchronize()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record()
        for _ in range(args.launches):
            fn()
        b.record()
        torch.cuda.synchronize()
        ms = a.elapsed_time(b) / args.launches
        gbs = bpt * N / (ms / 1e3) / 1e9
        res[name] = {"ms": ms, "bytes_per_token": bpt, "achieved_gbs": gbs, "frac": gbs / peaks["hbm_gbs"]}
    print(json.dumps(res), flush=True)


def _time_calls(fn, launches, warmup=3):
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    for _ in range(launches):
        fn()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / launches


def _time_graph(fn, launches, warmup=3):
    """Per-call GPU time of `launches` calls of fn captured into one CUDA graph
    and replayed: the kernels alone, without the host's per-call launch gaps
    (the calls must be capturable: stream-ordered, no synchronisation)."""
    for _ in range(warmup):
        fn()
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, capture_error_mode="thread_local"):
        for _ in range(launches):
            fn()
    g.replay()
    torch.cuda.synchronize()
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record()
    g.replay()
    b.record()
    torch.cuda.synchronize()
    return a.elapsed_time(b) / launches


def run_next(args):
    """Measurements of the rows beyond the main path (CUDA events over
    --launches calls each, after three untimed; the launch-bound merge and
    the 512-trajectory advantage from a CUDA-graph replay of those calls, with
    their eager per-call times beside), one JSON line:
    * the masked GRPO loss with the beta * KL term (reference log-probs) on
      64M tokens in 16,384 sequences: HBM GB/s for 4 + 4 + 4 + 1 B read and
      4 B written per token;
    * the vocabulary-sharded forward on the 9B-class fwd+bwd tokens: W in 4
      slices (a 4-way tensor-parallel LM head run in one process), TFLOP/s of
      2NdV over the 4 slice calls, and the merge's HBM GB/s (16 B per slice
      read + 12 B written per token);
    * the PrimeEcho reward and group advantage: the paper's batch (64
      prompts x groups of 8 = 512 trajectories, 4 turns: launch-bound) and 2^24."""
    from paper_2606_04847_gb300 import build as mcbuild
    from paper_2606_04847_gb300 import mc, workloads

    torch.cuda.set_device(0)
    if not os.path.exists(mc.lib_path()):
        mcbuild.build()
    peaks = _peaks()
    res = {"case": "next", "launches": args.launches, "peak_source": peaks["source"]}

    # masked GRPO loss + beta * KL
    N, B = 64 * 1024 * 1024, 16384
    g = torch.Generator(device="cuda").manual_seed(0)
    lp = -torch.rand(N, generator=g, device="cuda") * 8
    lb = lp + torch.randn(N, generator=g, device="cuda") * 0.2
    lr = lp + torch.randn(N, generator=g, device="cuda") * 0.1
    mask = (torch.rand(N, generator=g, device="cuda") < 0.9).to(torch.uint8)
    cu = torch.linspace(0, N, B + 1, device="cuda").round().to(torch.int64)
    adv = torch.randn(B, generator=g, device="cuda")
    flt = mc.seq_ratio_filter(lp, lb, mask, cu, 0.2, 0.2)
    out = mc.grpo_masked_loss(lp, lb, mask, cu, adv, flt["keep"], flt["n_tokens"], 0.2, 0.28, logp_ref=lr, beta=0.04)
    ms = _time_calls(lambda: mc.grpo_masked_loss(lp, lb, mask, cu, adv, flt["keep"], flt["n_tokens"], 0.2, 0.28,
                                                 logp_ref=lr, beta=0.04, out=out), args.launches)
    gbs = 17 * N / (ms / 1e3) / 1e9
    res["loss_kl"] = {"tokens": N, "ms": ms, "bytes_per_token": 17, "achieved_gbs": gbs,
                      "frac": gbs / peaks["hbm_gbs"], "peak_gbs": peaks["hbm_gbs"]}
    del lp, lb, lr, mask, cu, adv, flt, out
    torch.cuda.empty_cache()

    # vocabulary-sharded forward: 4 slices of W + merge
    spec = workloads.spec_for(CONFIG_ID)
    wl = workloads.build(spec, "cuda")
    h, w, y = wl.hidden, wl.w_vocab, wl.targets
    Nt, d, V, P = wl.N, spec.d, spec.V, 4
    bounds = [V * p // P for p in range(P + 1)]
    states = torch.empty((P, Nt, 4), dtype=torch.float32, device="cuda")
    ws = torch.empty(mc.forward_workspace_size(Nt, d, max(b - a for a, b in zip(bounds[:-1], bounds[1:]))),
                     dtype=torch.uint8, device="cuda")
    slices = [w[a:b] for a, b in zip(bounds[:-1], bounds[1:])]

    def shard_calls():
        for p in range(P):
            mc.token_logprob_state(h, slices[p], y, bounds[p], 1.0, state=states[p], workspace=ws)

    merged = mc.merge_logprob_states(states)
    ms_s = _time_calls(shard_calls, args.launches)
    ms_m_eager = _time_calls(lambda: mc.merge_logprob_states(states, out=merged), args.launches)
    ms_m = _time_graph(lambda: mc.merge_logprob_states(states, out=merged), args.launches)
    flop = 2.0 * Nt * d * V
    res["sharded_forward"] = {"tokens": Nt, "slices": P, "ms_slices": ms_s, "tflops": flop / (ms_s / 1e3) / 1e12,
                              "frac_of_sustained": flop / (ms_s / 1e3) / 1e12 / peaks["bf16_sustained"],
                              "merge_ms": ms_m, "merge_ms_eager_call": ms_m_eager,
                              "merge_bytes_per_token": 16 * P + 12,
                              "merge_gbs": (16 * P + 12) * Nt / (ms_m / 1e3) / 1e9}
    del wl, h, w, y, states, ws, slices, merged
    torch.cuda.empty_cache()

    # PrimeEcho reward + group advantage
    res["advantage"] = {}
    for T in (512, 1 << 24):
        K, G = 4, 8
        scores, success, n_turns = _advantage_inputs(T, K)
        call = lambda: mc.prime_echo_advantages(scores, success, n_turns, G, 0.75, 0.5, 0.2)  # noqa: E731
        ms_eager = _time_calls(call, args.launches)
        # Small batches are launch-bound: their kernel time comes from a graph replay.
        ms_a = _time_graph(call, args.launches) if T <= (1 << 16) else ms_eager
        bpt = 5 * K + 4 + 8
        res["advantage"][str(T)] = {"trajectories": T, "turns": K, "group": G, "us": ms_a * 1e3,
                                    "us_eager_call": ms_eager * 1e3, "bytes_per_trajectory": bpt,
                                    "achieved_gbs": bpt * T / (ms_a / 1e3) / 1e9}
    print(json.dumps(res), flush=True)


def _advantage_inputs(T, K):
    """Seeded per-turn scores in [-0.5, 1.5), success flags (30 % set) and turn
    counts in [1, K] for T trajectories, on the GPU."""
    gg = torch.Generator(device="cuda").manual_seed(1)
    scores = torch.rand((T, K), generator=gg, device="cuda") * 2 - 0.5
    success = (torch.rand((T, K), generator=gg, device="cuda") < 0.3).to(torch.uint8)
    n_turns = torch.randint(1, K + 1, (T,), generator=gg, device="cuda", dtype=torch.int32)
    return scores, success, n_turns


def run_advantage(args):
    """--case advantage: the reward + group advantage on 2^24 four-turn
    trajectories in groups of 8, `--launches` calls (for ncu captures), with
    the CUDA-event time per call."""
    from paper_2606_04847_gb300 import mc

    torch.cuda.set_device(0)
    T, K, G = 1 << 24, 4, 8
    scores, success, n_turns = _advantage_inputs(T, K)
    ms = _time_calls(lambda: mc.prime_echo_advantages(scores, success, n_turns, G, 0.75, 0.5, 0.2),
                     args.launches)
    bpt = 5 * K + 4 + 8
    print(json.dumps({"case": "advantage", "trajectories": T, "launches": args.launches, "us": ms * 1e3,
                      "bytes_per_trajectory": bpt, "achieved_gbs": bpt * T / (ms / 1e3) / 1e9}))


def run_case(args):
    """One call of the path, `--launches` times, for ncu captures (no timing printed
    beyond a one-line summary): --case fwd|bwd|filter|loss on the first `--rows`
    tokens of the `--config` workload (0 = all; bwd needs config 5, the one with
    advantage weights)."""
    from paper_2606_04847_gb300 import build as mcbuild
    from paper_2606_04847_gb300 import mc, workloads

    if args.case == "stream":
        return run_stream(args)
    if args.case == "next":
        return run_next(args)
    if args.case == "advantage":
        return run_advantage(args)
    torch.cuda.set_device(0)
    if not os.path.exists(mc.lib_path()):
        mcbuild.build()
    spec = workloads.spec_for(args.config)
    if args.case in ("bwd", "loss") and not spec.advantages:
        raise SystemExit(f"--case {args.case} needs a workload with advantage weights (--config 5)")
    # A --rows case draws only those rows (one sequence of the configuration's
    # shapes and distributions), so that a small capture holds little memory.
    wl = workloads.build(spec, "cuda", lengths=[args.rows] if args.rows > 0 else None)
    R = wl.N if args.rows <= 0 else min(args.rows, wl.N)
    h, w, y = wl.hidden[:R].contiguous(), wl.w_vocab, wl.targets[:R].contiguous()
    fw = mc.token_logprobs(h, w, y)
    cu = torch.tensor([0, R], dtype=torch.int64, device="cuda")
    lb = (fw["logp"] + wl.gap[:R]).contiguous()
    flt = mc.seq_ratio_filter(fw["logp"], lb, None, cu, spec.delta, spec.delta)
    adv = wl.advantages[:R].contiguous() if spec.advantages else None
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(args.launches):
        if args.case == "fwd":
            mc.token_logprobs(h, w, y, out=fw)
        elif args.case == "filter":
            mc.seq_ratio_filter(fw["logp"], lb, None, cu, spec.delta, spec.delta)
        elif args.case == "loss":
            mc.grpo_masked_loss(fw["logp"], lb, None, cu, adv[:1].contiguous(), flt["keep"], flt["n_tokens"],
                                0.2, 0.28)
        else:  # every row live, so the capture does not depend on whether the filter keeps this slice
            mc.token_logprobs_bwd(h, w, y, fw["lse"], fw["entropy"], adv, None)
    torch.cuda.synchronize()
    print(json.dumps({"case": args.case, "config": args.config, "rows": R, "launches": args.launches,
                      "wall_ms_per_launch": (time.perf_counter() - t0) * 1e3 / args.launches}))


def run_reference(args):
    """The CPU fp64 oracle, as it stands, on a bounded sample per step."""
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    from paper_2606_04847_gb300 import workloads

    spec = workloads.spec_for(args.config)
    wl = workloads.build(spec, "cuda" if torch.cuda.is_available() else "cpu")
    rows = min(args.ref_rows, wl.N)
    for _ in range(args.warmup):
        oracle_sample_step(wl, rows, spec.delta)
    total = 0.0
    for _ in range(args.steps):
        total += oracle_sample_step(wl, rows, spec.delta)
    value = rows * args.steps / total
    line = {
        "impl": "reference",
        "metric": METRIC if spec.advantages else METRIC_FWD,
        "value": value,
        "unit": "tokens/s",
        "n_gpus": world,
        "steps": args.steps,
        "warmup": args.warmup,
        "ms_per_step": total / args.steps * 1e3,
        "higher_is_better": True,
        "scaling": "weak",
        "vs_baseline": None,
        "dtype": "f64",
        "data": "synthetic",
        "config": {"workload": spec.name, "tokens_per_step": rows, "d": spec.d, "V": spec.V,
                   "note": "each step: the oracle on the first packed tokens of the workload"},
        "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": _cores(), "kind": "oracle", "blas": _blas(),
                         "sample": f"{rows} tokens per step"},
        "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", type=int, choices=[1, 2, 3, 4, 5], default=CONFIG_ID,
                    help="workload: 5 (default) = 9B-class fwd+bwd; 1-4 = the forward-only workloads "
                         "(step = forward + filter)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--graph", choices=["auto", "on", "off"], default="auto",
                    help="replay each call of the step as a CUDA graph (auto: when a step is launch-bound)")
    ap.add_argument("--no-cpu", action="store_true")
    ap.add_argument("--cpu-rows", type=int, default=512)
    ap.add_argument("--ref-rows", type=int, default=64)
    ap.add_argument("--case", choices=["step", "fwd", "bwd", "filter", "loss", "stream", "next", "advantage"],
                    default="step",
                    help="profiling aid: run one call of the path --launches times")
    ap.add_argument("--rows", type=int, default=0, help="--case: tokens to use (0 = the whole batch)")
    ap.add_argument("--launches", type=int, default=2)
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args)
    elif args.case != "step":
        run_case(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
