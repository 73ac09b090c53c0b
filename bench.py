"""Throughput of the SOLO shared-readout local loss (forward + backward) on GB300.

One step = one call of solo_readout_fwd_bwd over all K modules: final
RMSNorm, logits through the shared readout, softmax cross-entropy, dH for
every module, dW and dgamma for the final module.  The default workload is
the headline one: K=4 modules of N=8192 tokens, d=2048, V=32000.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

Prints ONE JSON line (rank 0).  Under torchrun each rank runs an independent
replica of the workload on its own GPU (the path has no exchange step), and
the value is the tokens of all ranks over the slowest rank's time.

Timing: inputs are resident in HBM; hidden states and W (265 MB) exceed the
129 MB L2 and every step writes its 2.1 GB logit-gradient buffer, so no step
finds its inputs in L2.  CUDA events on the launching stream, W >= 3 warm-up
steps, a barrier and a device synchronize on both sides of the timed region.
``e2e`` repeats the measurement through the same C ABI call with every step's
inputs copied from pinned host memory (on a copy stream, into one of two
device buffers, overlapping the previous step's compute) and its losses read
back, all inside the timed region.  ``cpu_baseline`` times the fp64 oracle
on a bounded sample of the same workload on the host cores.  ``gpu_launches``
is the library's own count of the kernels it enqueued during the timed calls.
"""
from __future__ import annotations

import argparse
import hashlib
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

from paper_2609_35440_gb300 import costmodel, synth, workloads  # noqa: E402

METRIC = "local-readout CE fwd+bwd tokens/s at d=2048,V=32000; % of bf16 tensor peak"
EXIT_METRIC = "early-exit readout (forward: loss, top-1) tokens/s at d=2048,V=32000"
PRIVATE_METRIC = ("private readouts (PRIV) fwd+bwd with dW_k, dgamma_k for every module "
                  "tokens/s at d=2048,V=32000")
HEADS_METRIC = ("local-readout CE fwd+bwd with head temperature and bias (+dtau, dbias) "
                "tokens/s at d=2048,V=32000")
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
KERNEL_SOURCES = ["paper_2609_35440_gb300/csrc/gemm_tc.cu", "paper_2609_35440_gb300/csrc/ptx.cuh",
                  "paper_2609_35440_gb300/csrc/internal.h"]
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "logits_gemm_traffic.txt")


def parse():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", default="ours", choices=["ours", "reference"])
    p.add_argument("--workload", default=workloads.HEADLINE.name,
                   help="a workload name, or k<K>_n<N>_d<d>_v<V> for a custom uniform one")
    p.add_argument("--no-e2e", action="store_true")
    p.add_argument("--no-cpu", action="store_true")
    p.add_argument("--cpu-seconds", type=float, default=25.0)
    p.add_argument("--mode", default="train",
                   choices=["train", "heads", "exit", "private", "onchip"],
                   help="train: forward + backward (the headline); heads: the same with "
                        "each head's temperature and bias and their gradients; exit: "
                        "forward-only early-exit readout (losses, top-1); onchip: the "
                        "forward + backward with the auxiliary modules' logits kept on chip")
    return p.parse_args()


def workload_from_name(name: str) -> workloads.Workload:
    if name in workloads.BY_NAME:
        return workloads.BY_NAME[name]
    import re
    m = re.fullmatch(r"k(\d+)_n(\d+)_d(\d+)_v(\d+)", name)
    if not m:
        raise SystemExit(f"unknown workload {name}")
    K, N, d, V = map(int, m.groups())
    return workloads.Workload(name, K=K, N=N, d=d, V=V, seed=7)


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return p, "measured"
    except (OSError, ValueError):
        return FALLBACK_PEAKS, "fallback"


SUSTAINED_AFTER_S = 1.0   # timed regions at least this long run under the power cap


def tensor_peak(peaks, src: str, timed_s: float):
    """The bf16 peak that matches how the kernels were timed: the burst figure
    (torch.matmul best of 10) for a timed region shorter than a second, the
    sustained one (seconds back to back under the power cap) otherwise."""
    if timed_s < SUSTAINED_AFTER_S:
        key, why = "bf16_tflops", f"timed region {timed_s:.2f} s < {SUSTAINED_AFTER_S:.0f} s"
    else:
        key, why = "bf16_tflops_sustained", f"timed region {timed_s:.2f} s >= " \
                                            f"{SUSTAINED_AFTER_S:.0f} s"
    return float(peaks.get(key, FALLBACK_PEAKS[key])), f"{src} {key} ({why})"


def kept_counts(wl, targets) -> list:
    """Kept tokens per module: targets in [0, V) (ignore_index and anything out
    of range are masked, as the library treats them)."""
    t = np.asarray(targets)
    return [int(np.sum((t[k] >= 0) & (t[k] < wl.V))) for k in range(wl.K)]


def strip_comments(src: str) -> str:
    """C++ source without comments, every run of whitespace made one space, so
    that neither comments nor layout count as a change of the code (string
    literals in these files hold no comment markers and no significant runs of
    spaces)."""
    import re
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    src = re.sub(r"//[^\n]*", "", src)
    return " ".join(src.split())


def kernel_hash() -> str:
    """Hash of the GEMM kernel's code (comments ignored): a committed traffic
    capture applies only while this is unchanged.  Of the shared header only
    the part before the on-chip pass's and the row kernels' declarations
    counts (the GEMM's constants and arguments)."""
    h = hashlib.sha256()
    for rel in KERNEL_SOURCES:
        with open(os.path.join(ROOT, rel), encoding="utf-8") as f:
            src = f.read()
        if rel.endswith("internal.h"):
            src = src.split("struct FlashArgs", 1)[0]
        h.update(strip_comments(src).encode())
    return h.hexdigest()[:16]


def committed_traffic(wl, kept_tokens: int, kernel: str = "logits"):
    """Bytes per launch of the logits or the dX GEMM from the committed ncu
    capture, if the kernel source is unchanged since.  The logits GEMM's figure
    is scaled to this workload's kept tokens x vocabulary tiles (the reads also
    by d); the dX GEMM's (which reads the exponentials, W once per raster group
    and the hidden rows, and writes dH) only to its kept tokens, at the captured
    d and V (None otherwise)."""
    try:
        kv = {}
        with open(TRAFFIC_FILE) as f:
            for ln in f:
                if "=" in ln and not ln.startswith("#"):
                    k, v = ln.split("=", 1)
                    kv[k.strip()] = v.strip()
        if kv.get("kernel_sha") != kernel_hash():
            return None
        if kernel == "dxhat":
            if wl.d != int(kv["d"]) or wl.V != int(kv["V"]):
                return None
            return kept_tokens * float(kv["dxhat_dram_bytes_per_token"])
        if kernel != "logits":
            return None
        w = float(kv["dram_write_bytes_per_token_per_vocab_tile"])
        r = float(kv["dram_read_bytes_per_token_per_vocab_tile"])
        return kept_tokens * ((wl.V + 255) // 256) * (w + r * wl.d / float(kv["d"]))
    except (OSError, KeyError, ValueError):
        return None


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    Q = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index: int):
        self.index = 0 if index is None else index
        self.proc = None
        self.window = None          # (first, last) sample indices of the timed region
        self.lines = []

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.index), f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            # nvidia-smi takes a moment to start: the timed region begins once it samples
            t0 = time.time()
            while not self.lines and self.proc.poll() is None and time.time() - t0 < 5.0:
                time.sleep(0.01)
        except OSError:
            self.proc = None
        return self

    def _read(self):
        for ln in self.proc.stdout:
            self.lines.append(ln.strip())

    def __exit__(self, *exc):
        if self.proc is not None:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=2)

    def mark_start(self):
        """Call right before the timed region is enqueued."""
        self.window = (len(self.lines), None)

    def mark_end(self):
        """Call once the timed region has completed on the device.  A region
        shorter than the sampling period waits (at most a second) for the first
        sample after its start."""
        if self.window is None:
            return
        t0 = time.time()
        while (len(self.lines) <= self.window[0] and self.proc is not None
               and self.proc.poll() is None and time.time() - t0 < 1.0):
            time.sleep(0.005)
        self.window = (self.window[0], len(self.lines))

    def summary(self):
        sm, mx, pw, reasons = [], [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        lines = self.lines
        if self.window is not None and self.window[1] is not None:
            # the samples taken while the timed calls ran; a region shorter than
            # the sampling period keeps the first sample after its start
            lo, hi = self.window
            lines = self.lines[lo:max(hi, lo + 1)]
        for ln in lines:
            parts = [x.strip() for x in ln.split(",")]
            if len(parts) < 8:
                continue
            try:
                sm.append(float(parts[0]))
                mx.append(float(parts[1]))
            except ValueError:
                continue
            try:
                pw.append(float(parts[2]))
            except ValueError:
                pass
            for nm, v in zip(names, parts[4:8]):
                if v.lower().startswith("active"):
                    reasons.add(nm)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx),
                "sm_mhz_min": min(sm),
                "power_w": statistics.median(pw) if pw else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ----------------------------------------------------------------------- ranks

def max_over_ranks(value: float, device=None) -> float:
    """The largest value over all ranks (the slowest rank's time); identity at N=1."""
    import torch
    import torch.distributed as dist
    if not (dist.is_available() and dist.is_initialized()) or dist.get_world_size() == 1:
        return float(value)
    t = torch.tensor([float(value)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(tokens_per_rank_step: int, steps: int, world: int, ms_max: float) -> float:
    """Whole-job tokens/s: every rank's tokens over the slowest rank's time."""
    return world * tokens_per_rank_step * steps / (ms_max / 1e3)


def replica_workload(wl, rank: int):
    """Rank r runs an independent replica of the workload with its own inputs."""
    return wl.with_(seed=wl.seed + 1000 * rank) if rank else wl


# ----------------------------------------------------------------------- e2e

E2E_METHOD = ("every step: its hidden states and targets copied from pinned host memory "
              "into one of two device buffers on a copy stream (overlapping the previous "
              "step's compute), the call, and its losses copied back; all inside the timed "
              "region.  Returned to the host: loss_tok and loss_mean only; dH, dW and dgamma "
              "stay on the device for the caller's backward pass")

def pipelined_e2e(torch, dev, stream, h_host, t_host, hidden, targets, compute, read_back,
                  steps, warm=2):
    """Times `steps` end-to-end steps: each step's inputs are copied from pinned host
    memory on a copy stream into one of two device buffers while the previous step
    computes; `compute(hidden, targets)` runs on `stream` and `read_back()` queues the
    device-to-host copies of its results.  Returns the elapsed ms of the whole chain."""
    copy_stream = torch.cuda.Stream(dev)
    bufs = [([torch.empty_like(h) for h in hidden], torch.empty_like(targets)) for _ in range(2)]
    copied = [torch.cuda.Event() for _ in range(2)]
    consumed = [torch.cuda.Event() for _ in range(2)]
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)

    def issue_copy(i):
        b = i % 2
        with torch.cuda.stream(copy_stream):
            copy_stream.wait_event(consumed[b])
            for dst, src in zip(bufs[b][0], h_host):
                dst.copy_(src, non_blocking=True)
            bufs[b][1].copy_(t_host, non_blocking=True)
            copied[b].record(copy_stream)

    def run(n):
        issue_copy(0)
        for i in range(n):
            if i + 1 < n:
                issue_copy(i + 1)
            b = i % 2
            stream.wait_event(copied[b])
            compute(bufs[b][0], bufs[b][1])
            consumed[b].record(stream)
            read_back()

    with torch.cuda.stream(stream):
        run(warm)
        torch.cuda.synchronize(dev)
        start.record(stream)
        copy_stream.wait_event(start)
        run(steps)
        end.record(stream)
    torch.cuda.synchronize(dev)
    return start.elapsed_time(end)


# ----------------------------------------------------------------------- CPU legs

def oracle_sample(wl, rows: int, inp_rows=None):
    """One bounded oracle pass: the first `rows` tokens of every module, forward and
    dH, plus dW/dgamma contributions of the final module's sampled rows."""
    import oracle.solo_oracle as orc
    if inp_rows is None:
        inp_rows = prepare_oracle_sample(wl, rows)
    hidden, gamma, W, targets = inp_rows
    for k in range(wl.K):
        y = targets[k].astype(np.int64)
        kept, _ = orc.kept_tokens(y, None, wl.V, wl.ignore_index)
        res = orc.module_rows(hidden[k], gamma, W, y, kept, max(int(kept.sum()), 1),
                              float(np.float32(wl.eps)), True)
        if k == wl.K - 1:
            orc.readout_grads(res["g"], res["xhat"], res["dxhat"], hidden[k], res["r"])
    return wl.K * rows


def prepare_oracle_sample(wl, rows: int):
    import oracle.solo_oracle as orc
    dec = orc.bf16_bits_to_f64
    hidden = [dec(synth.gen_hidden(wl, k, 0, rows)) for k in range(wl.K)]
    W = dec(synth.gen_W(wl))
    gamma = dec(synth.gen_gamma(wl))
    targets = synth.gen_targets(wl)[:, :rows]
    return hidden, gamma, W, targets


def blas_threads() -> int:
    try:
        from threadpoolctl import threadpool_info
        n = [i.get("num_threads", 0) for i in threadpool_info() if i.get("user_api") == "blas"]
        if n:
            return int(max(n))
    except Exception:
        pass
    return len(os.sched_getaffinity(0))


L2_BYTES = 129e6   # GB300 L2


def l2_note(wl, writes_exponentials: bool) -> str:
    """How the timed steps relate to L2: the timing rules want inputs larger
    than L2, or L2 flushed between steps."""
    inputs = wl.M * wl.d * 2 + wl.V * wl.d * 2                 # hidden + W, bf16
    buf = wl.M * (wl.V + (-wl.V) % 8) * 2 if writes_exponentials else 0
    if inputs > L2_BYTES:
        return f"inputs larger than L2 (hidden+W {inputs / 1e6:.0f} MB)"
    if buf > L2_BYTES:
        return (f"hidden+W {inputs / 1e6:.0f} MB fit in L2, but every step writes a "
                f"{buf / 1e9:.2f} GB exponential/gradient buffer, which evicts them")
    return (f"inputs fit in L2 ({inputs / 1e6:.0f} MB) and are not flushed between steps: "
            f"not a reportable configuration")


def cpu_baseline(wl, seconds: float):
    cap = min(4096, wl.N)                 # a sample never exceeds the module's tokens
    probe = min(16, cap)
    data = prepare_oracle_sample(wl, cap)
    sub = lambda n: ([h[:n] for h in data[0]], data[1], data[2], data[3][:, :n])
    oracle_sample(wl, probe, sub(probe))
    t = time.perf_counter()
    oracle_sample(wl, probe, sub(probe))
    per_row = (time.perf_counter() - t) / probe
    # the per-row cost falls with the sample size (larger matrix products), so
    # the target is set above the 10-30 s the sample should take
    rows = int(min(cap, max(probe, seconds / max(per_row, 1e-9))))
    t = time.perf_counter()
    toks = oracle_sample(wl, rows, sub(rows))
    dt = time.perf_counter() - t
    return {"value": toks / dt, "unit": "tokens/s", "cores": blas_threads(), "kind": "oracle",
            "sample": f"first {rows} tokens of each of the {wl.K} modules (full V={wl.V}, "
                      f"d={wl.d}), forward + dH, dW/dgamma terms of the final module's "
                      f"sample; fp64 numpy oracle, {dt:.1f} s"}


def run_reference(args, wl):
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    rows = min(32, wl.N)
    data = prepare_oracle_sample(wl, rows)
    for _ in range(args.warmup):
        oracle_sample(wl, rows, data)
    t = time.perf_counter()
    toks = 0
    for _ in range(args.steps):
        toks += oracle_sample(wl, rows, data)
    dt = time.perf_counter() - t
    value = toks / dt
    line = {"metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": args.gpus,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": dt / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic", "impl": "reference",
            "config": {"workload": wl.name, "K": wl.K, "N": wl.N, "d": wl.d, "V": wl.V,
                       "parallelism": "rank 0 only"},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": blas_threads(),
                             "kind": "oracle",
                             "sample": f"each step: first {rows} tokens of each of the {wl.K} "
                                       f"modules at full V and d"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ----------------------------------------------------------------------- GPU leg

def run_ours(args, wl):
    import torch
    import torch.distributed as dist
    from paper_2609_35440_gb300 import solo_readout as sr
    from paper_2609_35440_gb300 import build

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        torch.cuda.set_device(local)
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))
    dev = torch.device("cuda", local if world > 1 else torch.cuda.current_device())

    build.ensure_built()
    sr.load()
    stream = torch.cuda.current_stream(dev)

    # inputs resident in HBM (seeded; ranks use distinct seeds: independent replicas)
    wlr = replica_workload(wl, rank)
    inp = synth.generate(wlr)
    to_dev = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).to(dev).view(
        torch.bfloat16)
    hidden = [to_dev(inp.hidden[k]) for k in range(wl.K)]
    gamma, W = to_dev(inp.gamma), to_dev(inp.W)
    targets = torch.from_numpy(inp.targets).to(dev)
    onchip = args.mode == "onchip"
    ro = sr.Readout(wl.K, wl.N, wl.d, wl.V, eps=wl.eps, ignore_index=wl.ignore_index, device=dev,
                    onchip=onchip)
    n_stages = sr.SOLO_ONCHIP_NUM_STAGES if onchip else sr.SOLO_NUM_STAGES
    heads = {}
    if args.mode == "heads":
        tau, bias = synth.gen_heads(wlr)
        heads = dict(tau=torch.from_numpy(tau).to(dev), bias=torch.from_numpy(bias).to(dev),
                     head_grads=True)
    def barrier():
        if world > 1:
            dist.barrier()
        torch.cuda.synchronize(dev)

    clk = ClockSampler(dev.index).__enter__()
    time.sleep(1.0)                      # let the sampler start before the warm-up
    for _ in range(max(args.warmup, 0)):
        ro(hidden, gamma, W, targets, stream=stream, **heads)
    barrier()

    # ---- device-resident timing of exactly `steps` calls; events recorded on the
    # launching stream between the stages of every call (read after the loop)
    step_evs = [[torch.cuda.Event(enable_timing=True) for _ in range(n_stages + 1)]
                for _ in range(args.steps)]
    for evl in step_evs:
        for e in evl:
            e.record(stream)
    barrier()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    barrier()
    launches0 = sr.solo_readout_kernel_launches()
    clk.mark_start()
    t0.record(stream)
    for i in range(args.steps):
        ro(hidden, gamma, W, targets, stream=stream, events=step_evs[i], **heads)
    t1.record(stream)
    launches = sr.solo_readout_kernel_launches() - launches0
    barrier()
    clk.mark_end()
    clk.__exit__(None, None, None)
    flags = ro.flags(stream)
    ms = t0.elapsed_time(t1)
    stage_ms = np.zeros(n_stages)
    for evl in step_evs:
        stage_ms += [evl[i].elapsed_time(evl[i + 1]) for i in range(n_stages)]
    stage_ms /= args.steps
    # each call from its first stage's start to its last stage's end
    call_ms = [evl[0].elapsed_time(evl[n_stages]) for evl in step_evs]

    ms = max_over_ranks(ms, dev)
    tokens_step = wl.M
    value = job_throughput(tokens_step, args.steps, world, ms)

    # ---- end to end through the C ABI with host buffers
    e2e = None
    if not args.no_e2e:
        h_host = [torch.from_numpy(np.ascontiguousarray(inp.hidden[k]).view(np.int16)).view(
            torch.bfloat16).pin_memory() for k in range(wl.K)]
        t_host = torch.from_numpy(inp.targets).pin_memory()
        lt_host = torch.empty(wl.K, wl.N, dtype=torch.float32).pin_memory()
        lm_host = torch.empty(wl.K, dtype=torch.float32).pin_memory()
        steps_e2e = max(3, args.steps)

        def compute(hid, tg):
            ro(hid, gamma, W, tg, stream=stream, **heads)

        def read_back():
            lt_host.copy_(ro.loss_tok, non_blocking=True)
            lm_host.copy_(ro.loss_mean, non_blocking=True)

        barrier()
        ems = pipelined_e2e(torch, dev, stream, h_host, t_host, hidden, targets, compute,
                            read_back, steps_e2e)
        barrier()
        ems = max_over_ranks(ems, dev)
        h2d = sum(h.numel() * 2 for h in h_host) + t_host.numel() * 4
        d2h = lt_host.numel() * 4 + lm_host.numel() * 4
        e2e = {"value": job_throughput(tokens_step, steps_e2e, world, ems), "unit": "tokens/s",
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h, "method": E2E_METHOD}

    if rank != 0:
        if world > 1:
            dist.destroy_process_group()
        return

    peaks, peak_src = load_peaks()
    G = costmodel.gemm_flops(wl.M, wl.V, wl.d)     # one module-GEMM over all K modules
    n_kept = kept_counts(wl, inp.targets)
    Gk = costmodel.gemm_flops(sum(n_kept), wl.V, wl.d)   # over the kept tokens
    if onchip:
        names = sr.ONCHIP_STAGE_NAMES
        # final module: logits, dX and dW over its N tokens; auxiliary modules: the
        # logits and sum_v P_v W_v of K-1 modules in one pass
        gemm_stage_flops = {"final": 3 * G / wl.K, "aux_onchip": 2 * G * (wl.K - 1) / wl.K}
    else:
        names = sr.STAGE_NAMES
        # masked tokens are skipped: the logits and dX products run over the kept
        # tokens; dW reduces over the final module's kept tokens in whole blocks of
        # 128 rows (the last one completed with zeros)
        dw_rows = -(-(n_kept[-1] if n_kept[-1] > 0 else wl.N) // 128) * 128
        gemm_stage_flops = {"logits": Gk, "dxhat": Gk,
                            "dW": costmodel.gemm_flops(dw_rows, wl.V, wl.d)}
    dom = max(gemm_stage_flops, key=lambda s: stage_ms[names.index(s)])
    dom_ms = stage_ms[names.index(dom)]
    achieved = gemm_stage_flops[dom] / (dom_ms / 1e3) / 1e12
    peak, peak_name = tensor_peak(peaks, peak_src, ms / 1e3)
    traffic = None if onchip else committed_traffic(wl, sum(n_kept), dom)
    algo = costmodel.call_flops(wl.K, wl.N, wl.d, wl.V)
    kept = costmodel.kept_call_flops(n_kept, wl.d, wl.V)
    executed = sum(gemm_stage_flops.values())
    step_s = ms / 1e3 / args.steps
    cpu = None
    if not args.no_cpu:
        cpu = cpu_baseline(wl, args.cpu_seconds)
    line = {
        "metric": HEADS_METRIC if heads else METRIC, "value": value, "unit": "tokens/s",
        "workspace_bytes": int(ro.workspace.numel()),
        "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic", "mode": args.mode,
        "config": {"workload": wl.name, "K": wl.K, "N": wl.N, "d": wl.d, "V": wl.V,
                   "global_batch_tokens": world * wl.M, "parallelism": f"replicas{world}",
                   "l2": l2_note(wl, True)},
        # the paper's count, (2K+1) 2NVd over every token of the call, per second
        # (a rate, not a fraction of peak: masked tokens are skipped)
        "algo_tflops": algo / step_s / 1e12,
        # the paper's work on the kept tokens (the mean loss counts kept tokens),
        # against the same peak as the roofline: the whole call's fraction
        "kept_algo_tflops": kept / step_s / 1e12,
        "kept_algo_frac_of_peak": kept / step_s / 1e12 / peak,
        # what the tensor cores execute: no logits are recomputed (the forward
        # stores its exponentials), masked tokens are skipped except in dW's
        # reduction over the final module's N rows
        "executed_tflops": executed / step_s / 1e12,
        "executed_frac_of_peak": executed / step_s / 1e12 / peak,
        "stages_ms": {n: round(float(v), 4) for n, v in zip(names, stage_ms)},
        # per call (first stage start to last stage end, CUDA events): the
        # median and the minimum over the timed calls, beside the mean above
        "call_ms": {"median": round(float(np.median(call_ms)), 4),
                    "min": round(float(np.min(call_ms)), 4)},
        "roofline": {"bound": "tensor",
                     "kernel": ("auxiliary on-chip pass (tcgen05, cluster split of d)"
                                if dom == "aux_onchip" else f"{dom} GEMM (tcgen05)"
                                if not onchip else "final module, stored path (tcgen05)"),
                     "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "peak_source": peak_name},
        "cpu_baseline": cpu,
        "e2e": e2e,
        "clocks": clk.summary(),
        "gpu_launches": launches,       # the library's own count over the timed calls
        "device_flags": flags,
    }
    print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()


def exit_oracle_sample(wl, rows: int, data):
    import oracle.solo_oracle as orc
    hidden, gamma, W, targets = data
    orc.exit_readout([h[:rows] for h in hidden], gamma, W, targets[:, :rows],
                     eps=float(np.float32(wl.eps)), ignore_index=wl.ignore_index)
    return wl.K * rows


def run_exit_bench(args, wl):
    """The forward-only early-exit readout on the same workload (single GPU line)."""
    import torch
    from paper_2609_35440_gb300 import solo_readout as sr
    from paper_2609_35440_gb300 import build
    build.ensure_built()
    sr.load()
    dev = torch.device("cuda", torch.cuda.current_device())
    stream = torch.cuda.current_stream(dev)
    inp = synth.generate(wl)
    to_dev = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).to(dev).view(
        torch.bfloat16)
    hidden = [to_dev(inp.hidden[k]) for k in range(wl.K)]
    gamma, W = to_dev(inp.gamma), to_dev(inp.W)
    targets = torch.from_numpy(inp.targets).to(dev)
    ex = sr.ExitReadout(wl.K, wl.N, wl.d, wl.V, eps=wl.eps, ignore_index=wl.ignore_index,
                        device=dev)
    clk = ClockSampler(dev.index).__enter__()
    time.sleep(1.0)
    for _ in range(max(args.warmup, 0)):
        ex(hidden, gamma, W, targets, stream=stream)
    torch.cuda.synchronize(dev)
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(sr.SOLO_EXIT_NUM_STAGES + 1)]
           for _ in range(args.steps)]
    for evl in evs:
        for e in evl:
            e.record(stream)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    torch.cuda.synchronize(dev)
    launches0 = sr.solo_readout_kernel_launches()
    clk.mark_start()
    t0.record(stream)
    for i in range(args.steps):
        ex(hidden, gamma, W, targets, stream=stream, events=evs[i])
    t1.record(stream)
    launches = sr.solo_readout_kernel_launches() - launches0
    torch.cuda.synchronize(dev)
    clk.mark_end()
    clk.__exit__(None, None, None)
    ms = t0.elapsed_time(t1)
    stage_ms = np.zeros(sr.SOLO_EXIT_NUM_STAGES)
    for evl in evs:
        stage_ms += [evl[i].elapsed_time(evl[i + 1]) for i in range(sr.SOLO_EXIT_NUM_STAGES)]
    stage_ms /= args.steps
    call_ms = [evl[0].elapsed_time(evl[sr.SOLO_EXIT_NUM_STAGES]) for evl in evs]
    flags = ex.flags(stream)
    value = job_throughput(wl.M, args.steps, 1, ms)
    # end to end: hidden states and targets from pinned host memory, losses and
    # top-1 back to the host
    h_host = [torch.from_numpy(np.ascontiguousarray(inp.hidden[k]).view(np.int16)).view(
        torch.bfloat16).pin_memory() for k in range(wl.K)]
    t_host = torch.from_numpy(inp.targets).pin_memory()
    lt_host = torch.empty(wl.K, wl.N, dtype=torch.float32).pin_memory()
    top_host = torch.empty(wl.K, wl.N, dtype=torch.int32).pin_memory()
    steps_e2e = max(3, args.steps)

    def compute(hid, tg):
        ex(hid, gamma, W, tg, stream=stream)

    def read_back():
        lt_host.copy_(ex.loss_tok, non_blocking=True)
        top_host.copy_(ex.top1, non_blocking=True)

    ems = pipelined_e2e(torch, dev, stream, h_host, t_host, hidden, targets, compute, read_back,
                        steps_e2e)
    peaks, peak_src = load_peaks()
    peak, peak_name = tensor_peak(peaks, peak_src, ms / 1e3)
    G = costmodel.gemm_flops(wl.M, wl.V, wl.d)
    achieved = G / (stage_ms[1] / 1e3) / 1e12
    cpu = None
    if not args.no_cpu:
        cap = min(4096, wl.N)
        probe = min(16, cap)
        data = prepare_oracle_sample(wl, cap)
        exit_oracle_sample(wl, probe, data)
        t = time.perf_counter()
        exit_oracle_sample(wl, probe, data)
        per_row = (time.perf_counter() - t) / probe
        rows = int(min(cap, max(probe, args.cpu_seconds / max(per_row, 1e-9))))
        t = time.perf_counter()
        toks = exit_oracle_sample(wl, rows, data)
        dt = time.perf_counter() - t
        cpu = {"value": toks / dt, "unit": "tokens/s", "cores": blas_threads(), "kind": "oracle",
               "sample": f"first {rows} tokens of each of the {wl.K} modules, exit readout "
                         f"(logits, log-sum-exp, argmax, losses) in fp64 numpy, {dt:.1f} s"}
    line = {
        "metric": EXIT_METRIC, "value": value, "unit": "tokens/s", "n_gpus": 1,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic", "mode": "exit",
        "config": {"workload": wl.name, "K": wl.K, "N": wl.N, "d": wl.d, "V": wl.V,
                   "parallelism": "replicas1",
                   "l2": l2_note(wl, False)},
        "stages_ms": {n: round(float(v), 4) for n, v in zip(sr.EXIT_STAGE_NAMES, stage_ms)},
        "call_ms": {"median": round(float(np.median(call_ms)), 4),
                    "min": round(float(np.min(call_ms)), 4)},
        "roofline": {"bound": "tensor", "kernel": "exit logits GEMM (tcgen05)",
                     "achieved": achieved, "peak": peak, "unit": "TFLOP/s",
                     "frac": achieved / peak, "traffic": None,
                     "peak_source": peak_name},
        "cpu_baseline": cpu,
        "e2e": {"value": job_throughput(wl.M, steps_e2e, 1, ems), "unit": "tokens/s",
                "h2d_bytes_per_step": sum(h.numel() * 2 for h in h_host) + t_host.numel() * 4,
                "d2h_bytes_per_step": lt_host.numel() * 4 + top_host.numel() * 4,
                "method": E2E_METHOD.split("  Returned")[0].replace(
                    "its losses", "its losses and top-1") +
                          "  Returned to the host: loss_tok and top1"},
        "clocks": clk.summary(),
        "gpu_launches": launches,       # the library's own count over the timed calls
        "device_flags": flags,
    }
    print(json.dumps(line), flush=True)


def run_private_bench(args, wl):
    """Private readouts: every module its own W_k and gain gamma_k (dW_k, dgamma_k)."""
    import torch
    from paper_2609_35440_gb300 import solo_readout as sr
    from paper_2609_35440_gb300 import build
    build.ensure_built()
    sr.load()
    dev = torch.device("cuda", torch.cuda.current_device())
    stream = torch.cuda.current_stream(dev)
    inp = synth.generate(wl)
    to_dev = lambda b: torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).to(dev).view(
        torch.bfloat16)
    K, N, d, V = wl.K, wl.N, wl.d, wl.V
    hidden = [to_dev(inp.hidden[k]) for k in range(K)]
    Ws = [to_dev(synth.gen_W(wl.with_(seed=wl.seed + 100 * k))) for k in range(K)]
    gs = [to_dev(synth.gen_gamma(wl.with_(seed=wl.seed + 100 * k))) for k in range(K)]
    targets = torch.from_numpy(inp.targets).to(dev)
    dims = sr.make_dims(K, N, d, V, wl.eps, wl.ignore_index)
    ws = torch.empty(sr.solo_readout_private_workspace_bytes(dims), dtype=torch.uint8, device=dev)
    loss_tok = torch.empty(K, N, device=dev)
    loss_mean = torch.empty(K, device=dev)
    dh = [torch.empty(N, d, dtype=torch.bfloat16, device=dev) for _ in range(K)]
    dW = [torch.empty(V, d, device=dev) for _ in range(K)]
    dg = [torch.empty(d, device=dev) for _ in range(K)]
    call = lambda: sr.solo_readout_fwd_bwd_private(dims, hidden, gs, Ws, targets, None, loss_tok,
                                                   loss_mean, dh, dW, dg, ws, stream=stream)
    clk = ClockSampler(dev.index).__enter__()
    time.sleep(1.0)
    for _ in range(max(args.warmup, 0)):
        call()
    torch.cuda.synchronize(dev)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    launches0 = sr.solo_readout_kernel_launches()
    clk.mark_start()
    t0.record(stream)
    for _ in range(args.steps):
        call()
    t1.record(stream)
    launches = sr.solo_readout_kernel_launches() - launches0
    torch.cuda.synchronize(dev)
    clk.mark_end()
    clk.__exit__(None, None, None)
    ms = t0.elapsed_time(t1)
    peaks, peak_src = load_peaks()
    peak, peak_name = tensor_peak(peaks, peak_src, ms / 1e3)
    algo = 3 * K * costmodel.gemm_flops(N, V, d)      # per module: logits, dX, dW_k
    tflops = algo / (ms / args.steps / 1e3) / 1e12
    line = {"metric": PRIVATE_METRIC, "value": job_throughput(wl.M, args.steps, 1, ms),
            "unit": "tokens/s", "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": ms / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic", "mode": "private",
            "config": {"workload": wl.name, "K": K, "N": N, "d": d, "V": V,
                       "parallelism": "replicas1", "l2": l2_note(wl, True)},
            "algo_tflops": tflops,
            "algo_frac_of_peak": tflops / peak,
            "peak_source": peak_name,
            "clocks": clk.summary(), "gpu_launches": launches,
            "device_flags": sr.solo_readout_get_flags(ws, stream)}
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    wl = workload_from_name(args.workload)
    if args.warmup < 0 or args.steps < 1:
        raise SystemExit("need --steps >= 1")
    if args.impl == "reference":
        run_reference(args, wl)
    elif args.mode == "exit":
        run_exit_bench(args, wl)
    elif args.mode == "private":
        run_private_bench(args, wl)
    else:
        run_ours(args, wl)


if __name__ == "__main__":
    main()
