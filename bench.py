"""Benchmark of one draft-tree verify step (GRIFFIN, arXiv 2502.11018).

    python bench.py [--gpus N] [--steps K] [--warmup W] [--config NAME] [--impl ours|reference]

A step is one pass of the whole verify path over one seeded synthetic batch:
tree build, tree attention for every layer, LM head + argmax (or logits for
T = 1), acceptance and KV compaction, all through the C ABI of libgv.so,
replayed as one CUDA graph.  The default workload is the LLaMA-3-8B shaped
step (32 layers, GQA 32/8 x 128, prefix 4096, vocab 128256, 60-node tree of
depth 8).  Its working set (1.6 GB of weights and caches) is far above the
129 MB L2, so no L2 flush is needed between steps.

Prints one JSON line (rank 0).  Under torchrun with N > 1 every rank runs an
independent replica of the step on its own GPU (the verify path of one
decoding stream does not shard: replicas only), and `value` is the total over
ranks divided by the slowest rank's time.
"""

import argparse
import contextlib
import ctypes
import hashlib
import json
import os
import platform
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

import torch  # noqa: E402

from paper_2502_11018_gb300 import build as gv_build  # noqa: E402
from paper_2502_11018_gb300 import gv, inputs  # noqa: E402

METRIC = "verify steps/s and accepted tok/s (LLaMA-3-8B shape, 60-node tree); % HBM roofline"
UNIT = "verify_steps/s"
# DRAM bytes per launch (dram__bytes_read.sum + dram__bytes_write.sum) from one
# ncu capture, keyed by (kernel, workload), with the SHA-256 of the kernel's
# source files at capture time: when the sources have changed since, the
# figure no longer describes the kernel and the line reports null.
TRAFFIC = {
    # tree_prep_kernel + attn_layers_kernel of one gv_verify_attention_layers
    # call over the 32 layers (23.6 MB + 577.3 MB), per layer
    ("verify_attention", "llama3_8b"): {
        "bytes": 18778672,
        "sources": ["paper_2502_11018_gb300/csrc/attention_layers_sm103.cu",
                    "paper_2502_11018_gb300/csrc/attn_common.cuh", "paper_2502_11018_gb300/csrc/sm103.cuh"],
        "sha256": "9f530270965a268f699ed610bc391db4cac47cfd852901e7c9f828a0de29b2f3"},
    ("lmhead_select", "llama3_8b"): {
        "bytes": 1058401280,
        "sources": ["paper_2502_11018_gb300/csrc/lmhead_sm103.cu", "paper_2502_11018_gb300/csrc/sm103.cuh"],
        "sha256": "67e6139a14cf3f2221a497fbc99ff4c54a1f111451c6cea1c8969d9b5fd805d7"},
}
OTHER_CONFIGS = ("llama2_7b", "llama2_13b_b4", "mixtral_attn", "tiny_f32")


def sources_sha256(files):
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()


def traffic_of(kernel, workload):
    e = TRAFFIC.get((kernel, workload))
    if e is None:
        return None
    try:
        return e["bytes"] if sources_sha256(e["sources"]) == e["sha256"] else None
    except OSError:
        return None


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            p = json.load(f)
        return {"hbm_gbs": float(p["hbm_gbs"]), "source": "measured"}
    except Exception:
        return {"hbm_gbs": 6800.0, "source": "fallback"}


def step_bytes(cfg, accept_len):
    """Algorithmic HBM bytes of one step: what the method must move once."""
    es = 2 if cfg["dtype"] == "bf16" else 4
    L, B, N, H, V = cfg["L"], cfg["B"], cfg["N"], cfg["H"], cfg["V"]
    Hq, Hkv, d = cfg["Hq"], cfg["Hkv"], cfg["d"]
    attn = 0
    for P in cfg["P"]:
        attn += 2 * P * Hkv * d * es                       # prefix K and V, read once
    attn += B * N * (Hq + 2 * Hkv) * d * es               # tree q, k, v read
    attn += B * N * Hq * d * es + 2 * B * N * Hkv * d * es  # output + tree K/V scratch written
    attn *= L
    lm = V * H * es + B * N * H * es                      # W once, hidden states
    if cfg.get("temperature", 0.0) > 0:
        lm += B * N * V * 4                               # fp32 logits written
        lm += 2 * B * N * V * 4                           # target + draft logits read by accept
    else:
        lm += B * N * 8
    compact = 2 * 2 * int(sum(accept_len)) * Hkv * d * es * L   # K,V rows read + written
    return {"attention": attn, "lmhead": lm, "compact": compact,
            "total": attn + lm + compact + B * N * 64}


def attention_bytes(cfg):
    """Algorithmic HBM bytes of one gv_verify_attention launch (one layer):
    the prefix K/V read once, the tree's q/k/v read, the output and the rotated
    tree K/V written, plus the per-node RoPE rows and ancestor masks."""
    es = 2 if cfg["dtype"] == "bf16" else 4
    B, N, Hq, Hkv, d = cfg["B"], cfg["N"], cfg["Hq"], cfg["Hkv"], cfg["d"]
    b = sum(2 * P * Hkv * d * es for P in cfg["P"])
    b += B * N * (Hq + 2 * Hkv) * d * es                  # q, k_new, v_new
    b += B * N * Hq * d * es + 2 * B * N * Hkv * d * es    # out, tree K/V
    b += B * N * (d // 2) * 2 * 4 + B * N * 8              # RoPE rows, ancestor masks
    return b


def attention_splits(cfg):
    """Key splits per attention unit, the rule the library applies: as many as
    fit the SMs in one wave (at most 16, at least 4 when the cache holds 4096
    keys or more, never more than a unit's blocks)."""
    tiles = (cfg["G"] * cfg["N"] + 127) // 128 if "G" in cfg else (cfg["Hq"] // cfg["Hkv"] * cfg["N"] + 127) // 128
    units = cfg["B"] * cfg["Hkv"] * tiles
    c = torch.cuda.get_device_properties(0).multi_processor_count // units
    if cfg["S_max"] >= 4096 and c < 4:
        c = 4
    c = min(c, (cfg["S_max"] + 127) // 128 + 1, 16)
    return max(c, 1)


def layers_call(cfg):
    """Whether the step runs every layer's attention in one
    gv_verify_attention_layers call (bf16, d = 128, G * N <= 256, B <= 64)."""
    G = cfg["Hq"] // cfg["Hkv"]
    return cfg["dtype"] == "bf16" and cfg["d"] == 128 and G * cfg["N"] <= 256 and cfg["B"] <= 64


def launches_per_step(cfg):
    """Kernels of this library one step launches: tree build, RoPE table, the
    attention (one multi-layer call -- its rotation pass and the persistent
    kernel -- on the bf16 path; otherwise one rotation of every layer's
    queries and tree keys -- two launches -- then split attention + merge per
    layer, no merge when a unit has a single split; rotate + split + combine
    per layer on the fp32 path), LM head + merge, accept, compaction."""
    if layers_call(cfg):
        return 2 + 2 + 2 + 1 + 1
    if cfg["dtype"] == "bf16":
        per_layer = 1 if attention_splits(cfg) == 1 else 2
        rotate = 2 if cfg["d"] == 128 else 0
    else:
        per_layer = 3
        rotate = 0
    return 2 + rotate + per_layer * cfg["L"] + 2 + 1 + 1


def lmhead_bytes(cfg):
    es = 2 if cfg["dtype"] == "bf16" else 4
    B, N, H, V = cfg["B"], cfg["N"], cfg["H"], cfg["V"]
    b = V * H * es + B * N * H * es
    if cfg.get("temperature", 0.0) > 0:
        b += B * N * V * 4
    return b


class NvmlClocks:
    """SM clock and clock-event reasons of the benchmark's GPU, read through
    NVML (read-only queries, through ctypes) by a background thread about
    every half millisecond; samples taken between start() and stop() count."""

    REASONS = {0x8: "hw_slowdown", 0x40: "hw_thermal_slowdown", 0x20: "sw_thermal_slowdown",
               0x4: "sw_power_cap"}
    NVML_CLOCK_SM = 1

    def __init__(self, device_index):
        self.lib = self.h = None
        self.samples = []
        self.window = None
        self._stop = threading.Event()
        self._thread = None
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            uuid = getattr(torch.cuda.get_device_properties(device_index), "uuid", None)
            ok = False
            if uuid is not None:
                u = str(uuid)
                u = u if u.startswith("GPU-") else "GPU-" + u
                ok = lib.nvmlDeviceGetHandleByUUID(u.encode(), ctypes.byref(h)) == 0
            if not ok and lib.nvmlDeviceGetHandleByIndex_v2(device_index, ctypes.byref(h)) != 0:
                return
            self.reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                lib.nvmlDeviceGetCurrentClocksThrottleReasons
            self.lib, self.h = lib, h
        except (OSError, AttributeError):
            self.lib = None

    def _run(self):
        clk, rs = ctypes.c_uint(), ctypes.c_ulonglong()
        while not self._stop.is_set():
            if self.lib.nvmlDeviceGetClockInfo(self.h, self.NVML_CLOCK_SM, ctypes.byref(clk)) == 0 and \
                    self.reasons_fn(self.h, ctypes.byref(rs)) == 0:
                self.samples.append((time.perf_counter(), clk.value, rs.value))
            time.sleep(0.0005)

    def begin(self):
        """Start sampling (before the region, so the thread is running)."""
        if self.lib is None:
            return
        self._thread = threading.Thread(target=self._run, daemon=True)
        self._thread.start()
        time.sleep(0.005)

    def start(self):
        self.window = [time.perf_counter(), None]

    def stop(self):
        if self.window is not None:
            self.window[1] = time.perf_counter()

    def end(self):
        if self._thread is None or self.window is None:
            return None
        self._stop.set()
        self._thread.join(timeout=5)
        t0, t1 = self.window
        inside = [x for x in self.samples if t0 <= x[0] <= t1]
        if not inside:
            return None
        mx = ctypes.c_uint()
        self.lib.nvmlDeviceGetMaxClockInfo(self.h, self.NVML_CLOCK_SM, ctypes.byref(mx))
        reasons = sorted({n for _, _, r in inside for bit, n in self.REASONS.items() if r & bit})
        return {"sm_mhz": statistics.median(c for _, c, _ in inside), "sm_max_mhz": float(mx.value),
                "reasons": reasons, "samples": len(inside), "source": "nvml"}


class ClockSampler:
    """nvidia-smi clocks / throttle reasons sampled during the timed region
    (used where NVML cannot be loaded)."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index):
        self.gpu = gpu_index
        self.proc = None
        self.lines = []

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except Exception:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except Exception:
            self.proc.kill()
            out, _ = self.proc.communicate()
        sm, mx, reasons = [], 0.0, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in out.strip().splitlines():
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx = max(mx, float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def graph_of(fn):
    """CUDA graph of one call of `fn` (host launch overhead out of the timing)."""
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        fn()
    torch.cuda.current_stream().wait_stream(s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        fn()
    return g


def event_time_ms(fn, iters, stream):
    start = torch.cuda.Event(enable_timing=True)
    end = torch.cuda.Event(enable_timing=True)
    start.record(stream)
    for _ in range(iters):
        fn()
    end.record(stream)
    end.synchronize()
    return start.elapsed_time(end) / iters


def replay_times_ms(fn, iters, stream, flush=None):
    """Time `iters` calls with one event pair each (events on the launching
    stream): the mean and each call's time.  Back to back, the mean is over
    the whole region; with `flush` (run between calls, outside the pairs: an
    L2 flush for a working set that fits in L2) it is the mean of the calls."""
    if flush is None:
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(iters + 1)]
        ev[0].record(stream)
        for i in range(iters):
            fn()
            ev[i + 1].record(stream)
        ev[-1].synchronize()
        per = [ev[i].elapsed_time(ev[i + 1]) for i in range(iters)]
        return ev[0].elapsed_time(ev[-1]) / iters, per
    pairs = []
    for _ in range(iters):
        flush()
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        pairs.append((a, b))
    pairs[-1][1].synchronize()
    per = [a.elapsed_time(b) for a, b in pairs]
    return sum(per) / iters, per


def percentiles(per):
    q = sorted(per)

    def at(f):
        return q[min(len(q) - 1, max(0, int(round(f * (len(q) - 1)))))]
    return {"ms_p10": at(0.10), "ms_p50": at(0.50), "ms_p90": at(0.90)}


def cpu_model():
    """The host CPU's model name (lscpu, else /proc/cpuinfo, else the machine)."""
    try:
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.startswith("Model name:"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if line.lower().startswith("model name"):
                    return line.split(":", 1)[1].strip()
    except OSError:
        pass
    return platform.machine()


def _openblas_thread_apis():
    """(set, get) thread-count functions of every OpenBLAS library loaded in
    this process (numpy's BLAS), for hosts without threadpoolctl."""
    names = [("openblas_set_num_threads", "openblas_get_num_threads"),
             ("scipy_openblas_set_num_threads64_", "scipy_openblas_get_num_threads64_"),
             ("openblas_set_num_threads64_", "openblas_get_num_threads64_"),
             ("scipy_openblas_set_num_threads", "scipy_openblas_get_num_threads")]
    apis = []
    try:
        paths = set()
        with open("/proc/self/maps") as f:
            for line in f:
                parts = line.split()
                if len(parts) >= 6 and "openblas" in parts[-1].lower():
                    paths.add(parts[-1])
        for path in sorted(paths):
            lib = ctypes.CDLL(path)
            for sn, gn in names:
                if hasattr(lib, sn) and hasattr(lib, gn):
                    apis.append((getattr(lib, sn), getattr(lib, gn)))
                    break
    except OSError:
        pass
    return apis


@contextlib.contextmanager
def blas_threads(n):
    """Run the block with numpy's BLAS and torch's CPU ops on n threads."""
    import numpy  # noqa: F401  (loads the BLAS library)
    prev_torch = torch.get_num_threads()
    torch.set_num_threads(n)
    try:
        try:
            from threadpoolctl import threadpool_limits
        except ImportError:
            threadpool_limits = None
        if threadpool_limits is not None:
            with threadpool_limits(n):
                yield
        else:
            apis = _openblas_thread_apis()
            prev = [g() for _, g in apis]
            for sfn, _ in apis:
                sfn(n)
            try:
                yield
            finally:
                for (sfn, _), v in zip(apis, prev):
                    sfn(v)
    finally:
        torch.set_num_threads(prev_torch)


def oracle_full_step(host_inp):
    """Seconds the float64 oracle takes for one whole verify step: tree build,
    every layer's tree attention, the whole LM head, acceptance and the
    compaction of every layer's cache."""
    import oracle
    t0 = time.perf_counter()
    oracle.verify_step(host_inp)
    return time.perf_counter() - t0


def full_step_desc(cfg):
    return (f"one whole step of the float64 numpy oracle: tree build, all {cfg['L']} layers' tree attention, "
            f"the LM head over all {cfg['V']} vocabulary rows, acceptance and the compaction of every layer's "
            f"cache (inputs converted from the device copies inside the timing)")


def host_inputs(cfg, seed, layers, dev_inp=None):
    """Host copy of the first `layers` layers of the workload (from the device
    inputs when given, else generated on the host)."""
    if dev_inp is None:
        return inputs.make_step_inputs(cfg, seed, device="cpu", layers=layers)
    import dataclasses
    kw = {}
    for f in dataclasses.fields(dev_inp):
        v = getattr(dev_inp, f.name)
        if isinstance(v, torch.Tensor):
            v = v[:layers] if f.name in ("q", "k_new", "v_new", "cacheK", "cacheV") else v
            v = v.cpu()
        kw[f.name] = v
    return type(dev_inp)(**kw)


def cpu_baseline(cfg, seed, dev_inp=None):
    """The oracle as it stands, timed on the host cores: one whole step with
    every core, and one on a single thread."""
    inp = host_inputs(cfg, seed, cfg["L"], dev_inp)
    cores = len(os.sched_getaffinity(0))
    with blas_threads(cores):
        t_all = oracle_full_step(inp)
    with blas_threads(1):
        t_one = oracle_full_step(inp)
    return {"value": 1.0 / t_all, "unit": UNIT, "cores": cores, "kind": "oracle",
            "sample": full_step_desc(cfg) + f"; {t_all:.2f} s on {cores} threads, {t_one:.2f} s on 1 thread",
            "seconds_per_step": t_all, "seconds_per_step_1thread": t_one, "cpu_model": cpu_model()}


def bench_config(cfg, world):
    """The `config` object of the JSON line (both arms)."""
    return {"workload": cfg["name"], "batch": cfg["B"], "layers": cfg["L"],
            "hidden": cfg["H"], "heads_q": cfg["Hq"], "heads_kv": cfg["Hkv"],
            "head_dim": cfg["d"], "vocab": cfg["V"], "prefix": list(cfg["P"]),
            "tree_nodes": cfg["N"], "tree_depth": cfg["D"],
            "temperature": cfg.get("temperature", 0.0),
            "l2": "working set above L2 (no flush needed)", "parallelism": f"replicas{world}"}


def run_reference(args):
    """The reference arm: the float64 oracle on the host cores, every step one
    whole verify step of the workload.  Steps run until --steps or until about
    two minutes of steps have run; `steps` is the number that ran."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return
    cfg = inputs.config(args.config)
    inp = host_inputs(cfg, args.seed, cfg["L"])
    cores = len(os.sched_getaffinity(0))
    budget_s = 120.0
    wall0 = time.perf_counter()
    with blas_threads(cores):
        warm = min(args.warmup, 1)
        for _ in range(warm):
            oracle_full_step(inp)
        times = []
        t0 = time.perf_counter()
        while len(times) < max(1, args.steps):
            times.append(oracle_full_step(inp))
            if time.perf_counter() - t0 + statistics.mean(times) > budget_s:
                break
    wall = time.perf_counter() - wall0
    mean = statistics.mean(times)
    v = 1.0 / mean
    desc = full_step_desc(cfg) + f"; {len(times)} steps of {args.steps} requested (about {budget_s:.0f} s of steps)"
    line = {"metric": METRIC, "value": v, "unit": UNIT, "n_gpus": args.gpus, "steps": len(times),
            "steps_requested": args.steps, "warmup": warm, "ms_per_step": 1000.0 * mean,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded random weights, caches and draft trees)", "impl": "reference",
            "config": bench_config(cfg, args.gpus), **percentiles([1000.0 * t for t in times]),
            "cpu_baseline": {"value": v, "unit": UNIT, "cores": cores, "kind": "oracle", "sample": desc,
                             "cpu_model": cpu_model()},
            "e2e": {"value": v, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
            "wall_s": wall}
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=1000)
    ap.add_argument("--warmup", type=int, default=20)
    ap.add_argument("--config", default="llama3_8b", choices=sorted(inputs.CONFIGS))
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--seed", type=int, default=1000)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-other-configs", action="store_true",
                    help="measure only --config (not also the other workloads under `configs`)")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--layers", type=int, default=0,
                    help="--kernel attention_layers: layers of the call (default: the workload's)")
    ap.add_argument("--kernel", default="step", choices=["step", "lmhead", "attention", "attention_layers", "tat",
                                                           "forward", "tgf", "draft_tree"],
                    help="step: the benchmark; lmhead / attention: time that call alone "
                         "(a small, self-contained launch sequence for profiler captures); "
                         "attention_layers: one gv_verify_attention_layers call over --layers layers; "
                         "tat: one token-alignable training pass (gv_tat_loss) on a "
                         "4 x 2048-token batch, vocabulary 32000; forward: the whole verify "
                         "forward of the target (decoder layers around the path, random "
                         "weights of the --config model's shape); tgf: the draft model's "
                         "token-guided fusion (gv_tgf) over 60 rows, d 4096, expansion 11008; "
                         "draft_tree: one cycle's dynamic draft tree (6 top-10 expansion steps "
                         "over a 128256-token vocabulary, rerank to 60 nodes)")
    args = ap.parse_args()
    args.warmup = max(args.warmup, 3) if args.impl == "ours" else args.warmup

    if args.impl == "reference":
        run_reference(args)
        return

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)
    if rank == 0:
        gv_build.build()
    if dist is not None:
        dist.barrier()
    gv.lib()

    from paper_2502_11018_gb300.step import VerifyStep
    if args.kernel == "tat":
        run_tat(args, dev)
        return
    if args.kernel == "forward":
        run_forward(args, dev)
        return
    if args.kernel == "tgf":
        run_tgf(args, dev)
        return
    if args.kernel == "draft_tree":
        run_draft_tree(args, dev)
        return
    cfg = inputs.config(args.config)
    if args.kernel == "attention_layers":
        run_attention_layers(args, cfg, dev)
        return
    if args.kernel != "step":
        run_kernel_only(args, cfg, dev)
        return
    inp = inputs.make_step_inputs(cfg, args.seed + rank, device=dev)
    step = VerifyStep(inp)
    step.capture()
    stream = torch.cuda.current_stream()
    for _ in range(args.warmup):
        step.replay()
    torch.cuda.synchronize()

    clocks = NvmlClocks(local)
    smi = None
    if clocks.lib is None:
        smi = ClockSampler(local)
    clocks.begin()
    if dist is not None:
        dist.barrier()
    torch.cuda.synchronize()
    if smi is not None:
        smi.start()
    flush, l2_note = l2_flush_for(cfg, dev)
    clocks.start()
    ms, per = replay_times_ms(step.replay, args.steps, stream, flush)
    torch.cuda.synchronize()
    clocks.stop()
    if dist is not None:
        dist.barrier()
    clk = smi.stop() if smi is not None else clocks.end()
    accept_len = step.accept_len.cpu().tolist()
    t_max = ms
    if dist is not None:
        t = torch.tensor([ms], device=dev)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        t_max = float(t.item())

    kernels = kernel_times(step, cfg, stream)
    peaks = load_peaks()
    dom = max(kernels, key=lambda k: kernels[k]["ms_per_launch"] * kernels[k]["launches_per_step"])
    dk = kernels[dom]
    sb = step_bytes(cfg, accept_len)
    step_gbs = sb["total"] / (t_max * 1e-3) / 1e9

    # End to end through the public API with host buffers: pinned host inputs
    # copied in, step, result read back, every step.
    e2e = e2e_measure(step, inp, args.e2e_steps, stream)

    line = {
        "metric": METRIC, "value": world * 1000.0 / t_max, "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": t_max, **percentiles(per),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": cfg["dtype"],
        "data": "synthetic (seeded random weights, caches and draft trees)",
        "config": {**bench_config(cfg, world), "l2": l2_note},
        "accepted_tok_per_s": world * sum(accept_len) * 1000.0 / t_max,
        "accept_len": accept_len,
        "hbm_roofline": {"step_bytes": sb["total"], "achieved_gbs": step_gbs,
                         "peak_gbs": peaks["hbm_gbs"], "frac": step_gbs / peaks["hbm_gbs"],
                         "peak_source": peaks["source"]},
        "roofline": {"kernel": dom, "bound": "hbm", "achieved": dk["achieved_gbs"],
                     "peak": peaks["hbm_gbs"], "unit": "GB/s",
                     "frac": dk["achieved_gbs"] / peaks["hbm_gbs"], "traffic": traffic_of(dom, cfg["name"]),
                     "ms_per_launch": dk["ms_per_launch"], "peak_source": peaks["source"]},
        "kernels": kernels,
        "gpu_launches": launches_per_step(cfg) * args.steps,
        "e2e": e2e,
        "clocks": clk,
    }
    del step, inp
    torch.cuda.empty_cache()
    if not args.no_other_configs:
        # The other workloads, each measured the same way in this process
        # (per-replay events over max(--steps, 20) graph replays).
        line["configs"] = {name: measure_config(name, args.seed + rank, max(args.steps, 20), args.warmup, dev,
                                                stream, peaks)
                           for name in OTHER_CONFIGS}
    if rank == 0 and not args.no_cpu_baseline:
        cb = cpu_baseline(cfg, args.seed)
        line["cpu_baseline"] = {k: cb[k] for k in ("value", "unit", "cores", "kind", "sample",
                                                   "seconds_per_step_1thread", "cpu_model")}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


def kernel_times(step, cfg, stream):
    """The two kernels that dominate a step, each timed alone (replayed from a
    CUDA graph on the stream it is launched on): the LM head, and the
    attention layers in order as the step runs them (the layers' caches cycle
    through far more than L2 holds)."""
    L = cfg["L"]
    g_lm = graph_of(lambda: step.lmhead(torch.cuda.current_stream()))
    lm_ms = event_time_ms(g_lm.replay, 20, stream)
    g_attn = graph_of(lambda: (step.attention_layers(torch.cuda.current_stream()),
                               step.join_merges(torch.cuda.current_stream())))
    attn_ms = event_time_ms(g_attn.replay, 10, stream) / L
    peaks = load_peaks()
    lm_gbs = lmhead_bytes(cfg) / (lm_ms * 1e-3) / 1e9
    attn_gbs = attention_bytes(cfg) / (attn_ms * 1e-3) / 1e9
    return {
        "lmhead_select": {"ms_per_launch": lm_ms, "launches_per_step": 1, "algorithmic_bytes": lmhead_bytes(cfg),
                          "achieved_gbs": lm_gbs, "frac": lm_gbs / peaks["hbm_gbs"]},
        "verify_attention": {"ms_per_launch": attn_ms, "launches_per_step": L,
                             "algorithmic_bytes": attention_bytes(cfg), "achieved_gbs": attn_gbs,
                             "frac": attn_gbs / peaks["hbm_gbs"]},
    }


def l2_flush_for(cfg, dev):
    """(flush, note): a working set that fits in the 129 MB L2 (the tiny
    workload) is flushed between replays by writing a 512 MB buffer."""
    if step_bytes(cfg, [cfg["D"]] * cfg["B"])["total"] >= 256 * 2**20:
        return None, "working set above L2 (no flush needed)"
    junk = torch.empty(512 * 2**20, dtype=torch.uint8, device=dev)
    return (lambda: junk.fill_(1)), "flushed between replays (512 MB write, outside the timed pairs)"


def measure_config(name, seed, steps, warmup, dev, stream, peaks):
    """One workload's step: per-replay times of its CUDA graph, throughput,
    HBM roofline fraction of the step and of its two dominant kernels."""
    from paper_2502_11018_gb300.step import VerifyStep
    cfg = inputs.config(name)
    inp = inputs.make_step_inputs(cfg, seed, device=dev)
    step = VerifyStep(inp)
    step.capture()
    for _ in range(max(warmup, 3)):
        step.replay()
    torch.cuda.synchronize()
    flush, note = l2_flush_for(cfg, dev)
    config = bench_config(cfg, 1)
    config["l2"] = note
    ms, per = replay_times_ms(step.replay, steps, stream, flush)
    accept_len = step.accept_len.cpu().tolist()
    sb = step_bytes(cfg, accept_len)
    gbs = sb["total"] / (ms * 1e-3) / 1e9
    out = {"ms_per_step": ms, **percentiles(per), "steps": steps, "verify_steps_per_s": 1000.0 / ms,
           "accepted_tok_per_s": sum(accept_len) * 1000.0 / ms, "accept_len": accept_len, "dtype": cfg["dtype"],
           "config": config, "gpu_launches_per_step": launches_per_step(cfg),
           "hbm_roofline": {"step_bytes": sb["total"], "achieved_gbs": gbs, "frac": gbs / peaks["hbm_gbs"],
                            "peak_gbs": peaks["hbm_gbs"], "peak_source": peaks["source"]},
           "kernels": kernel_times(step, cfg, stream)}
    del step, inp
    torch.cuda.empty_cache()
    return out


def run_kernel_only(args, cfg, dev):
    """Time one call of the verify path alone (one layer for attention), on a
    workload whose inputs hold only that call's tensors."""
    from paper_2502_11018_gb300.step import VerifyStep
    # Attention cycles through all layers so that its caches are read from HBM.
    layers = 1 if args.kernel == "lmhead" else cfg["L"]
    inp = inputs.make_step_inputs(cfg, args.seed, device=dev, layers=layers)
    step = VerifyStep(inp)
    step.tree()
    stream = torch.cuda.current_stream()
    it = [0]

    def attn():
        step.attention(it[0] % layers)
        it[0] += 1

    fn = step.lmhead if args.kernel == "lmhead" else attn
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    ms = event_time_ms(fn, args.steps, stream)
    # The same launches replayed from a CUDA graph (no host launch overhead).
    per_graph = 1 if args.kernel == "lmhead" else layers
    g = graph_of(lambda: [fn() for _ in range(per_graph)])
    g.replay()
    torch.cuda.synchronize()
    ms_graph = event_time_ms(g.replay, max(1, args.steps // per_graph), stream) / per_graph
    if args.kernel == "lmhead":
        nbytes = lmhead_bytes(cfg)
    else:
        es = 2 if cfg["dtype"] == "bf16" else 4
        B, N, Hq, Hkv, d = cfg["B"], cfg["N"], cfg["Hq"], cfg["Hkv"], cfg["d"]
        nbytes = attention_bytes(cfg)
    peaks = load_peaks()
    gbs_graph = nbytes / (ms_graph * 1e-3) / 1e9
    print(json.dumps({"kernel": args.kernel, "workload": cfg["name"], "ms_per_call_eager": ms,
                      "ms_per_call_graph": ms_graph, "algorithmic_bytes": nbytes,
                      "achieved_gbs_graph": gbs_graph,
                      "frac_of_measured_hbm_graph": gbs_graph / peaks["hbm_gbs"]}), flush=True)


def run_attention_layers(args, cfg, dev):
    """One gv_verify_attention_layers call over the first --layers layers of
    the workload (its rotation pass and the persistent attention kernel),
    replayed from a CUDA graph; calls cycle over two copies of the caches
    when one copy fits in L2."""
    from paper_2502_11018_gb300.step import VerifyStep
    layers = args.layers if args.layers > 0 else cfg["L"]
    inp = inputs.make_step_inputs(cfg, args.seed, device=dev, layers=layers)
    step = VerifyStep(inp)
    if not step.layers_call:
        raise SystemExit(f"{cfg['name']}: no multi-layer attention for this shape")
    step.tree()
    stream = torch.cuda.current_stream()
    fn = lambda: step.attention_layers(torch.cuda.current_stream())  # noqa: E731
    for _ in range(args.warmup):
        fn()
    torch.cuda.synchronize()
    g = graph_of(fn)
    g.replay()
    torch.cuda.synchronize()
    reps = max(3, min(args.steps, 200))
    ms = event_time_ms(g.replay, reps, stream)
    nbytes = attention_bytes(cfg) * layers
    peaks = load_peaks()
    gbs = nbytes / (ms * 1e-3) / 1e9
    print(json.dumps({"kernel": "attention_layers", "workload": cfg["name"], "layers": layers,
                      "ms_per_call_graph": ms, "us_per_layer": ms * 1e3 / layers, "algorithmic_bytes": nbytes,
                      "achieved_gbs_graph": gbs, "frac_of_measured_hbm_graph": gbs / peaks["hbm_gbs"]}), flush=True)


def forward_bytes(cfg, F, accept_len):
    """Algorithmic bytes of the whole verify forward: every weight read once
    (per layer Q/K/V/O, gate/up, down and the two norms; the final norm), the
    verify path's own bytes (prefix K/V, LM head weight, compaction), and the
    node activations each layer writes and reads back (x, q/k/v, attention
    output, h twice, the MLP hidden)."""
    es = 2
    L, B, N, H, Hq, Hkv, d = cfg["L"], cfg["B"], cfg["N"], cfg["H"], cfg["Hq"], cfg["Hkv"], cfg["d"]
    R = B * N
    weights = L * es * (H * (Hq + 2 * Hkv) * d + Hq * d * H + 3 * H * F + 2 * H) + es * H
    acts = L * R * es * (2 * H + (2 * Hq + 2 * Hkv) * d + 4 * H + 2 * F + 2 * H)
    return weights + acts + step_bytes(cfg, accept_len)["total"]


def run_forward(args, dev):
    """The whole verify forward of the --config target, timed from a CUDA graph
    with inputs (14 GB of LLaMA-3-8B-shaped weights) resident in HBM."""
    from paper_2502_11018_gb300.forward import VerifyForward
    cfg = inputs.config(args.config)
    inp = inputs.make_step_inputs(cfg, args.seed, device=dev)
    fw = inputs.make_forward_weights(cfg, args.seed, device=dev)
    fwd = VerifyForward(inp, fw)
    fwd.capture()
    stream = torch.cuda.current_stream()
    for _ in range(max(args.warmup, 3)):
        fwd.replay()
    torch.cuda.synchronize()
    steps = max(3, min(args.steps, 100))
    ms = event_time_ms(fwd.replay, steps, stream)
    alen = fwd.step.accept_len.cpu().numpy()
    nbytes = forward_bytes(cfg, fw.F, alen)
    peaks = load_peaks()
    gbs = nbytes / (ms * 1e-3) / 1e9
    print(json.dumps({"kernel": "forward", "workload": cfg["name"], "ffn": fw.F, "layers": cfg["L"],
                      "ms_per_step": ms, "verify_steps_per_s": 1e3 / ms,
                      "accepted_tok_per_s": float(alen.sum()) * 1e3 / ms, "algorithmic_bytes": nbytes,
                      "achieved_gbs": gbs, "frac_of_measured_hbm": gbs / peaks["hbm_gbs"],
                      "data": "synthetic (seeded random weights, caches and draft trees)"}), flush=True)


def tat_bytes(cfg):
    """Algorithmic bytes of one token-alignable training pass: every logit and
    both feature rows read once, the tokens, the earlier passes' masks, and
    the per-position outputs (two masks, the loss) plus the sequence losses."""
    B, T, V, H, n = cfg["B"], cfg["T"], cfg["V"], cfg["H"], cfg["n"]
    el = 2 if cfg["logits"] == "bf16" else 4
    ef = 2 if cfg["feat"] == "bf16" else 4
    rows = B * T
    return rows * (V * el + 2 * H * ef + 4 + (n - 1) + 1 + 1 + 4) + 4 * B


def run_tat(args, dev):
    """One token-alignable training pass over the LLaMA-2-7B-sized batch, timed
    from a CUDA graph of back-to-back calls (the 1.2 GB of inputs are far above
    L2, so every call reads them from HBM)."""
    cfg = inputs.TAT_CONFIGS["tat_llama2_7b"]
    inp = inputs.make_tat_inputs(cfg, args.seed, device=dev)
    B, T = cfg["B"], cfg["T"]
    mbar = torch.zeros((B, T), dtype=torch.uint8, device=dev)
    mask = torch.zeros((B, T), dtype=torch.uint8, device=dev)
    ell = torch.zeros((B, T), dtype=torch.float32, device=dev)
    seq = torch.zeros((B,), dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream()

    def call():
        gv.gv_tat_loss(inp.logits, inp.tokens, inp.feat_draft, inp.feat_target, cfg["k"], cfg["n"],
                       inp.mbar_prev, mbar, mask, ell, seq)

    for _ in range(args.warmup):
        call()
    torch.cuda.synchronize()
    reps = max(3, min(args.steps, 200))
    g = graph_of(lambda: [call() for _ in range(4)])
    g.replay()
    torch.cuda.synchronize()
    ms = event_time_ms(g.replay, reps, stream) / 4
    nbytes = tat_bytes(cfg)
    peaks = load_peaks()
    gbs = nbytes / (ms * 1e-3) / 1e9
    line = {"kernel": "tat", "workload": "tat_llama2_7b", "config": cfg, "ms_per_call_graph": ms,
            "algorithmic_bytes": nbytes, "achieved_gbs_graph": gbs,
            "frac_of_measured_hbm_graph": gbs / peaks["hbm_gbs"], "rows_per_s": B * T / (ms * 1e-3)}
    if not args.no_cpu_baseline:
        # The float64 oracle on the host cores, on the first 256 positions of
        # every sequence (the alignment mask needs whole chains), scaled to
        # the whole pass.
        import oracle
        ts = 256
        f = lambda t: t[:, :ts].detach().cpu().double().numpy()
        t0 = time.perf_counter()
        oracle.tat_pass(f(inp.logits), inp.tokens[:, :ts].cpu().numpy(), f(inp.feat_draft), f(inp.feat_target),
                        cfg["k"], cfg["n"], inp.mbar_prev[:, :, :ts].cpu().numpy())
        sec = (time.perf_counter() - t0) * (T / ts)
        line["cpu_baseline"] = {"value": B * T / sec, "unit": "rows/s", "cores": os.cpu_count(),
                                "kind": "oracle",
                                "sample": f"float64 numpy oracle on {B} x {ts} of the {B} x {T} positions, "
                                          f"scaled linearly ({sec:.2f} s per pass)"}
    print(json.dumps(line), flush=True)


def tgf_bytes(cfg):
    """Algorithmic bytes of one token-guided fusion call: the three weight
    matrices and the seven vectors read once, F and x read, h and o written."""
    rows, d, e = cfg["rows"], cfg["d"], cfg["e"]
    return 2 * (2 * d * d + 2 * d * e + d * e + 6 * d + e) + 2 * rows * d * 4


def run_tgf(args, dev):
    """gv_tgf on the LLaMA-2-7B drafter's shape (60 rows, d 4096, expansion
    11008), timed from a CUDA graph of back-to-back calls: the 337 MB of
    weights are far above L2, so every call streams them from HBM."""
    name = "tgf_llama2_7b"
    cfg = inputs.TGF_CONFIGS[name]
    ti = inputs.make_tgf_inputs(cfg, args.seed, device=dev)
    rows, d, e = cfg["rows"], cfg["d"], cfg["e"]
    h = torch.empty(rows, d, dtype=torch.bfloat16, device=dev)
    o = torch.empty(rows, d, dtype=torch.bfloat16, device=dev)
    ws = torch.empty(gv.gv_tgf_workspace(rows, d, e), dtype=torch.uint8, device=dev)
    stream = torch.cuda.current_stream()

    def call():
        gv.gv_tgf(ti.F, ti.x, ti.w, h, o, ws, stream=torch.cuda.current_stream())

    for _ in range(args.warmup):
        call()
    torch.cuda.synchronize()
    reps = max(3, min(args.steps, 200))
    g = graph_of(lambda: [call() for _ in range(4)])
    g.replay()
    torch.cuda.synchronize()
    ms = event_time_ms(g.replay, reps, stream) / 4
    nbytes = tgf_bytes(cfg)
    peaks = load_peaks()
    gbs = nbytes / (ms * 1e-3) / 1e9
    line = {"kernel": "tgf", "workload": name, "config": cfg, "ms_per_call_graph": ms, "launches_per_call": 5,
            "algorithmic_bytes": nbytes, "achieved_gbs_graph": gbs,
            "frac_of_measured_hbm_graph": gbs / peaks["hbm_gbs"], "rows_per_s": rows / (ms * 1e-3)}
    if not args.no_cpu_baseline:
        # the float64 oracle on the host cores, on 8 of the 60 rows (its cost
        # is the three float64 matrix products, linear in the rows), scaled
        import oracle
        rs = 8
        w = {k: v.detach().cpu().double().numpy() for k, v in ti.w.items()}
        t0 = time.perf_counter()
        oracle.tgf_forward(ti.F[:rs].cpu().double().numpy(), ti.x[:rs].cpu().double().numpy(), w)
        sec = (time.perf_counter() - t0) * (rows / rs)
        line["cpu_baseline"] = {"value": rows / sec, "unit": "rows/s", "cores": torch.get_num_threads(),
                                "kind": "oracle",
                                "sample": f"float64 numpy oracle on {rs} of the {rows} rows, scaled linearly "
                                          f"({sec:.2f} s per call)"}
    print(json.dumps(line), flush=True)


def draft_tree_bytes(cfg):
    """Algorithmic bytes of one draft-tree construction: every step's logits
    read once, the tree written."""
    B, k, D, V, N = cfg["B"], cfg["k"], cfg["D"], cfg["V"], cfg["N"]
    es = 2 if cfg["dtype"] == "bf16" else 4
    return B * (1 + (D - 1) * k) * V * es + B * N * 8


def run_draft_tree(args, dev):
    """One cycle's draft tree on the LLaMA-3-8B drafter's shape (top-10 per
    node, 6 steps, vocabulary 128256, 60 nodes), timed from a CUDA graph of
    back-to-back constructions with the steps' logits resident in HBM."""
    name = "draft_llama3_8b"
    cfg = inputs.DRAFT_CONFIGS[name]
    B, k, D, V, N = cfg["B"], cfg["k"], cfg["D"], cfg["V"], cfg["N"]
    root, steps = inputs.make_draft_logits(cfg, args.seed, device=dev)
    ws = torch.empty(gv.gv_draft_tree_workspace(B, k, D, V), dtype=torch.uint8, device=dev)
    parents = torch.zeros((B, N), dtype=torch.int32, device=dev)
    tokens = torch.zeros((B, N), dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    def call():
        st = torch.cuda.current_stream()
        for j in range(D):
            gv.gv_draft_tree_expand(j, k, D, steps[j], ws, root_token=root, stream=st)
        gv.gv_draft_tree_finish(k, D, V, parents, tokens, ws, stream=st)

    for _ in range(args.warmup):
        call()
    torch.cuda.synchronize()
    reps = max(3, min(args.steps, 200))
    g = graph_of(lambda: [call() for _ in range(4)])
    g.replay()
    torch.cuda.synchronize()
    ms = event_time_ms(g.replay, reps, stream) / 4
    nbytes = draft_tree_bytes(cfg)
    peaks = load_peaks()
    gbs = nbytes / (ms * 1e-3) / 1e9
    line = {"kernel": "draft_tree", "workload": name, "config": cfg, "us_per_tree": ms * 1e3,
            "launches_per_tree": 2 * D + 1, "algorithmic_bytes": nbytes, "achieved_gbs_graph": gbs,
            "frac_of_measured_hbm_graph": gbs / peaks["hbm_gbs"], "trees_per_s": B / (ms * 1e-3)}
    if not args.no_cpu_baseline:
        import oracle
        lg = [s.detach().cpu().float().numpy() for s in steps]
        t0 = time.perf_counter()
        for b in range(B):
            oracle.draft_tree(int(root[b]), [x[b] for x in lg], k, D, N)
        sec = time.perf_counter() - t0
        line["cpu_baseline"] = {"value": B / sec, "unit": "trees/s", "cores": torch.get_num_threads(),
                                "kind": "oracle", "sample": f"float64 numpy oracle on the whole workload "
                                                            f"({B} tree, {sec:.2f} s)"}
    print(json.dumps(line), flush=True)


def e2e_measure(step, inp, steps, stream):
    """Same metric through VerifyStep with host buffers: every step copies its
    inputs (tree, tokens, per-layer q/k/v, hidden states, uniforms) from pinned
    host memory -- the per-layer ones on a side stream, overlapping the earlier
    layers -- runs, and reads the accepted tokens back (one CUDA graph)."""
    host, pinned_out = step.host_buffers()
    h2d = sum(t.numel() * t.element_size() for t in host.values())
    d2h = pinned_out.numel() * pinned_out.element_size()
    g = step.capture_from_host(host, pinned_out)
    g.replay()
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        g.replay()
        torch.cuda.current_stream().synchronize()
    dt = (time.perf_counter() - t0) / steps
    return {"value": 1.0 / dt, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
            "ms_per_step": dt * 1000.0}


if __name__ == "__main__":
    main()
