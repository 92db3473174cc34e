#!/usr/bin/env python3
"""Throughput of the MoSA layer (forward + backward) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl mosa|reference]
                    [--config NAME] [--no-cpu-baseline]

A step is one forward and one backward pass of the layer over one batch of
the workload (default: B=4 sequences of T=4096 tokens, d=1024, H=8 heads of
size 64, k=2048 tokens per head, bf16 storage: the configuration with the
most work per step) with inputs resident in HBM.
L2 is flushed (a 256 MiB write) before every timed step, outside the step's
CUDA events.  Under torchrun every rank runs its own copy of the workload
(weak scaling, no collective on the data path); the reported time is the
maximum over ranks.

Rank 0 prints one JSON line: tokens/s, the roofline of the dominant kernel
(timed live with CUDA events on the library's stream, every 2nd timed step), the fp64 CPU oracle
timed on a bounded sample of the same workload, an end-to-end figure through
the public API with host buffers, SM clocks sampled during the timed region
and the number of library kernels launched.

``--impl reference`` times the CPU oracle (the only reference this layer
has) on the host cores instead.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import statistics
import subprocess
import sys
import tempfile
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "MoSA layer fwd+bwd tokens/s; achieved TFLOP/s and HBM GB/s vs GB300 peak"
L2_FLUSH_BYTES = 256 << 20
PROFILE_EVERY = 2   # timed steps per live timing of the dominant stage
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
                  "sm_max_mhz": 2070.0}
NUM_SM = 152
FP32_LANES_PER_SM = 128


def parse_args():
    p = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=10)
    p.add_argument("--impl", choices=["mosa", "reference"], default="mosa")
    p.add_argument("--config", default=None)
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--cpu-budget-s", type=float, default=15.0)
    p.add_argument("--rope", action="store_true",
                   help="rotary position encoding at the original positions (Sec. 2.2)")
    p.add_argument("--first-token", action="store_true",
                   help="every head keeps token 0 and selects k-1 more (Sec. 3.2)")
    p.add_argument("--dense-heads", type=int, default=0,
                   help="hybrid layer: this many dense heads beside the MoSA heads (Sec. 2.2)")
    p.add_argument("--window", type=int, default=0,
                   help="with --dense-heads: local heads over blocks of this many tokens "
                        "(Sec. 3.4); 0 = dense causal heads")
    p.add_argument("--profile-run", action="store_true",
                   help="for profilers: run --warmup then --steps plain layer steps (no "
                        "timing, stage profiling, graph or end-to-end passes) and exit")
    p.add_argument("--ingest-ncu", metavar="CSV", default=None,
                   help="turn an ncu CSV with dram__bytes_read/write.sum per kernel (taken on "
                        "this command's workload) into profiles/traffic.json and exit")
    return p.parse_args()


def load_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            d = json.load(f)
        return {k: float(d.get(k, FALLBACK_PEAKS[k])) for k in FALLBACK_PEAKS}, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


# ----------------------------------------------------------------- clocks

class ClockSampler:
    """nvidia-smi samples (200 ms) kept only while the timed region runs."""
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.lines: list[tuple[float, str]] = []
        self.window = (0.0, 0.0)

    def start(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (FileNotFoundError, OSError):
            self.proc = None
            return
        self.reader = threading.Thread(target=self._read, daemon=True)
        self.reader.start()
        time.sleep(0.6)

    def _read(self):
        for line in self.proc.stdout:
            self.lines.append((time.time(), line.strip()))

    def mark(self, t0, t1):
        self.window = (t0, t1)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.3)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        t0, t1 = self.window
        rows = [l for (t, l) in self.lines if t0 - 0.25 <= t <= t1 + 0.25]
        if not rows:
            rows = [l for (_, l) in self.lines]
        mhz, maxes, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for r in rows:
            f = [x.strip() for x in r.split(",")]
            if len(f) < 10:
                continue
            try:
                mhz.append(float(f[2]))
                maxes.append(float(f[3]))
            except ValueError:
                continue
            for name, val in zip(names, f[6:10]):
                if val.lower().startswith("active"):
                    reasons.add(name)
        if not mhz:
            return None
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": max(maxes),
                "reasons": sorted(reasons), "samples": len(mhz)}


# ------------------------------------------------------------ CPU oracle

def oracle_sample(cfg, x, n_seq):
    """Time the oracle's forward + backward on the first n_seq sequences (with
    the dense heads of a hybrid layer when x holds their weights)."""
    import oracle
    W = (x["Wr"], x["Wq"], x["Wk"], x["Wv"], x["Wo"])
    batches = list(range(n_seq))
    t0 = time.perf_counter()
    if "Dq" in x:
        D = (x["Dq"], x["Dk"], x["Dv"], x["Do"])
        _, I, _, _ = oracle.hybrid_forward(x["X"], *W, *D, k=cfg.k, window=x["window"],
                                           batches=batches, first_token=cfg.first_token,
                                           rope=cfg.rope)
        if cfg.backward:
            oracle.hybrid_backward(x["X"], *W, *D, I=I, dY=x["dY"], window=x["window"],
                                   batches=batches, rope=cfg.rope)
        return time.perf_counter() - t0
    _, I, _, _ = oracle.forward(x["X"], *W, k=cfg.k, batches=batches,
                                first_token=cfg.first_token, rope=cfg.rope)
    if cfg.backward:
        oracle.backward(x["X"], *W, I=I, dY=x["dY"], batches=batches, rope=cfg.rope)
    return time.perf_counter() - t0


def choose_sample(cfg, x, budget_s):
    t1 = oracle_sample(cfg, x, 1)
    n = int(max(1, min(cfg.B, budget_s // max(t1, 1e-6))))
    return n, t1


def single_thread_seconds():
    """The oracle on one host thread: the whole fp32 forward-only workload
    (B1 T256 d128 H4 k64) and the forward + backward of one sequence of
    B8 T1024 d512 H16 k128."""
    import oracle
    from paper_2505_00315_gb300 import workloads as W
    out = {}
    n0 = oracle.num_threads()
    oracle.set_num_threads(1)
    try:
        for name in ("f32_B1_T256_d128_H4_k64", "B8_T1024_d512_H16_k128"):
            c = W.CONFIGS[name]
            out[name] = {"seconds": round(oracle_sample(c, W.make_inputs(c), 1), 4),
                         "sample": ("forward" if not c.backward else "forward+backward") +
                                   " of 1 sequence"}
    finally:
        oracle.set_num_threads(n0)
    return out


def cpu_baseline(cfg, x, budget_s):
    import oracle
    n, t1 = choose_sample(cfg, x, budget_s)
    t = oracle_sample(cfg, x, n) if n > 1 else t1
    what = "forward+backward" if cfg.backward else "forward"
    return {"value": n * cfg.T / t, "unit": "tokens/s", "cores": oracle.num_threads(),
            "kind": "oracle",
            "sample": f"{what} of {n} of the {cfg.B} sequences of {cfg.name} "
                      f"(all heads, fp64, {t:.2f} s)",
            "single_thread": single_thread_seconds()}


# ------------------------------------------------------------ roofline

STAGES = ["router", "select", "qkv", "attn_fwd", "out", "out_bwd", "attn_bwd", "in_bwd",
          "w_bwd", "dwo", "fwd_unit", "bwd_unit"]


def stage_bound(stage, peaks, kind):
    """(bound, peak, unit) for a stage implemented as `kind` ('tensor', 'simt', 'mem')."""
    if kind == "mem":
        return "hbm", peaks["hbm_gbs"], "GB/s"
    if kind == "tensor":
        return "tensor", peaks["bf16_tflops_sustained"], "TFLOP/s"
    ffma = NUM_SM * FP32_LANES_PER_SM * 2 * peaks["sm_max_mhz"] * 1e6 / 1e12
    return "alu", ffma, "TFLOP/s"


def stage_kind(stage, lib_impl):
    return lib_impl.get(stage, "simt")


def traffic_for(stage, cfg_name):
    """DRAM bytes per step of `stage` from the committed ncu summary, or None
    when the summary is missing or was taken on a different kernel source."""
    path = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(path):
        return None
    with open(path) as f:
        d = json.load(f)
    ent = d.get(cfg_name, {}).get(stage)
    if not ent:
        return None
    if ent.get("source_sha256") != source_digest():
        return None
    return ent.get("bytes_per_step")


# Kernel name (as ncu prints it) -> bench stage.
KERNEL_STAGE = [("tc_gemm_kernel<5>", "router"), ("tc_gemm_kernel<(int)5>", "router"),
                ("pad_wr_kernel", "router"),
                ("topk_select", "select"), ("tc_gemm_kernel<0>", "qkv"),
                ("tc_gemm_kernel<(int)0>", "qkv"), ("attn_fwd", "attn_fwd"),
                ("tc_gemm_kernel<2>", "out_bwd"), ("tc_gemm_kernel<(int)2>", "out_bwd"),
                ("attn_bwd", "attn_bwd"), ("dq_finish", "attn_bwd"),
                ("scatter_product_kernel<0>", "in_bwd"), ("scatter_product_kernel<false>", "in_bwd"),
                ("scatter_product_kernel<(bool)0>", "in_bwd"),
                ("scatter_product_kernel<1>", "out"), ("scatter_product_kernel<true>", "out"),
                ("scatter_product_kernel<(bool)1>", "out"),
                ("head_sum_kernel<true>", "out"), ("head_sum_kernel<(bool)1>", "out"),
                ("head_sum_kernel<1>", "out"),
                ("tc_gemm_kernel<4>", "w_bwd"), ("tc_gemm_kernel<(int)4>", "w_bwd"),
                ("tc_gemm_kernel<6>", "w_bwd"), ("tc_gemm_kernel<(int)6>", "w_bwd"),
                ("tc_gemm_kernel<3>", "dwo"), ("tc_gemm_kernel<(int)3>", "dwo"),
                ("fused_fwd_kernel", "fwd_unit"), ("fused_bwd_kernel", "bwd_unit"),
                ("dense_rows", "select")]
# RoPE passes (rope_rows_kernel) run inside the qkv and attn_bwd stages alike,
# and the fp16 copies (to_f16_kernel) beside TopK on the side stream: both are
# left unattributed.


def ingest_ncu(csv_path, cfg_name):
    """DRAM bytes per step of each stage from an ncu CSV (one row per kernel
    launch and metric) into profiles/traffic.json.  A stage may launch several
    kernels a step (the large-k attention backward and its dQ split; both head
    groups of a hybrid layer); the steps are counted by the TopK launches, one
    per layer step."""
    import csv
    import collections
    per = collections.defaultdict(lambda: collections.defaultdict(float))
    steps = set()
    with open(csv_path) as f:
        lines = [l for l in f if not l.startswith("==")]
    for row in csv.DictReader(lines):
        name, metric = row.get("Kernel Name", ""), row.get("Metric Name", "")
        if "topk_select" in name:
            steps.add(row["ID"])
        if metric not in ("dram__bytes_read.sum", "dram__bytes_write.sum"):
            continue
        stage = next((st for key, st in KERNEL_STAGE if key in name), None)
        if stage is None:
            continue
        unit = row.get("Metric Unit", "byte")
        scale = {"byte": 1, "Kbyte": 1e3, "Mbyte": 1e6, "Gbyte": 1e9, "KB": 1e3, "MB": 1e6}.get(unit, 1)
        per[stage][row["ID"]] += float(row["Metric Value"].replace(",", "")) * scale
    path = os.path.join(ROOT, "profiles", "traffic.json")
    data = json.load(open(path)) if os.path.exists(path) else {}
    digest = source_digest()
    n_steps = max(1, len(steps))
    ent = {}
    for stage, launches in per.items():
        vals = list(launches.values())
        ent[stage] = {"bytes_per_step": sum(vals) / n_steps, "launches": len(vals),
                      "steps": n_steps, "source_sha256": digest}
    data[cfg_name] = ent
    with open(path, "w") as f:
        json.dump(data, f, indent=1, sort_keys=True)
    print(json.dumps({k: round(v["bytes_per_step"] / 1e6, 3) for k, v in ent.items()}))


def source_digest():
    import glob
    h = hashlib.sha256()
    for p in sorted(glob.glob(os.path.join(ROOT, "paper_2505_00315_gb300", "csrc", "*"))):
        with open(p, "rb") as f:
            h.update(f.read())
    return h.hexdigest()


# ------------------------------------------------------------ multi-rank

def combine_ranks(local_ms: float, tokens_per_rank: int, dist=None, device="cpu"):
    """Whole-job throughput under weak scaling: every rank processes its own
    batch, the job's time is the slowest rank's.  Returns (tokens/s, max ms)."""
    world = 1
    ms = float(local_ms)
    if dist is not None and dist.is_initialized():
        import torch
        world = dist.get_world_size()
        t = torch.tensor([ms], dtype=torch.float64, device=device)
        dist.all_reduce(t, op=dist.ReduceOp.MAX)
        ms = float(t.item())
    return world * tokens_per_rank / (ms / 1e3), ms


# ------------------------------------------------------------------ main

def run_reference(args, cfg, rank, world):
    """The oracle as the reference arm: rank 0 times it on the host cores."""
    if rank != 0:
        return
    import oracle
    x = make_workload(cfg, args)
    per_step_budget = max(1.0, 150.0 / max(1, args.steps + args.warmup))
    n, _ = choose_sample(cfg, x, per_step_budget)
    for _ in range(args.warmup):
        oracle_sample(cfg, x, n)
    times = [oracle_sample(cfg, x, n) for _ in range(args.steps)]
    total = sum(times)
    value = n * cfg.T * args.steps / total
    what = "forward+backward" if cfg.backward else "forward"
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * total / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": config_block(cfg, args),
            "cpu_baseline": {"value": value, "unit": "tokens/s", "kind": "oracle",
                             "cores": oracle.num_threads(),
                             "sample": f"{what} of {n} of the {cfg.B} sequences per step"},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def variant(cfg, args):
    """The workload with the option flags applied, and its name."""
    cfg = cfg.with_(rope=bool(args.rope), first_token=bool(args.first_token))
    name = cfg.name + ("+rope" if cfg.rope else "") + ("+first" if cfg.first_token else "")
    if args.dense_heads:
        name += f"+dense{args.dense_heads}" + (f"w{args.window}" if args.window else "")
    return cfg.with_(name=name)


def config_block(cfg, args=None):
    extra = {}
    if cfg.rope or cfg.first_token:
        extra.update(rope=cfg.rope, first_token=cfg.first_token)
    if args is not None and args.dense_heads:
        extra.update(H_dense=args.dense_heads, window=args.window)
    return {"workload": cfg.name, "B": cfg.B, "T": cfg.T, "d": cfg.d, "H": cfg.H, "hp": cfg.hp,
            "k": cfg.k, "storage": cfg.dtype, **extra,
            "inputs": "seeded Gaussian X, weights N(0,1/d), dY; planted router margin",
            "l2": "flushed before every timed step by a 256 MiB write outside the step's events"}


def make_workload(cfg, args):
    """Seeded inputs of the workload, plus the dense heads' weights and window
    of a hybrid layer."""
    from paper_2505_00315_gb300 import workloads as W
    x = W.make_inputs(cfg)
    if args.dense_heads:
        x.update(W.make_dense_weights(cfg, args.dense_heads))
        x["window"] = args.window
    return x


def main():
    args = parse_args()
    import torch
    from paper_2505_00315_gb300 import workloads as W

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    cfg = variant(W.CONFIGS[args.config or W.BENCH_CONFIG], args)

    if args.ingest_ncu:
        ingest_ncu(args.ingest_ncu, cfg.name)
        return

    if args.impl == "reference":
        run_reference(args, cfg, rank, world)
        return

    import paper_2505_00315_gb300 as mosa
    from paper_2505_00315_gb300 import flops

    torch.cuda.set_device(local)
    dist = None
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", device_id=torch.device("cuda", local))

    def barrier():
        if dist is not None:
            dist.barrier()

    x = make_workload(cfg, args)
    tdt = torch.bfloat16 if cfg.dtype == "bf16" else torch.float32
    dev = torch.device("cuda", local)
    D = {n: torch.from_numpy(x[n]).to(dev).to(tdt) for n in x if n != "window"}
    shape = mosa.make_shape(D["X"], D["Wq"], cfg.k, cfg.first_token, cfg.rope)
    hybrid = args.dense_heads > 0
    if hybrid:
        ws = mosa.alloc_hybrid_workspace(
            mosa.make_hybrid_shape(D["X"], D["Wq"], cfg.k, args.dense_heads, args.window,
                                   cfg.first_token, cfg.rope), dev)
    else:
        ws = mosa.alloc_workspace(shape, dev)
    f32 = dict(dtype=torch.float32, device=dev)
    outs = {"Y": torch.empty((cfg.B, cfg.T, cfg.d), **f32),
            "I": torch.empty((cfg.B, cfg.H, cfg.k), dtype=torch.int32, device=dev),
            "r_sel": torch.empty((cfg.B, cfg.H, cfg.k), **f32)}
    grads = {"dX": torch.empty((cfg.B, cfg.T, cfg.d), **f32),
             "dW_r": torch.empty((cfg.d, cfg.H), **f32),
             "dW_q": torch.empty((cfg.H, cfg.d, cfg.hp), **f32),
             "dW_k": torch.empty((cfg.H, cfg.d, cfg.hp), **f32),
             "dW_v": torch.empty((cfg.H, cfg.d, cfg.hp), **f32),
             "dW_o": torch.empty((cfg.H, cfg.hp, cfg.d), **f32)}
    if hybrid:
        for n in ("Dq", "Dk", "Dv", "Do"):
            grads["dD_" + n[1]] = torch.empty(D[n].shape, **f32)
    flush_buf = torch.empty(L2_FLUSH_BYTES // 4, **f32)
    Wm = (D["Wr"], D["Wq"], D["Wk"], D["Wv"], D["Wo"])

    def layer(Xd, dYd, o, g):
        """One forward (+ backward) through the public API."""
        if hybrid:
            Dw = (D["Dq"], D["Dk"], D["Dv"], D["Do"])
            _, I, rs, _ = mosa.mosa_hybrid_forward(Xd, *Wm, *Dw, cfg.k, window=args.window,
                                                   workspace=ws, out=o,
                                                   first_token=cfg.first_token, rope=cfg.rope)
            if cfg.backward:
                mosa.mosa_hybrid_backward(Xd, *Wm, *Dw, I, rs, dYd, ws, window=args.window,
                                          out=g, rope=cfg.rope)
            return
        _, I, rs, _, _ = mosa.mosa_forward(Xd, *Wm, cfg.k, workspace=ws, out=o,
                                           first_token=cfg.first_token, rope=cfg.rope)
        if cfg.backward:
            mosa.mosa_backward(Xd, *Wm, I, rs, dYd, ws, out=g, rope=cfg.rope)

    def step():
        layer(D["X"], D["dY"], outs, grads)

    if args.profile_run:
        # a short, fixed launch sequence for ncu: warm-up steps, then the steps to capture
        for _ in range(args.warmup + args.steps):
            step()
        torch.cuda.synchronize()
        st = mosa.mosa_check_status(shape, ws) if not hybrid else 0
        print(json.dumps({"profile_run": cfg.name, "steps": args.steps, "warmup": args.warmup,
                          "launches": int(mosa.mosa_kernel_launches()), "status": int(st)}))
        if st != 0:
            raise SystemExit(f"device status {st}")
        return

    # Warm-up, then one profiled pass to find the dominant stage.
    for _ in range(max(3, args.warmup)):
        flush_buf.zero_()
        step()
    torch.cuda.synchronize()
    # Stage times are per step: a hybrid layer runs each stage twice a step
    # (MoSA heads, then dense heads), and its algorithmic work is per step.
    mosa.mosa_profile_stages((1 << len(STAGES)) - 1)
    n_prof = 5
    for _ in range(n_prof):
        flush_buf.zero_()
        step()
    torch.cuda.synchronize()
    prof = mosa.mosa_profile_read()
    mosa.mosa_profile_stages(0)
    stage_ms = {s: prof[s][0] / n_prof for s in STAGES if prof[s][1]}
    dominant = max(stage_ms, key=stage_ms.get)

    # Timed region: K steps, L2 flushed before each, the dominant stage timed
    # live with CUDA events on every PROFILE_EVERY-th step.  Its event pair sits
    # inside the step's graph (and cuts the early-launch chain around it), so
    # timing it on every step would slow the steps it measures; both graph
    # variants are captured before timing starts.  Nothing is read back during
    # the timed region (a read waits for the device, and the next step would
    # then start from an idle GPU with the host's launch latency inside its
    # events): the events are read after it, and each timed step's kernel
    # spans are copied on the device, outside the step's events, into a
    # per-step buffer read after it as well.
    K = args.steps
    starts = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    ends = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
    dom_mask = 1 << STAGES.index(dominant)
    for mask in (dom_mask, 0):
        mosa.mosa_profile_stages(mask)
        flush_buf.zero_()
        step()
    torch.cuda.synchronize()
    mosa.mosa_profile_read()
    sampler = ClockSampler(local) if rank == 0 else None
    if sampler:
        sampler.start()
    barrier()
    torch.cuda.synchronize()
    launches0 = mosa.mosa_kernel_launches()
    span_slots = torch.zeros((K, 32), dtype=torch.int64, device=dev)
    n_timed = 0
    t_host0 = time.time()
    for i in range(K):
        timed = i % PROFILE_EVERY == 0
        mosa.mosa_profile_stages(dom_mask if timed else 0)
        flush_buf.zero_()
        starts[i].record()
        step()
        ends[i].record()
        if timed:
            n_timed += 1
            if not hybrid:
                mosa.mosa_profile_spans_copy(shape, ws, span_slots[i])
    torch.cuda.synchronize()
    t_host1 = time.time()
    ms_d, n_d = mosa.mosa_profile_read()[dominant]
    dom = [ms_d, n_d, n_timed]   # ms over the timed steps, launches, steps
    span = [0.0, 0]              # kernel-span ms, steps
    di = STAGES.index(dominant)
    m64 = (1 << 64) - 1
    for i in range(0, K, PROFILE_EVERY):
        # unsigned, as the library decodes them: start all ones or end 0 = no record
        a, b = (int(v) & m64 for v in span_slots[i, 2 * di:2 * di + 2].tolist())
        if not hybrid and a != m64 and b != 0 and b >= a:
            span[0] += (b - a) * 1e-6
            span[1] += 1
    barrier()
    launches = mosa.mosa_kernel_launches() - launches0
    mosa.mosa_profile_stages(0)
    clocks = None
    if sampler:
        sampler.mark(t_host0, t_host1)
        clocks = sampler.stop()
    total_ms = sum(s.elapsed_time(e) for s, e in zip(starts, ends))
    value, total_ms = combine_ranks(total_ms, cfg.B * cfg.T * K, dist, dev)

    # Diagnostic: the stage timeline of one step (kernel spans stamped by the
    # kernels, no events between them; outside the timed region), the median
    # step of a few, each after an L2 flush.
    timeline = None
    if not hybrid:
        mosa.mosa_profile_timeline(True)
        try:
            tls = []
            for _ in range(5):
                flush_buf.zero_()
                step()
                tls.append(mosa.mosa_profile_timeline_read(shape, ws))
        finally:
            mosa.mosa_profile_timeline(False)
        tls.sort(key=lambda t: max(v[1] for v in t.values()))
        mid = tls[len(tls) // 2]
        timeline = {"what": "first CTA start and last CTA end of each stage's kernels in one "
                            "step (the median of 5, after an L2 flush), microseconds from the "
                            "step's first kernel start; no events between the kernels",
                    "us": {k: [round(a, 1), round(b, 1)] for k, (a, b) in
                           sorted(mid.items(), key=lambda kv: kv[1][0])}}

    # Diagnostic: the same step replayed from a CUDA graph captured by torch
    # around the eager calls (the library's own graph cache switched off).
    graph_ms = None
    os.environ["MOSA_GRAPHS"] = "0"
    try:
        g = torch.cuda.CUDAGraph()
        side = torch.cuda.Stream()
        side.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(side):
            step()
        torch.cuda.current_stream().wait_stream(side)
        torch.cuda.synchronize()
        with torch.cuda.graph(g):
            step()
        for _ in range(3):
            flush_buf.zero_()
            g.replay()
        torch.cuda.synchronize()
        gs = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
        ge = [torch.cuda.Event(enable_timing=True) for _ in range(K)]
        for i in range(K):
            flush_buf.zero_()
            gs[i].record()
            g.replay()
            ge[i].record()
        torch.cuda.synchronize()
        graph_ms = sum(a.elapsed_time(b) for a, b in zip(gs, ge)) / K
        del g
    except Exception as exc:  # capture unsupported: report why
        graph_ms = f"unavailable: {exc}"
    finally:
        os.environ.pop("MOSA_GRAPHS", None)

    # End to end through the public API with pinned host buffers, pipelined as a
    # training loop runs it: step i's inputs are copied in on one stream while
    # step i-1 computes, and its outputs copied out on another while step i+1
    # computes (two device buffer sets).  The timed region holds every step's
    # copies and compute; it ends when the last step's outputs are on the host.
    hX = torch.from_numpy(x["X"]).to(tdt).pin_memory()
    hdY = torch.from_numpy(x["dY"]).to(tdt).pin_memory()
    hY = torch.empty((cfg.B, cfg.T, cfg.d), dtype=torch.float32).pin_memory()
    hdX = torch.empty((cfg.B, cfg.T, cfg.d), dtype=torch.float32).pin_memory()
    slots = [{"X": torch.empty_like(D["X"]), "dY": torch.empty_like(D["dY"]),
              "outs": {n: torch.empty_like(v) for n, v in outs.items()},
              "grads": {n: torch.empty_like(v) for n, v in grads.items()}} for _ in range(2)]
    comp = torch.cuda.current_stream()
    s_in, s_out = torch.cuda.Stream(), torch.cuda.Stream()
    in_ready = [torch.cuda.Event() for _ in range(2)]
    in_free = [torch.cuda.Event() for _ in range(2)]
    done = [torch.cuda.Event() for _ in range(2)]
    out_free = [torch.cuda.Event() for _ in range(2)]
    e2e_steps = max(10, K // 4)

    def e2e_run(n, start_event=None):
        if start_event is not None:
            s_in.wait_event(start_event)
            s_out.wait_event(start_event)
        for i in range(n):
            j = i % 2
            sl = slots[j]
            with torch.cuda.stream(s_in):
                if i >= 2:
                    s_in.wait_event(in_free[j])   # step i-2 is done with these inputs
                sl["X"].copy_(hX, non_blocking=True)
                if cfg.backward:
                    sl["dY"].copy_(hdY, non_blocking=True)
                in_ready[j].record(s_in)
            comp.wait_event(in_ready[j])
            if i >= 2:
                comp.wait_event(out_free[j])      # step i-2's outputs have left
            layer(sl["X"], sl["dY"], sl["outs"], sl["grads"])
            in_free[j].record(comp)
            done[j].record(comp)
            with torch.cuda.stream(s_out):
                s_out.wait_event(done[j])
                hY.copy_(sl["outs"]["Y"], non_blocking=True)
                if cfg.backward:
                    hdX.copy_(sl["grads"]["dX"], non_blocking=True)
                out_free[j].record(s_out)
        comp.wait_stream(s_in)
        comp.wait_stream(s_out)

    e2e_run(4)   # captures the layer's graphs for both buffer sets
    torch.cuda.synchronize()
    barrier()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record()
    e2e_run(e2e_steps, start_event=e0)
    e1.record()
    torch.cuda.synchronize()
    e2e_value, e2e_ms = combine_ranks(e0.elapsed_time(e1), cfg.B * cfg.T * e2e_steps, dist, dev)
    h2d = hX.numel() * hX.element_size() + (hdY.numel() * hdY.element_size() if cfg.backward else 0)
    d2h = hY.numel() * 4 + (hdX.numel() * 4 if cfg.backward else 0)

    if rank != 0:
        if dist is not None:
            dist.destroy_process_group()
        return

    # Roofline of the dominant kernel.
    peaks, peak_src = load_peaks()
    work = flops.hybrid_work(cfg.B, cfg.T, cfg.d, cfg.H, cfg.hp, cfg.k, args.dense_heads,
                             args.window, elem_bytes=2 if cfg.dtype == "bf16" else 4)
    impl = mosa.stage_impl(shape)
    kind = stage_kind(dominant, impl)
    bound, peak, unit = stage_bound(dominant, peaks, kind)
    dom_ms = dom[0] / max(dom[2], 1)   # per step
    if unit == "GB/s":
        achieved = work[dominant]["bytes"] / (dom_ms / 1e3) / 1e9
    else:
        achieved = work[dominant]["flops"] / (dom_ms / 1e3) / 1e12
    key = "flops" if unit != "GB/s" else "bytes"
    scale = 1e12 if unit != "GB/s" else 1e9
    span_ms = span[0] / span[1] if span[1] else None
    span_achieved = work[dominant][key] / (span_ms / 1e3) / scale if span_ms else None
    layer_flops = work["forward_flops"] + (work["backward_flops"] if cfg.backward else 0)
    full = flops.hybrid_work(cfg.B, cfg.T, cfg.d, cfg.H, cfg.hp, cfg.k, args.dense_heads,
                             args.window, causal=False)
    layer_flops_full = full["forward_flops"] + (full["backward_flops"] if cfg.backward else 0)
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": args.warmup, "ms_per_step": total_ms / K, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": cfg.dtype, "data": "synthetic",
        "config": config_block(cfg, args),
        "roofline": {"kernel": dominant, "bound": bound, "achieved": achieved, "peak": peak,
                     "unit": unit, "frac": achieved / peak, "peak_source": peak_src,
                     "traffic": traffic_for(dominant, cfg.name),
                     "algorithmic": work[dominant]["flops" if unit != "GB/s" else "bytes"],
                     "stage_ms_per_step": dom_ms, "launches_per_step": dom[1] / max(dom[2], 1),
                     "timed_steps": dom[2],
                     "kernel_span_ms_per_step": span_ms,
                     "kernel_span_achieved": span_achieved,
                     "kernel_span_frac": span_achieved / peak if span_achieved else None,
                     "kernel_span_what": "first CTA start to last CTA end of the stage's "
                                         "kernels (%globaltimer), same timed steps",
                     "timed_every_nth_step": PROFILE_EVERY},
        "layer_tflops": layer_flops * world * K / (total_ms / 1e3) / 1e12,
        "layer_tflops_counting": "causal attention counted as 2h'k(k+1) forward, "
                                 "5h'k(k+1) backward",
        "layer_tflops_paper_count": layer_flops_full * world * K / (total_ms / 1e3) / 1e12,
        "layer_tflops_paper_counting": "attention counted as the paper's App. A does, "
                                       "4h'k^2 forward (no causal halving), 10h'k^2 backward",
        "stage_ms": {s: round(v, 5) for s, v in stage_ms.items()},
        "e2e": {"value": e2e_value, "unit": "tokens/s",
                "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                "what": "pinned host X, dY -> device; forward+backward; Y, dX -> pinned host; "
                        "copies on two streams beside the compute of the neighbouring steps "
                        "(two device buffer sets)"},
        "gpu_launches": int(launches),
        "graph_ms_per_step": graph_ms,
        "timeline": timeline,
        "clocks": clocks,
    }
    if world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(cfg, x, args.cpu_budget_s)
    print(json.dumps(line), flush=True)
    if dist is not None:
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
