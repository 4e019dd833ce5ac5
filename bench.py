"""Benchmark of the role-conditional KV-eviction hot path on GB300.

One step = the whole path over one batch of synthetic input: SnapKV windowed
score (both softmax passes in one persistent kernel), the role-conditional
selector with the max-pool fused into its load, and the K/V gather-compaction,
for every (layer, sequence, KV head) of the workload.  The default workload is the
long-context one the headline metric is quoted on: 32 layers, 4 sequences of
32768 tokens, 32 query / 8 KV heads, head dim 128, W = 64, pool 7, B = 0.10
(about 17 GB of bf16 K/V resident on the GPU, larger than L2, so no L2 flush
is needed between steps).

Prints one JSON line (rank 0).  `--impl reference` times the fp64 CPU oracle
on a bounded sample of the same workload instead.
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
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = "KV tokens scored+compressed/sec at N=32k; % of GB300 HBM roofline"
UNIT = "tokens/s"


# ----------------------------------------------------------------- helpers --

def dist_env():
    return int(os.environ.get("RANK", "0")), int(os.environ.get("WORLD_SIZE", "1")), \
        int(os.environ.get("LOCAL_RANK", "0"))


def max_over_ranks(x: float, world: int) -> float:
    """Largest value of x over all ranks (x on every rank)."""
    if world <= 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def job_throughput(world: int, units_per_rank: float, steps: int, elapsed_ms: float) -> float:
    """Whole-job rate: every rank processes units_per_rank per step (weak
    scaling), elapsed_ms is the slowest rank's time for `steps` steps."""
    return world * units_per_rank * steps / (elapsed_ms / 1e3)


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


HBM_NOMINAL_GBS = 7900.0   # GB300 HBM3e nominal bandwidth (context beside the measured peak)


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return {"hbm_gbs": d["hbm_gbs"], "bf16_tflops": d["bf16_tflops"],
                "bf16_tflops_sustained": d.get("bf16_tflops_sustained", d["bf16_tflops"]),
                "source": "measured"}
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "source": "fallback"}


class ClockSampler:
    """nvidia-smi clocks and throttle reasons sampled every 200 ms."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None
        time.sleep(0.25)

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        sm, smax, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        with open(self.path) as f:
            for line in f:
                parts = [x.strip() for x in line.split(",")]
                if len(parts) < 9:
                    continue
                try:
                    sm.append(float(parts[1]))
                    smax.append(float(parts[2]))
                except ValueError:
                    continue
                for nm, v in zip(names, parts[5:9]):
                    if v.lower() == "active":
                        reasons.add(nm)
        os.unlink(self.path)
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


# ------------------------------------------------------- algorithmic counts --

# DRAM bytes (read + write) of one launch of a kernel come from ncu's
# dram__bytes_read.sum + dram__bytes_write.sum, captured on a smaller case of
# the same workload and scaled by units (the kernels stream each unit's keys,
# so their traffic grows in proportion).  profiles/dram_traffic.md holds the
# captures, each with a hash of the kernel's source files at capture time; a
# capture whose sources have changed since is stale and gives null.
TRAFFIC_FILE = os.path.join(ROOT, "profiles", "dram_traffic.md")
KERNEL_SOURCES = {
    ("snapkv", "score"): ["attn_score.cu", "device_common.cuh", "internal.h"],
    ("h2o", "score"): ["attn_score.cu", "device_common.cuh", "internal.h"],
    ("quest", "score"): ["quest.cu", "device_common.cuh", "internal.h"],
    ("snapkv", "select"): ["select.cu", "device_common.cuh", "internal.h"],
    ("snapkv", "compact"): ["compact.cu", "device_common.cuh", "internal.h"],
}


def source_hash(files) -> str:
    import hashlib
    h = hashlib.sha256()
    for f in files:
        with open(os.path.join(ROOT, "paper_2607_13205_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def measured_traffic(workload: str, score_kind: str, kernel: str, single: bool = False):
    """(bytes per full launch, note) from profiles/dram_traffic.md, or (None,
    reason).  Rows: | workload | score | kernel | pass | units captured |
    units full | dram read MB | dram write MB | source hash |."""
    srcs = KERNEL_SOURCES.get((score_kind, kernel)) or KERNEL_SOURCES.get(("snapkv", kernel))
    if srcs is None or not os.path.exists(TRAFFIC_FILE):
        return None, "no capture"
    want = source_hash(srcs)
    mode = "one" if single else "two"
    with open(TRAFFIC_FILE) as f:
        for line in f:
            cells = [c.strip() for c in line.strip().strip("|").split("|")]
            if len(cells) != 9 or cells[0] != workload or cells[1] != score_kind or cells[2] != kernel:
                continue
            if kernel == "score" and score_kind != "quest" and cells[3] != mode:
                continue
            try:
                u_cap, u_full = float(cells[4]), float(cells[5])
                rd, wr = float(cells[6]), float(cells[7])
            except ValueError:
                continue
            if cells[8] != want:
                return None, f"stale: captured on sources {cells[8]}, now {want}"
            return (rd + wr) * 1e6 * u_full / u_cap, (f"ncu on {cells[4]} of {cells[5]} units, "
                                                      f"scaled by units; sources {want}")
    return None, "no capture for this workload"


def path_counts(w, B, score_kind="snapkv"):
    """Algorithmic bytes / flops per step of each kernel of the path (the
    method's own work: K read once, one Q K^T, the queries, the pre-pool score
    written and read once, the kept K/V rows read and written, the kept index
    written and read).  'hw_flops' is the contraction the exact two-pass
    kernel actually runs (Q K^T twice).  Variable-length batches use their
    mean length (exact for the sums of per-token terms)."""
    U = w.L * w.b * w.Hkv
    n = (sum(w.seqlens) / w.b) if w.varlen else w.n
    d = w.d
    K = (sum(math.ceil(B * x) for x in w.seqlens) / w.b) if w.varlen else math.ceil(B * n)
    if w.kind == "h2o":
        causal = n * (n + 1) / 2                     # query-key pairs per head
        flops = 2.0 * U * w.G * causal * d
        qbytes = U * w.G * n * d * 2
        kbytes = U * n * d * 2
        return {
            # K and the queries read once, the scores written once
            "score": {"bytes": kbytes + qbytes + U * n * 4, "flops": flops, "hw_flops": 2.0 * flops},
            "select": {"bytes": U * n * 4 + w.b * n + U * K * 4, "flops": 0.0},
            "compact": {"bytes": U * K * 4 + 2 * 2 * U * K * d * 2, "flops": 0.0},
            "path_bytes": kbytes + qbytes + U * n * 8 + U * K * 8 + 2 * 2 * U * K * d * 2 + w.b * n,
            "kept": K,
        }
    rows = w.G * w.W
    kbytes = U * n * d * 2
    qbytes = U * rows * d * 2
    flops = 2.0 * U * rows * n * d
    if score_kind == "quest":
        # one pass over K for the page bounds, no contraction
        flops = 0.0
    return {
        "score": {"bytes": kbytes + qbytes + U * n * 4, "flops": flops, "hw_flops": 2.0 * flops},
        "select": {"bytes": U * n * 4 + w.b * n + U * K * 4, "flops": 0.0},
        "compact": {"bytes": U * K * 4 + 2 * 2 * U * K * d * 2, "flops": 0.0},
        "path_bytes": kbytes + qbytes + U * n * 8 + U * K * 8 + 2 * 2 * U * K * d * 2 + w.b * n,
        "kept": K,
    }


def roofline(counts, per_kernel, peaks, names, workload, score_kind, layers_override, traffic_arg):
    """The dominant kernel's roofline: bound by its algorithmic bytes or
    flops, whichever takes longer at the measured peaks; achieved = that work
    / the kernel's mean launch time."""
    dom = max(names, key=lambda k: per_kernel[k])
    dk = counts[dom]
    t_dom = per_kernel[dom] / 1e3
    t_hbm = dk["bytes"] / (peaks["hbm_gbs"] * 1e9)
    t_tc = dk["flops"] / (peaks["bf16_tflops"] * 1e12) if dk["flops"] else 0.0
    if t_tc > t_hbm:
        roof = {"bound": "tensor", "achieved": dk["flops"] / t_dom / 1e12,
                "peak": peaks["bf16_tflops"], "unit": "TFLOP/s"}
    else:
        roof = {"bound": "hbm", "achieved": dk["bytes"] / t_dom / 1e9, "peak": peaks["hbm_gbs"],
                "unit": "GB/s"}
    roof["frac"] = roof["achieved"] / roof["peak"]
    roof["kernel"] = dom
    roof["algorithmic"] = {"bytes": dk["bytes"], "flops": dk["flops"]}
    if dk.get("hw_flops"):
        # the exact two-pass score runs Q K^T twice: tensor-pipe use of that work
        roof["hw_tensor_frac"] = dk["hw_flops"] / t_dom / 1e12 / peaks["bf16_tflops"]
    if traffic_arg is not None:
        roof["traffic"], roof["traffic_note"] = traffic_arg, "given on the command line"
    elif layers_override:
        roof["traffic"], roof["traffic_note"] = None, "layer count overridden"
    else:
        roof["traffic"], roof["traffic_note"] = measured_traffic(workload, score_kind, dom)
    roof["peak_source"] = peaks["source"] + " (burst)"
    return roof


# ----------------------------------------------------------------- GPU arm --

def run_gpu(args):
    import torch

    from paper_2607_13205_gb300 import inputs as I
    from paper_2607_13205_gb300 import rolekv as R

    rank, world, local = dist_env()
    torch.cuda.set_device(local)
    if world > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl")
    dev = torch.device("cuda", local)
    w = I.WORKLOADS[args.workload]
    if args.layers:
        w = w.scaled(L=args.layers)
    B = args.budget if args.budget else w.budgets[0]
    h2o = w.kind == "h2o"

    roles_np = I.workload_roles(w, seed=rank)
    K, V = I.make_kv(w, roles_np, seed=rank, device=dev)
    qw = I.make_q_full(w, seed=rank, device=dev) if h2o else I.make_q_window(w, seed=rank, device=dev)
    roles = torch.as_tensor(roles_np, device=dev)
    batch = R.Batch(w.L, w.b, w.Hq, w.Hkv, w.d, w.n, seqlens=list(w.seqlens) if w.varlen else None,
                    device=dev, kept_extra=kept_extra(args.policy))
    policy = POLICY_CODES[args.policy]
    params = R.select_params(B, I.PAPER_ALPHA, alpha_key=0.0, key_role=I.ROLE_KEY, policy=policy,
                             keep_last=args.keep_last)
    scores = torch.empty(batch.score_shape(), dtype=torch.float32, device=dev)
    keep = torch.empty(batch.kept_shape(B), dtype=torch.int32, device=dev)
    k_out = torch.empty(R.compact_shape(batch, B), dtype=torch.bfloat16, device=dev)
    v_out = torch.empty_like(k_out)
    ws = R.workspace(R.OP_H2O if h2o else R.OP_SNAPKV, batch, w.W, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream(dev)

    names = ["score", "select", "compact"]
    # the Quest page bound is selected as it is (no max-pool over the KV axis)
    pool_k = 1 if args.score == "quest" else w.pool_k
    ns = len(names) - 2                              # score kernels

    def score():
        if h2o:
            R.h2o_score(batch, qw, K, scores, ws=ws, status=status, stream=stream)
        elif args.score == "quest":
            R.quest_score(batch, qw, K, w.W, args.page, scores, stream=stream)
        else:
            # pool_k = 1: the pre-pool scores go straight out; the selector pools
            R.snapkv_score(batch, qw, K, w.W, 1, scores, ws=ws, status=status, stream=stream)

    def step(ev=None):
        # the path as three public calls: scores, selection (pool fused),
        # compaction
        if ev is not None:
            R.set_stage_events(ev[1:1 + ns])
        score()
        if ev is not None:
            R.set_stage_events(ev[1 + ns:2 + ns])
        R.role_alloc_select(batch, scores, roles, params, keep, pool_k=pool_k, status=status,
                            stream=stream)
        if ev is not None:
            R.set_stage_events(ev[2 + ns:3 + ns])
        R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=status, stream=stream)
        if ev is not None:
            R.set_stage_events([])

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize(dev)

    # per-step events: [0] step start, then one after each kernel
    events = [[torch.cuda.Event(enable_timing=True) for _ in range(len(names) + 1)]
              for _ in range(args.steps)]
    for evs in events:
        for e in evs:
            e.record(stream)       # create the underlying CUDA events
    torch.cuda.synchronize(dev)

    clocks = ClockSampler(local)
    clocks.start()
    barrier(world)
    torch.cuda.synchronize(dev)
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    t0.record(stream)
    for i in range(args.steps):
        events[i][0].record(stream)
        step(events[i])
    t1.record(stream)
    torch.cuda.synchronize(dev)
    barrier(world)
    clock_info = clocks.stop()
    elapsed_ms = t0.elapsed_time(t1)
    elapsed_ms = max_over_ranks(elapsed_ms, world)
    st = int(status.item())
    if st != 0:
        raise SystemExit(f"device status {st} during the timed steps")

    per_kernel = {nm: 0.0 for nm in names}
    for evs in events:
        for j, nm in enumerate(names):
            per_kernel[nm] += evs[j].elapsed_time(evs[j + 1])
    per_kernel = {nm: v / args.steps for nm, v in per_kernel.items()}

    seq_tokens = w.b * w.n if not w.varlen else sum(w.seqlens)
    ms_step = elapsed_ms / args.steps
    value = job_throughput(world, seq_tokens, args.steps, elapsed_ms)

    peaks = load_peaks()
    counts = path_counts(w, B, args.score)
    roof = roofline(counts, per_kernel, peaks, names, w.name, "h2o" if h2o else args.score,
                    args.layers, args.traffic)
    path_frac = counts["path_bytes"] / (ms_step / 1e3) / 1e9 / peaks["hbm_gbs"]
    tensor_util = {nm: counts[nm]["flops"] / (per_kernel[nm] / 1e3) / 1e12 / peaks["bf16_tflops"]
                   for nm in names if counts[nm]["flops"] > 0}

    result = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": f"{w.name}: L={w.L} b={w.b} Hq={w.Hq} Hkv={w.Hkv} d={w.d} "
                               f"N={'varlen<=' if w.varlen else ''}{w.n} W={w.W} pool={w.pool_k} B={B}"
                               + (f" score=quest page={args.page}" if args.score == "quest" else "")
                               + (f" policy={args.policy}" if args.policy != "quota" else "")
                               + (f" keep_last={args.keep_last}" if args.keep_last else ""),
                   "global_batch": world * w.b, "seq_len": w.n, "parallelism": f"replicas x{world}",
                   "l2": "inputs larger than L2, no flush"},
        "hbm_path_frac": path_frac,
        "hbm_path_frac_nominal": counts["path_bytes"] / (ms_step / 1e3) / 1e9 / HBM_NOMINAL_GBS,
        "tensor_frac_of_measured_peak": tensor_util or None,
        "per_kernel_ms": per_kernel,
        "unit_tokens_per_s": world * w.L * w.Hkv * seq_tokens * args.steps / (elapsed_ms / 1e3),
        "roofline": roof,
        "clocks": clock_info,
        "gpu_launches": len(names) * args.steps,
    }

    if not h2o and args.score == "snapkv" and not args.no_single_pass:
        result["single_pass"] = run_single_pass(args, batch, params, w, B, qw, K, V, roles, scores,
                                                keep, k_out, v_out, ws, status, stream, world,
                                                seq_tokens)
    if h2o and not args.no_single_pass:
        result["single_pass"] = run_h2o_single_pass(args, batch, params, w, B, qw, K, V, roles, scores,
                                                    keep, k_out, v_out, ws, status, stream, world,
                                                    seq_tokens, peaks, counts)
    if not h2o and not args.no_decode:
        result["decode"] = run_decode(args, batch, w, B, K, V, keep, k_out, v_out, stream, world, peaks)
    if not args.no_e2e:
        result["e2e"] = run_e2e(args, score, batch, params, w, B, qw, K, V, roles, scores, keep,
                                k_out, v_out, status, stream, world, seq_tokens)
    if rank == 0 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(w, B, args.cpu_seconds, host_inputs=(qw, K, V, roles_np),
                                              policy=args.policy, keep_last=args.keep_last,
                                              score_kind=args.score, page=args.page)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


def window_lse(w, qw, K):
    """Natural-log softmax normalisers of the window rows, [L][b][Hq][W] fp32,
    as an attention prefill would hand them over (computed here once, with
    fp32 torch matmuls, outside any timed region)."""
    import torch

    L, b, G, W, d = w.L, w.b, w.G, w.W, w.d
    lse = torch.zeros((L, b, w.Hq, W), dtype=torch.float32, device=qw.device)
    lens = list(w.seqlens) if w.varlen else [w.n] * b
    starts = [0]
    for x in lens[:-1]:
        starts.append(starts[-1] + x)
    scale = 1.0 / math.sqrt(d)
    for l in range(L):
        for s in range(b):
            n = lens[s]
            if n == 0:
                continue
            we = min(W, n)
            for h in range(w.Hkv):
                if w.varlen:
                    k = K[l, starts[s]:starts[s] + n, h].float()
                else:
                    k = K[l, s, h, :n].float()
                q = qw[l, s, h * G:(h + 1) * G, :we].float().reshape(G * we, d)
                logits = (q @ k.T) * scale
                pos = (n - we + torch.arange(we, device=q.device)).repeat(G)
                mask = torch.arange(n, device=q.device)[None, :] > pos[:, None]
                logits.masked_fill_(mask, float("-inf"))
                lse[l, s, h * G:(h + 1) * G, :we] = torch.logsumexp(logits, dim=1).reshape(G, we)
    return lse


def run_single_pass(args, batch, params, w, B, qw, K, V, roles, scores, keep, k_out, v_out, ws,
                    status, stream, world, seq_tokens):
    """The step with the window normalisers supplied by the caller: the score
    is one pass over K (no row statistics), then selection and compaction."""
    import torch

    from paper_2607_13205_gb300 import rolekv as R

    torch.backends.cuda.matmul.allow_tf32 = False
    lse = window_lse(w, qw, K)
    torch.cuda.synchronize()

    def step():
        R.snapkv_score(batch, qw, K, w.W, 1, scores, lse_win=lse, ws=ws, status=status, stream=stream)
        R.role_alloc_select(batch, scores, roles, params, keep, pool_k=w.pool_k, status=status,
                            stream=stream)
        R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=status, stream=stream)

    for _ in range(3):
        step()
    steps = max(1, args.steps)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * steps + 1)]
    torch.cuda.synchronize()
    barrier(world)
    ev[0].record(stream)
    for i in range(steps):
        R.snapkv_score(batch, qw, K, w.W, 1, scores, lse_win=lse, ws=ws, status=status, stream=stream)
        ev[2 * i + 1].record(stream)
        R.role_alloc_select(batch, scores, roles, params, keep, pool_k=w.pool_k, status=status,
                            stream=stream)
        R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=status, stream=stream)
        ev[2 * i + 2].record(stream)
    torch.cuda.synchronize()
    barrier(world)
    total = max_over_ranks(ev[0].elapsed_time(ev[-1]), world)
    score_ms = sum(ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(steps)) / steps
    if int(status.item()) != 0:
        raise SystemExit(f"device status {int(status.item())} in the single-pass steps")
    return {"value": world * seq_tokens * steps / (total / 1e3), "unit": UNIT,
            "ms_per_step": total / steps, "score_ms": score_ms, "steps": steps,
            "lse": "window normalisers supplied by the caller (computed once, untimed)"}


def prefill_lse(w, Q, K):
    """Natural-log softmax normaliser of every causal prefill query row, in
    h2o_score's layout (dense [L][b][Hq][n]), as the prefill attention would
    hand it over (computed here once, with fp32 torch matmuls, outside any
    timed region)."""
    import torch

    L, b, G, n, d = w.L, w.b, w.G, w.n, w.d
    lse = torch.empty((L, b, w.Hq, n), dtype=torch.float32, device=Q.device)
    scale = 1.0 / math.sqrt(d)
    above = torch.ones((n, n), dtype=torch.bool, device=Q.device).triu_(1)   # keys after the query
    for l in range(L):
        for s in range(b):
            for h in range(w.Hkv):
                k = K[l, s, h].float()
                q = Q[l, s, h * G:(h + 1) * G].float()                 # [G][n][d]
                logits = torch.matmul(q, k.T) * scale
                logits.masked_fill_(above, float("-inf"))
                lse[l, s, h * G:(h + 1) * G] = torch.logsumexp(logits, dim=-1)
                del logits
    return lse


def run_h2o_single_pass(args, batch, params, w, B, Q, K, V, roles, scores, keep, k_out, v_out, ws,
                        status, stream, world, seq_tokens, peaks, counts):
    """The H2O step with every query row's normaliser supplied by the caller
    (the prefill attention's softmax LSE): the score multiplies the keys once,
    then selection and compaction."""
    import torch

    from paper_2607_13205_gb300 import rolekv as R

    if w.varlen:
        return None
    torch.backends.cuda.matmul.allow_tf32 = False
    lse = prefill_lse(w, Q, K)
    torch.cuda.synchronize()

    def score():
        R.h2o_score(batch, Q, K, scores, lse=lse, ws=ws, status=status, stream=stream)

    def rest():
        R.role_alloc_select(batch, scores, roles, params, keep, pool_k=1, status=status, stream=stream)
        R.kv_compact(batch, K, V, keep, B, k_out, v_out, status=status, stream=stream)

    for _ in range(3):
        score()
        rest()
    steps = max(1, args.steps)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2 * steps + 1)]
    torch.cuda.synchronize()
    barrier(world)
    ev[0].record(stream)
    for i in range(steps):
        score()
        ev[2 * i + 1].record(stream)
        rest()
        ev[2 * i + 2].record(stream)
    torch.cuda.synchronize()
    barrier(world)
    total = max_over_ranks(ev[0].elapsed_time(ev[-1]), world)
    score_ms = sum(ev[2 * i].elapsed_time(ev[2 * i + 1]) for i in range(steps)) / steps
    if int(status.item()) != 0:
        raise SystemExit(f"device status {int(status.item())} in the single-pass H2O steps")
    flops = counts["score"]["flops"]
    return {"value": world * seq_tokens * steps / (total / 1e3), "unit": UNIT,
            "ms_per_step": total / steps, "score_ms": score_ms, "steps": steps,
            "score_tensor_frac": flops / (score_ms / 1e3) / 1e12 / peaks["bf16_tflops"],
            "lse": "every query row's normaliser supplied by the caller (computed once, untimed)"}


def run_decode(args, batch, w, B, K, V, keep, k_out, v_out, stream, world, peaks):
    """One decode step of attention (a new token per sequence, every head)
    through the compacted cache the step just built, and through the full
    cache, each timed over the same number of iterations."""
    import torch

    from paper_2607_13205_gb300 import inputs as I
    from paper_2607_13205_gb300 import rolekv as R

    qd = I.make_q_decode(w, 11, device=K.device)
    out = torch.empty((w.L, w.b, w.Hq, w.d), dtype=torch.float32, device=K.device)
    ws_c = R.decode_workspace(batch, B, device=K.device)
    ws_f = R.decode_workspace(batch, 1.0, device=K.device)
    units = w.L * w.b * w.Hkv
    rows_c = (sum(math.ceil(B * x) for x in w.seqlens) if w.varlen else w.b * math.ceil(B * w.n)) * w.L * w.Hkv
    rows_f = (sum(w.seqlens) if w.varlen else w.b * w.n) * w.L * w.Hkv
    del units

    def timed(fn, reps):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        barrier(world)
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            fn()
        e1.record(stream)
        torch.cuda.synchronize()
        return max_over_ranks(e0.elapsed_time(e1) / reps, world)

    reps = max(3, args.steps)
    t_c = timed(lambda: R.decode_attention(batch, qd, k_out, v_out, keep, B, out, ws=ws_c, stream=stream), reps)
    t_f = timed(lambda: R.decode_attention(batch, qd, K, V, None, 1.0, out, compacted=False, ws=ws_f,
                                           stream=stream), reps)
    by_c = rows_c * w.d * 2 * 2 + rows_c * 4
    by_f = rows_f * w.d * 2 * 2
    return {"compacted_ms": t_c, "full_ms": t_f, "speedup": t_f / t_c,
            "compacted_hbm_frac": by_c / (t_c / 1e3) / 1e9 / peaks["hbm_gbs"],
            "full_hbm_frac": by_f / (t_f / 1e3) / 1e9 / peaks["hbm_gbs"],
            "bytes": {"compacted": by_c, "full": by_f},
            "what": "one decode token per sequence, all heads; full = budget 1, no index"}


def run_e2e(args, score, batch, params, w, B, qw, K, V, roles, scores, keep, k_out, v_out, status,
            stream, world, seq_tokens):
    """The same step through the public calls with host buffers: the step's
    inputs come from pinned host memory and the kept indices and the
    compressed K/V are read back, inside the timed region.  K, the window
    queries and the roles are copied to the device (the score reads all of
    K); V stays in pinned host memory and kv_compact reads only its kept rows
    over the host link.  The step runs layer slice by layer slice on three
    streams, so that a slice's host-to-device copy, another slice's kernels
    and a third slice's read-back overlap (as a prefill that hands its cache
    over layer by layer would)."""
    import torch

    from paper_2607_13205_gb300 import rolekv as R

    h2o = w.kind == "h2o"
    dev = K.device
    h_qw = torch.empty(qw.shape, dtype=qw.dtype, pin_memory=True)
    h_k = torch.empty(K.shape, dtype=K.dtype, pin_memory=True)
    h_v = torch.empty(V.shape, dtype=V.dtype, pin_memory=True)
    h_roles = torch.empty(roles.shape, dtype=roles.dtype, pin_memory=True)
    h_qw.copy_(qw)
    h_k.copy_(K)
    h_v.copy_(V)
    h_roles.copy_(roles)
    o_keep = torch.empty(keep.shape, dtype=keep.dtype, pin_memory=True)
    o_k = torch.empty(k_out.shape, dtype=k_out.dtype, pin_memory=True)
    o_v = torch.empty(v_out.shape, dtype=v_out.dtype, pin_memory=True)
    torch.cuda.synchronize()
    bo = sum(t.numel() * t.element_size() for t in (o_keep, o_k, o_v))

    # layer slices; every tensor of the path has the layer axis first
    S = min(w.L, 8)
    bounds = [(w.L * i // S, w.L * (i + 1) // S) for i in range(S)]
    seqlens = list(w.seqlens) if w.varlen else None
    sbatch = {}
    for l0, l1 in bounds:
        if l1 - l0 not in sbatch:
            sbatch[l1 - l0] = R.Batch(l1 - l0, w.b, w.Hq, w.Hkv, w.d, w.n, seqlens=seqlens, device=dev,
                                      kept_extra=kept_extra(args.policy))
    big = sbatch[max(sbatch)]
    ws = R.workspace(R.OP_H2O if h2o else R.OP_SNAPKV, big, w.W, device=dev)
    pool_k = 1 if args.score == "quest" else w.pool_k
    s_in, s_out = torch.cuda.Stream(dev), torch.cuda.Stream(dev)
    ev_roles = torch.cuda.Event()
    ev_in = [torch.cuda.Event() for _ in bounds]
    ev_done = [torch.cuda.Event() for _ in bounds]
    ev_out = [torch.cuda.Event() for _ in bounds]

    def slice_kernels(i):
        l0, l1 = bounds[i]
        sb = sbatch[l1 - l0]
        if h2o:
            R.h2o_score(sb, qw[l0:l1], K[l0:l1], scores[l0:l1], ws=ws, status=status, stream=stream)
        elif args.score == "quest":
            R.quest_score(sb, qw[l0:l1], K[l0:l1], w.W, args.page, scores[l0:l1], stream=stream)
        else:
            R.snapkv_score(sb, qw[l0:l1], K[l0:l1], w.W, 1, scores[l0:l1], ws=ws, status=status,
                           stream=stream)
        R.role_alloc_select(sb, scores[l0:l1], roles, params, keep[l0:l1], pool_k=pool_k, status=status,
                            stream=stream)
        R.kv_compact(sb, K[l0:l1], h_v[l0:l1], keep[l0:l1], B, k_out[l0:l1], v_out[l0:l1], status=status,
                     stream=stream)

    def e2e_step():
        with torch.cuda.stream(s_in):
            s_in.wait_event(ev_done[-1])              # the roles' last use by the kernels
            roles.copy_(h_roles, non_blocking=True)
            ev_roles.record(s_in)
            for i, (l0, l1) in enumerate(bounds):
                s_in.wait_event(ev_done[i])            # the slice's last use by the kernels
                qw[l0:l1].copy_(h_qw[l0:l1], non_blocking=True)
                K[l0:l1].copy_(h_k[l0:l1], non_blocking=True)
                ev_in[i].record(s_in)
        stream.wait_event(ev_roles)
        for i in range(S):
            stream.wait_event(ev_in[i])
            stream.wait_event(ev_out[i])               # the slice's outputs were read back
            slice_kernels(i)
            ev_done[i].record(stream)
        with torch.cuda.stream(s_out):
            for i, (l0, l1) in enumerate(bounds):
                s_out.wait_event(ev_done[i])
                o_keep[l0:l1].copy_(keep[l0:l1], non_blocking=True)
                o_k[l0:l1].copy_(k_out[l0:l1], non_blocking=True)
                o_v[l0:l1].copy_(v_out[l0:l1], non_blocking=True)
                ev_out[i].record(s_out)

    e2e_step()
    torch.cuda.synchronize()
    # bytes in per step: the copies plus the kept V rows the compaction reads
    # from host memory (the step is the same every time)
    v_rows = int((keep >= 0).sum().item())
    bi = sum(t.numel() * t.element_size() for t in (h_qw, h_k, h_roles)) + v_rows * w.d * V.element_size()
    steps = max(1, min(args.steps, args.e2e_steps))
    barrier(world)
    torch.cuda.synchronize()
    t0 = time.perf_counter()
    for _ in range(steps):
        e2e_step()
    torch.cuda.synchronize()
    dt = time.perf_counter() - t0
    barrier(world)
    dt = max_over_ranks(dt, world)
    return {"value": world * seq_tokens * steps / dt, "unit": UNIT, "h2d_bytes_per_step": bi,
            "d2h_bytes_per_step": bo, "steps": steps, "ms_per_step": dt / steps * 1e3,
            "slices": S, "overlap": "layer slices: copy in (K, queries, roles), kernels (the compaction "
                                    "gathers the kept V rows from pinned host memory) and read-back on three streams"}


# ------------------------------------------------------ CPU oracle baseline --

POLICY_CODES = {"quota": 0, "global": 1, "fair": 2, "slack": 3, "ceil": 4}


def kept_extra(policy: str) -> int:
    """Kept-row slots beyond ceil(B n): the ceiling split's total can exceed
    the budget by one slot per weighted role but one."""
    return 3 if policy == "ceil" else 0      # four roles


def oracle_units(w, B, units, qw_bits, k_bits, v_bits, roles_np, policy="quota", keep_last=0,
                 score_kind="snapkv", page=16):
    """Score, select and compact the given units with the fp64 oracle."""
    from oracle import rolekv_oracle as O
    from paper_2607_13205_gb300 import inputs as I

    ob = O.Batch(w.L, w.b, w.Hq, w.Hkv, w.d, w.n, seqlens=list(w.seqlens) if w.varlen else None,
                 kept_extra=kept_extra(policy))
    if w.kind == "h2o":
        sc = O.h2o_batch(ob, qw_bits, k_bits, units=units)
        pooled = sc
    elif score_kind == "quest":
        pooled = O.quest_batch(ob, qw_bits, k_bits, w.W, page, units=units)
    else:
        sc = O.snapkv_batch(ob, qw_bits, k_bits, w.W, w.pool_k, units=units)
        pooled = {u: sc[u][1] for u in sc}
    sel = O.select_batch(ob, pooled, roles_np, I.N_ROLES, I.PAPER_ALPHA, I.ROLE_KEY, 0.0, B,
                         policy=POLICY_CODES[policy], keep_last=keep_last)
    for u, (idx, _) in sel.items():
        O.compact_unit(ob.kv_rows(k_bits, u), idx)
        O.compact_unit(ob.kv_rows(v_bits, u), idx)
    return sel


def _sample_arrays(w, units, host_inputs):
    """Host bf16 bit arrays holding (at least) the sampled units' data."""
    import numpy as np

    from paper_2607_13205_gb300 import inputs as I

    qw, K, V, roles_np = host_inputs
    layers = sorted({u // (w.b * w.Hkv) for u in units})
    assert layers == [0], "samples are taken from layer 0"
    qb = np.zeros((w.L,) + tuple(qw.shape[1:]), dtype=np.uint16)
    qb[0] = I.bf16_bits(qw[0])
    kb = np.zeros((1,) + tuple(K.shape[1:]), dtype=np.uint16)
    kb[0] = I.bf16_bits(K[0])
    vb = np.zeros_like(kb)
    vb[0] = I.bf16_bits(V[0])
    return qb, kb, vb, roles_np


def cpu_baseline(w, B, seconds: float, host_inputs, policy="quota", keep_last=0, score_kind="snapkv",
                 page=16):
    """The oracle as it stands on this host's cores, on units of layer 0 of
    the same workload until `seconds` of CPU work, extrapolated to a step."""
    U = w.L * w.b * w.Hkv
    per_layer = w.b * w.Hkv
    units = []
    qb = kb = vb = roles_np = None
    t_total = 0.0
    done = 0
    while True:
        u = done % per_layer
        if qb is None:
            qb, kb, vb, roles_np = _sample_arrays(w, [u], host_inputs)
        t0 = time.perf_counter()
        oracle_units(w, B, [u], qb, kb, vb, roles_np, policy, keep_last, score_kind, page)
        t_total += time.perf_counter() - t0
        done += 1
        units.append(u)
        # layer 0's units, repeated if they take less than `seconds`
        if t_total >= seconds or done >= 8 * per_layer:
            break
    seq_tokens = w.b * w.n if not w.varlen else sum(w.seqlens)
    value = (done / U) * seq_tokens / t_total
    return {"value": value, "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
            "sample": f"{done} unit passes over the {min(done, per_layer)} (sequence, KV head) units of "
                      f"layer 0 (the step has {U}), {t_total:.1f} s, extrapolated linearly to the full step",
            "seconds": t_total}


def blas_threads() -> int:
    for var in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(var):
            try:
                return int(os.environ[var])
            except ValueError:
                pass
    return os.cpu_count() or 1


def run_reference(args):
    """The reference arm: the fp64 oracle, timed as it stands, each step a
    bounded sample of the workload's units (rank 0 only)."""
    rank, world, _ = dist_env()
    if rank != 0:
        return
    import numpy as np
    import torch

    from paper_2607_13205_gb300 import inputs as I

    w = I.WORKLOADS[args.workload]
    B = args.budget if args.budget else w.budgets[0]
    w1 = w.scaled(L=1)
    roles_np = I.workload_roles(w1, seed=0)
    K, V = I.make_kv(w1, roles_np, seed=0, device="cpu")
    qw = (I.make_q_full if w.kind == "h2o" else I.make_q_window)(w1, seed=0, device="cpu")
    qb, kb, vb = I.bf16_bits(qw), I.bf16_bits(K), I.bf16_bits(V)
    U = w.L * w.b * w.Hkv
    per_step = max(1, args.ref_units)
    seq_tokens = w.b * w.n
    nxt = 0

    def step():
        nonlocal nxt
        units = [(nxt + i) % (w1.b * w1.Hkv) for i in range(per_step)]
        nxt += per_step
        oracle_units(w1, B, units, qb, kb, vb, roles_np, args.policy, args.keep_last, args.score,
                     args.page)

    for _ in range(args.warmup):
        step()
    t0 = time.perf_counter()
    for _ in range(args.steps):
        step()
    dt = time.perf_counter() - t0
    value = (per_step * args.steps / U) * seq_tokens / dt
    sample = (f"{per_step} of {U} (layer, sequence, KV head) units per step, extrapolated "
              "linearly to the full workload")
    out = {"metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
           "warmup": args.warmup, "ms_per_step": dt / args.steps * U / per_step * 1e3,
           "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
           "data": "synthetic", "impl": "reference",
           "config": {"workload": f"{w.name}: L={w.L} b={w.b} Hq={w.Hq} Hkv={w.Hkv} d={w.d} "
                                  f"N={w.n} W={w.W} pool={w.pool_k} B={B}",
                      "global_batch": w.b, "seq_len": w.n, "parallelism": "cpu"},
           "cpu_baseline": {"value": value, "unit": UNIT, "cores": blas_threads(), "kind": "oracle",
                            "sample": sample},
           "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="long")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-single-pass", action="store_true",
                    help="skip the step with caller-supplied window normalisers")
    ap.add_argument("--e2e-steps", type=int, default=3)
    ap.add_argument("--no-decode", action="store_true",
                    help="skip the decode-step timing through the compacted and the full cache")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-seconds", type=float, default=12.0)
    ap.add_argument("--ref-units", type=int, default=2)
    ap.add_argument("--budget", type=float, default=0.0, help="override the workload's budget")
    ap.add_argument("--score", choices=["snapkv", "quest"], default="snapkv",
                    help="score of the SnapKV workloads: windowed mass, or the Quest page bound")
    ap.add_argument("--page", type=int, default=16, help="tokens per page of the Quest bound")
    ap.add_argument("--policy", choices=["quota", "global", "fair", "slack", "ceil"], default="quota",
                    help="budget split: role quotas (the method), plain top-k, fair eviction, or "
                         "role quotas with the slack of saturated buckets filled by score")
    ap.add_argument("--keep-last", type=int, default=0,
                    help="recency floor: always keep each sequence's last tokens")
    ap.add_argument("--layers", type=int, default=0,
                    help="override the layer count (smaller cases for profiling)")
    ap.add_argument("--traffic", type=float, default=None,
                    help="dram bytes per launch of the dominant kernel from an ncu capture")
    ap.add_argument("--all-configs", action="store_true",
                    help="one JSON line per benchmark configuration: tiny, llama8b at each of "
                         "its budgets, long, h2o and ragged (no e2e or decode legs)")
    args = ap.parse_args(argv)
    if args.warmup < 3 and args.impl == "ours":
        print("warning: fewer than 3 warm-up steps", file=sys.stderr)
    if args.impl == "reference":
        run_reference(args)
    elif args.all_configs:
        run_all_configs(args)
    else:
        run_gpu(args)


def run_all_configs(args):
    """Every benchmark configuration in turn on one GPU (the budgets of the
    8B configuration each), one JSON line each, with a shorter CPU sample."""
    import gc

    import torch

    from paper_2607_13205_gb300 import inputs as I

    _, world, _ = dist_env()
    if world > 1:
        raise SystemExit("--all-configs runs on one GPU")
    sweep = [("tiny", B) for B in I.WORKLOADS["tiny"].budgets]
    sweep += [("llama8b", B) for B in I.WORKLOADS["llama8b"].budgets]
    sweep += [("long", B) for B in I.WORKLOADS["long"].budgets]
    sweep += [("h2o", B) for B in I.WORKLOADS["h2o"].budgets]
    sweep += [("ragged", B) for B in I.WORKLOADS["ragged"].budgets]
    for name, B in sweep:
        a = argparse.Namespace(**vars(args))
        a.workload, a.budget = name, B
        a.no_e2e, a.no_decode = True, True
        a.cpu_seconds = min(args.cpu_seconds, 5.0)
        run_gpu(a)
        gc.collect()
        torch.cuda.empty_cache()


if __name__ == "__main__":
    main()
