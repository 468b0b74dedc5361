#!/usr/bin/env python
"""Throughput of the DeLS-Spec per-block drafting hot path on GB300.

One step = one pass of the whole hot path over one batch: dels_draft_block
(position 0 from the DFlash logits, then for each later position the GRU
local head, the tcgen05 vocabulary projection fused with the Section 4.3
combine, and the merge that feeds the token back) followed by
dels_verify_block (greedy verification against the target logits).

Workload: Qwen3-8B-shaped batched drafting — B = 64 requests, block n = 16,
vocabulary V = 151936, the Appendix A GRU head (target embedding 4096, GRU
hidden 1024, rank 256), bf16 weights N(0, 0.02), bf16 DFlash logits N(0, 3)
plus a Zipf(1.1) bias, target logits = DFlash + N(0, 1). Synthetic data; the
paper's checkpoints and benchmark prompts are not used.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]
                  [--workload qwen3_8b_batched|qwen3_4b|qwen3_0p6b|tiny]

--workload picks one of the other Qwen3-shaped drafting workloads (same
step, their own head and logits): Qwen3-4B-shaped (B = 8, 1-layer causal
transformer head, d 2560, FFN 10240, float32 logits), Qwen3-0.6B-shaped
(B = 1, 2-layer window MLP head over the last 4 tokens, hidden 1024, float32
logits) and the tiny case (B = 1, V = 1024, float32 MLP head).

Prints one JSON line (rank 0). N > 1 runs one independent replica per GPU
(launched by torchrun): the drafting path has no cross-request exchange.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "drafted tokens/sec on 1 GB300; combine/argmax HBM GB/s vs 8 TB/s; oracle match"
UNIT = "drafted tokens/s"
WORKLOAD = "qwen3_8b_batched"
WORKLOADS = ("qwen3_8b_batched", "qwen3_4b", "qwen3_0p6b", "tiny")
FALLBACK_HBM_GBS = 6800.0
NOMINAL_HBM_GBS = 8000.0      # the "8 TB/s" of the metric (GB300 HBM3e nominal, rounded)
L2_BYTES = 129e6


def parse_args():
    p = argparse.ArgumentParser()
    p.add_argument("--gpus", type=int, default=1)
    p.add_argument("--steps", type=int, default=200)
    p.add_argument("--warmup", type=int, default=5)
    p.add_argument("--impl", choices=["ours", "reference"], default="ours")
    p.add_argument("--e2e-steps", type=int, default=20)
    p.add_argument("--cpu-rows", type=int, default=4, help="requests in the CPU-oracle baseline sample")
    p.add_argument("--no-cpu-baseline", action="store_true")
    p.add_argument("--sweep", action="store_true",
                   help="instead of the drafting step: HBM GB/s of dels_combine_argmax and dels_verify_block over "
                        "the combine/verify sweep grid (one JSON line per point)")
    p.add_argument("--point", default=None, metavar="V,DTYPE,B,N",
                   help="with --sweep: only this point of the grid, e.g. 151936,bf16,64,16")
    p.add_argument("--temperature", type=int, choices=[0, 1], default=0,
                   help="1: the temperature-1 step instead (Gumbel-max drafting + speculative-sampling "
                        "verification), printed as its own JSON line")
    p.add_argument("--variant", choices=["gru", "wide"], default="gru",
                   help="wide: the same step with a 4096-wide vocabulary projection (a Markov head over the "
                        "4096-wide token state, W [V, 4096]) instead of the GRU head, printed as its own line")
    p.add_argument("--prior", action="store_true",
                   help="instead of the drafting step: device unigram-prior estimation (masked token histogram, "
                        "smoothing, log) over a 2^28-position synthetic chat corpus")
    p.add_argument("--no-graph", action="store_true",
                   help="time stream launches instead of replays of a CUDA graph of the step")
    p.add_argument("--no-input-table", action="store_true",
                   help="recompute the GRU input product W_ih E[x] at every position instead of reading the "
                        "precomputed table G = E W_ih^T")
    p.add_argument("--workload", choices=WORKLOADS, default=WORKLOAD,
                   help="drafting workload of the step (default: the Qwen3-8B-shaped batched drafting)")
    p.add_argument("--cpu-positions", type=int, default=0,
                   help="block positions in the CPU-oracle sample (0: the workload's default)")
    p.add_argument("--oracle-single-thread", action="store_true", help=argparse.SUPPRESS)
    return p.parse_args()


# ----------------------------------------------------------------------------- helpers

def dist_setup(n_expected):
    import torch
    import torch.distributed as dist
    from paper_2607_07409_gb300 import replicas
    world, rank, local = replicas.rank_info()
    if world > 1 and not dist.is_initialized():
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    return world, rank, local


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as fh:
            d = json.load(fh)
        return float(d["hbm_gbs"]), "measured"
    except Exception:
        return FALLBACK_HBM_GBS, "fallback"


def kernel_source_digest():
    h = hashlib.sha256()
    for name in ("tc_gemm.cu", "tc_engine.cuh", "dels_device.cuh"):
        with open(os.path.join(ROOT, "paper_2607_07409_gb300", "csrc", name), "rb") as fh:
            h.update(fh.read())
    return h.hexdigest()[:16]


def ncu_traffic(profile_name):
    """Per-launch DRAM bytes of the dominant kernel from the committed ncu
    summary, if it was captured on the current kernel source."""
    path = os.path.join(ROOT, "profiles", profile_name)
    try:
        txt = open(path).read()
    except OSError:
        return None
    m = re.search(r"traffic_bytes_per_launch:\s*([0-9.eE+]+)", txt)
    s = re.search(r"kernel_source_digest:\s*([0-9a-f]+)", txt)
    if not m or not s or s.group(1) != kernel_source_digest():
        return None
    return float(m.group(1))


class ClockSampler:
    """nvidia-smi clock / throttle-reason samples while the timed region runs."""

    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id):
        self.gpu_id = gpu_id
        self.proc = None
        self.out = None

    def __enter__(self):
        try:
            self.out = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu_id), f"--query-gpu={self.FIELDS}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.out, stderr=subprocess.DEVNULL)
            time.sleep(0.3)
        except Exception:
            self.proc = None
        return self

    def __exit__(self, *exc):
        if self.proc is not None:
            time.sleep(0.15)
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self):
        if self.proc is None or self.out is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unavailable"]}
        self.out.flush()
        rows = []
        with open(self.out.name) as fh:
            for line in fh:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9 and parts[1].replace(".", "").isdigit():
                    rows.append(parts)
        os.unlink(self.out.name)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": float(rows[0][2]), "reasons": reasons,
                "samples": len(rows), "power_w_max": max(float(r[3]) for r in rows if _isnum(r[3]))}


def _isnum(s):
    try:
        float(s)
        return True
    except ValueError:
        return False


def _es(dtype):
    return 4 if dtype == "f32" else 2


def algorithmic_vocab_bytes(w):
    """Bytes one vocabulary-projection + combine launch must move: W_vocab once,
    the DFlash logits of one position for every request, the prior, and the
    projection's input r."""
    h = w.head
    esw, esl = _es(h.wdtype), _es(w.logit_dtype)
    return w.V * h.d_rank * esw + w.B * w.V * esl + w.V * 4 + w.B * h.d_rank * esw


def head_weight_bytes(w, table=False):
    """Bytes of the local head's own weights streamed at one drafted position,
    and of the inputs it gathers per position. table: the GRU's input product
    is read as B rows of G = E W_ih^T (3 * d_hidden float32 each) instead of
    streaming W_ih and gathering E rows."""
    h = w.head
    esw = _es(h.wdtype)
    if h.kind == "gru":
        if table:
            return (3 * h.d_hidden * h.d_hidden + h.d_rank * h.d_hidden) * esw, w.B * 3 * h.d_hidden * 4
        return (3 * h.d_hidden * (h.d_model + h.d_hidden) + h.d_rank * h.d_hidden) * esw, w.B * h.d_model * esw
    if h.kind == "mlp":
        wb = h.d_hidden * h.window * h.d_model + (h.d_hidden * h.d_hidden if h.n_layers == 2 else 0)
        return wb * esw, w.B * h.window * h.d_model * esw
    if h.kind == "xfmr":
        D, F = h.d_model, h.d_hidden
        return (4 * D * D + 2 * D * F) * esw, w.B * D * esw
    return 0, w.B * h.d_rank * esw                       # markov: one E_M row per request


def step_bytes(w, table=False):
    """Algorithmic bytes of one step (drafted block + verification): every
    weight once per drafted position j >= 1, W_vocab included, the DFlash
    logits of every position, the prior, the gathered head inputs, and the
    n + 1 target rows of every request. table=False is the streaming model
    (every head weight, W_ih included); table=True what the GRU input-table
    path reads."""
    h = w.head
    esl = _es(w.logit_dtype)
    hw, gather = head_weight_bytes(w, table)
    per_pos = w.V * h.d_rank * _es(h.wdtype) + hw + w.B * w.V * esl + w.V * 4 + gather
    return (w.n - 1) * per_pos + w.B * w.V * esl + w.B * (w.n + 1) * w.V * esl


# ----------------------------------------------------------------------------- CPU oracle leg

def default_cpu_positions(w):
    """Block positions in the CPU-oracle sample: the oracle decodes W_vocab to
    float64 at every position, which dominates for the wide heads."""
    return {"qwen3_4b": 6, "qwen3_0p6b": 12}.get(w.name, w.n)


def oracle_single_thread(args):
    """Child process: the oracle sample on one host thread (BLAS pinned to one
    thread by the parent's environment, torch's intra-op pool set to one);
    inputs from the same generators on the host. Prints one JSON line."""
    import torch
    import synth
    w = synth.WORKLOADS[args.workload]
    d = synth.make_inputs(w, device="cpu")
    torch.set_num_threads(1)
    positions = args.cpu_positions or default_cpu_positions(w)
    rows = min(args.cpu_rows, w.B)
    ntok, dt, _, _ = oracle_sample(w, d, rows, positions)
    print(json.dumps({"tokens": ntok, "seconds": dt, "rows": rows, "positions": positions}), flush=True)
    return 0


def single_thread_baseline(args, w):
    """The oracle sample timed on one host thread in a child process (None on failure)."""
    env = dict(os.environ, OMP_NUM_THREADS="1", OPENBLAS_NUM_THREADS="1", MKL_NUM_THREADS="1")
    cmd = [sys.executable, os.path.join(ROOT, "bench.py"), "--oracle-single-thread", "--workload", w.name,
           "--cpu-rows", str(max(1, min(args.cpu_rows, 2))), "--cpu-positions", str(args.cpu_positions)]
    try:
        r = subprocess.run(cmd, env=env, capture_output=True, text=True, timeout=600)
        out = json.loads(r.stdout.strip().splitlines()[-1])
    except Exception:
        return None
    return {"value": out["tokens"] / out["seconds"], "unit": UNIT, "cores": 1,
            "sample": f"{out['rows']} of {w.B} requests x positions 0..{out['positions'] - 1} of {w.name} "
                      f"(inputs from the host generators)"}


def oracle_sample(w, d, rows, positions, gpu_tokens=None):
    """Time the oracle on `rows` requests x `positions` positions of the block
    (plus their greedy verification); optionally check the device's tokens."""
    import numpy as np
    import oracle
    W = {k[5:]: v.cpu() for k, v in d.items() if k.startswith("head.")}
    long = d["long"][:rows, :positions].cpu()
    target = d["target"][:rows].cpu()
    prior = oracle.log_prior(d["counts"])
    t0 = time.perf_counter()
    forced = None if gpu_tokens is None else gpu_tokens[:rows, :positions]
    res = oracle.draft_block(oracle.make_head(w.head, W), long, prior, w.alpha, w.beta, forced=forced)
    if positions == w.n:
        oracle.verify_greedy(res.tokens, target)
    dt = time.perf_counter() - t0
    match = None
    if forced is not None:
        same = forced == res.argmax
        near = (res.gap < 1e-3) & (res.fused_at >= res.fused_max - 1e-3)
        match = {"rows": rows, "positions": positions, "tokens_equal": int(same.sum()),
                 "tokens_total": int(same.size), "near_ties": int((res.gap < 1e-3).sum()),
                 "ok": bool(np.all(same | near))}
    return rows * positions, dt, match, res


def cpu_cores():
    try:
        return len(os.sched_getaffinity(0))
    except Exception:
        return os.cpu_count()


# ----------------------------------------------------------------------------- reference arm

def run_reference(args):
    world, rank, _ = dist_setup(args.gpus)
    if rank != 0:
        return 0
    import torch
    import synth
    w = synth.WORKLOADS[args.workload]
    d = synth.make_inputs(w, device="cpu")
    rows, positions = 1, min(4, w.n)
    for _ in range(args.warmup):
        oracle_sample(w, d, rows, positions)
    times = []
    tokens = 0
    for _ in range(args.steps):
        t, dt, _, _ = oracle_sample(w, d, rows, positions)
        tokens += t
        times.append(dt)
    total = sum(times)
    value = tokens / total
    sample = f"{rows} of {w.B} requests x positions 0..{positions - 1} of {w.name} per step"
    line = {
        "impl": "reference", "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": args.gpus,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": 1e3 * total / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
        "config": {"workload": w.name, "B": w.B, "n": w.n, "V": w.V, "head": head_desc(w)},
        "cpu_baseline": {"value": value, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle", "sample": sample},
        "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)
    return 0


# ----------------------------------------------------------------------------- our arm

def head_desc(w):
    h = w.head
    if h.kind == "gru":
        return f"gru emb {h.d_model} / hidden {h.d_hidden} / rank {h.d_rank}, {h.wdtype}"
    if h.kind == "mlp":
        return f"{h.n_layers}-layer window-{h.window} mlp, d {h.d_model} / hidden {h.d_hidden}, {h.wdtype}"
    if h.kind == "xfmr":
        return f"1-layer causal transformer d {h.d_model} / {h.n_heads} heads / ffn {h.d_hidden}, {h.wdtype}"
    return f"markov d {h.d_rank}, {h.wdtype}"


def run_ours(args):
    import torch
    import torch.distributed as dist
    import synth
    import paper_2607_07409_gb300 as dels

    from paper_2607_07409_gb300 import replicas

    world, rank, local = dist_setup(args.gpus)
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    # weak scaling: every replica drafts its own batch of the same shape
    w0 = synth.WORKLOADS[args.workload]
    w = synth.with_sizes(w0, seed=replicas.replica_seed(w0.seed, rank))
    d = synth.make_inputs(w, device=dev)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = dels.dels_prior_from_counts(d["counts"]).to(dev)
    long, target = d["long"], d["target"]
    ldt, tdt = dels.dtype_code(long), dels.dtype_code(target)
    table_ms = None
    use_table = w.head.kind == "gru" and w.head.wdtype == "bf16" and not args.no_input_table
    if use_table:
        # head preparation, once per set of weights (not part of a step)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        W["input_table"] = dels.gru_input_table(w.head, W, w.V)
        torch.cuda.synchronize()
        table_ms = 1e3 * (time.perf_counter() - t0)
    drafter = dels.Drafter(w.head, W, w.B, w.n, w.V)
    vbytes = dels.dels_verify_workspace_bytes(w.B, w.n, w.V, tdt)
    vws = torch.zeros(vbytes, dtype=torch.uint8, device=dev)
    acc = torch.empty(w.B, dtype=torch.int32, device=dev)
    bonus = torch.empty(w.B, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    def step(long_in, target_in, st=stream):
        tok, lp, gap = drafter(long_in, prior, w.alpha, w.beta, st)
        r = dels.dels_verify_block(tok, target_in, tdt, w.B, w.n, w.V, acc, bonus, None, vws, vbytes, st)
        if r != 0:
            raise dels.DelsError(r, "dels_verify_block")
        return tok

    for _ in range(max(3, args.warmup)):
        step(long, target)
    torch.cuda.synchronize()
    if drafter.status() != 0 or dels.dels_read_status(vws) != 0:
        raise RuntimeError("device status set during warm-up")

    moved = step_bytes(w, table=use_table)
    survey = step_bytes(w, table=False)
    # a step whose bytes fit in L2 is timed launch by launch with an L2 flush
    # (a write larger than L2) between steps, outside the timed brackets
    flush_l2 = moved < 2 * L2_BYTES
    flush = torch.empty(int(2 * L2_BYTES), dtype=torch.uint8, device=dev) if flush_l2 else None

    # ---- timed region: device-resident inputs
    gpu_id = local
    try:
        gpu_id = "GPU-" + str(torch.cuda.get_device_properties(dev).uuid)
    except Exception:
        pass
    replicas.barrier()
    torch.cuda.synchronize()
    # The step is captured once as a CUDA graph (every launch of the library
    # is stream-ordered, with no host synchronisation); the timed region
    # replays it on the same stream.
    graph = None
    if not args.no_graph:
        cap = torch.cuda.Stream(device=dev)
        cap.wait_stream(stream)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=cap):
            step(long, target, cap)
        stream.wait_stream(cap)
        for _ in range(3):
            graph.replay()
        torch.cuda.synchronize()

    def one():
        if graph is not None:
            graph.replay()
        else:
            step(long, target)

    with ClockSampler(gpu_id) as clk:
        if flush_l2:
            evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                   for _ in range(args.steps)]
            for i in range(args.steps):
                flush.fill_(i & 0xFF)
                evs[i][0].record(stream)
                one()
                evs[i][1].record(stream)
            torch.cuda.synchronize()
            ms_local = sum(a.elapsed_time(b) for a, b in evs)
        else:
            e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            e0.record(stream)
            for _ in range(args.steps):
                one()
            e1.record(stream)
            torch.cuda.synchronize()
            ms_local = e0.elapsed_time(e1)
    replicas.barrier()
    ms_max = replicas.max_over_ranks(ms_local, dev)

    # ---- second timed region, same steps, with the library's per-kernel CUDA
    # events on (they serialise the kernels, so the value above is taken without)
    k_prof = max(1, min(args.steps, 50))
    dels.dels_profile_reset()
    dels.dels_profile_enable(True)
    torch.cuda.synchronize()
    for _ in range(k_prof):
        step(long, target)
    torch.cuda.synchronize()
    dels.dels_profile_enable(False)
    kernels = {}
    launches_prof = 0
    for name, cls in dels.KCLASS.items():
        n_l, tot = dels.dels_profile_read(cls)
        launches_prof += n_l
        if n_l:
            kernels[name] = {"launches_per_step": n_l / k_prof, "ms_per_step": tot / k_prof,
                             "us_per_launch": 1e3 * tot / n_l}
    dels.dels_profile_reset()
    launches = int(round(launches_prof / k_prof)) * args.steps
    if drafter.status() != 0 or dels.dels_read_status(vws) != 0:
        raise RuntimeError("device status set during the timed region")
    tokens_per_step = w.B * w.n
    value = replicas.job_throughput([tokens_per_step * args.steps] * world, ms_max)

    # ---- roofline of the dominant kernel (vocabulary projection + combine)
    peak, peak_kind = measured_peaks()
    vc = kernels.get("vocab_combine")
    roofline = None
    if vc:
        per_launch_s = vc["us_per_launch"] * 1e-6
        achieved = algorithmic_vocab_bytes(w) / per_launch_s / 1e9
        roofline = {"bound": "hbm", "achieved": round(achieved, 1), "peak": peak, "unit": "GB/s",
                    "frac": round(achieved / peak, 4), "peak_source": peak_kind,
                    "frac_of_nominal_8tbs": round(achieved / NOMINAL_HBM_GBS, 4),
                    "kernel": ("k_tc_gemm<1> (vocab projection + fused combine)" if w.head.wdtype == "bf16" else
                               "k_vocab_combine_f32 (vocab projection + fused combine, CUDA cores)"),
                    "algorithmic_bytes_per_launch": algorithmic_vocab_bytes(w),
                    "traffic": ncu_traffic(f"vocab_combine_{w.name}.md")}
    step_s = ms_max / args.steps * 1e-3

    # ---- end to end through the public API with host buffers: every step
    # copies its logits in from pinned host memory and reads its tokens,
    # accept lengths and bonus tokens back. Double-buffered like a serving
    # loop: the inputs of step k + 1 are copied on a second stream while step
    # k computes (the host link, ~210 GB/s on this machine whether the copy is
    # DMA on one or several streams or an SM kernel reading pinned memory,
    # is the bound).
    long_h = long.cpu().pin_memory()
    target_h = target.cpu().pin_memory()
    bufs = [(torch.empty_like(long), torch.empty_like(target)) for _ in range(2)]
    tok_h = torch.empty(w.B, w.n, dtype=torch.int32).pin_memory()
    acc_h = torch.empty(w.B, dtype=torch.int32).pin_memory()
    bonus_h = torch.empty(w.B, dtype=torch.int32).pin_memory()
    k_e2e = max(1, min(args.e2e_steps, args.steps))
    copy_s = torch.cuda.Stream(device=dev)
    copied = [torch.cuda.Event() for _ in range(2)]
    freed = [torch.cuda.Event() for _ in range(2)]
    replicas.barrier()
    torch.cuda.synchronize()
    f0, f1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    f0.record(stream)
    copy_s.wait_stream(stream)
    for k in range(k_e2e):
        i = k % 2
        long_d, target_d = bufs[i]
        if k >= 2:
            copy_s.wait_event(freed[i])           # step k - 2 is done with this buffer
        with torch.cuda.stream(copy_s):
            long_d.copy_(long_h, non_blocking=True)
            target_d.copy_(target_h, non_blocking=True)
            copied[i].record(copy_s)
        stream.wait_event(copied[i])
        tok = step(long_d, target_d)
        tok_h.copy_(tok, non_blocking=True)
        acc_h.copy_(acc, non_blocking=True)
        bonus_h.copy_(bonus, non_blocking=True)
        freed[i].record(stream)
    f1.record(stream)
    torch.cuda.synchronize()
    e2e_ms = replicas.max_over_ranks(f0.elapsed_time(f1), dev)
    e2e_val = replicas.job_throughput([tokens_per_step * k_e2e] * world, e2e_ms)
    h2d = long.numel() * long.element_size() + target.numel() * target.element_size()
    d2h = tok_h.numel() * 4 + acc_h.numel() * 4 + bonus_h.numel() * 4

    # ---- the recompute path of the same head (W_ih E[x] streamed every
    # position instead of rows of the input table), same inputs, same timing
    recompute = None
    if use_table and world == 1:
        W_rc = {k: v for k, v in W.items() if k != "input_table"}
        dr_rc = dels.Drafter(w.head, W_rc, w.B, w.n, w.V)

        def step_rc(long_in, target_in, st=stream):
            tok_rc, _, _ = dr_rc(long_in, prior, w.alpha, w.beta, st)
            r = dels.dels_verify_block(tok_rc, target_in, tdt, w.B, w.n, w.V, acc, bonus, None, vws, vbytes, st)
            if r != 0:
                raise dels.DelsError(r, "dels_verify_block")

        for _ in range(3):
            step_rc(long, target)
        torch.cuda.synchronize()
        g_rc = None
        if not args.no_graph:
            cap = torch.cuda.Stream(device=dev)
            cap.wait_stream(stream)
            g_rc = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g_rc, stream=cap):
                step_rc(long, target, cap)
            stream.wait_stream(cap)
            for _ in range(3):
                g_rc.replay()
        torch.cuda.synchronize()
        k_rc = max(1, min(args.steps, 100))
        h0, h1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        h0.record(stream)
        for _ in range(k_rc):
            if g_rc is not None:
                g_rc.replay()
            else:
                step_rc(long, target)
        h1.record(stream)
        torch.cuda.synchronize()
        if dr_rc.status() != 0 or dels.dels_read_status(vws) != 0:
            raise RuntimeError("device status set on the recompute path")
        rc_ms = h0.elapsed_time(h1) / k_rc
        rc_bytes = step_bytes(w, table=False)
        recompute = {"value": tokens_per_step / (rc_ms * 1e-3), "unit": UNIT, "ms_per_step": rc_ms,
                     "steps": k_rc, "bytes_read": rc_bytes,
                     "frac_read": round(rc_bytes / (rc_ms * 1e-3) / 1e9 / peak, 4),
                     "frac_read_of_nominal_8tbs": round(rc_bytes / (rc_ms * 1e-3) / 1e9 / NOMINAL_HBM_GBS, 4),
                     "note": "the same head without the input table (python bench.py --no-input-table)"}
        del g_rc, dr_rc

    # ---- acceptance statistics of the drafted blocks (Appendix D rate_i)
    a = acc.cpu().numpy()
    rates = [float((a + 1 >= i).mean()) for i in range(1, w.n + 2)]

    # ---- CPU oracle baseline + oracle match on a sample (rank 0, N = 1)
    cpu = None
    match = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        gpu_tok = drafter.tokens.cpu().numpy()
        rows = min(args.cpu_rows, w.B)
        positions = args.cpu_positions or default_cpu_positions(w)
        ntok, dt, match, _ = oracle_sample(w, d, rows, positions, gpu_tokens=gpu_tok)
        cpu = {"value": ntok / dt, "unit": UNIT, "cores": cpu_cores(), "kind": "oracle",
               "sample": f"{rows} of {w.B} requests x positions 0..{positions - 1} of {w.name} "
                         f"({'+ their verification, ' if positions == w.n else ''}forced to the device's tokens)",
               "single_thread": single_thread_baseline(args, w)}

    if rank == 0:
        esl = _es(w.logit_dtype)
        line = {
            "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
            "warmup": max(3, args.warmup), "ms_per_step": ms_max / args.steps, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": w.head.wdtype, "data": "synthetic",
            "config": {"workload": w.name, "B": w.B, "n": w.n, "V": w.V, "head": head_desc(w),
                       "logits": f"{w.logit_dtype} DFlash and target logits",
                       "alpha": w.alpha, "beta": w.beta,
                       "step": "dels_draft_block + dels_verify_block",
                       "launch": ("stream launches" if args.no_graph else
                                  "CUDA graph of the step (captured once, replayed)"),
                       "gru_input": (None if w.head.kind != "gru" else
                                     "W_ih E[x] recomputed every position" if table_ms is None else
                                     f"table G = E W_ih^T ({w.V * 3 * w.head.d_hidden * 4 / 1e9:.2f} GB f32) "
                                     f"built once before timing in {table_ms:.1f} ms"),
                       "l2": ("L2 flushed (a 258 MB write) before every step; steps timed one by one"
                              if flush_l2 else
                              f"inputs larger than L2 (weights, DFlash logits {w.B * w.n * w.V * esl / 1e6:.0f} MB "
                              f"and target logits {w.B * (w.n + 1) * w.V * esl / 1e6:.0f} MB per step, not flushed)"),
                       "parallelism": f"replicas x{world}"},
            "roofline": roofline,
            "step_roofline": {"bytes_read": moved,
                              "gbs_read": round(moved / step_s / 1e9, 1),
                              "frac_read": round(moved / step_s / 1e9 / peak, 4),
                              "frac_read_of_nominal_8tbs": round(moved / step_s / 1e9 / NOMINAL_HBM_GBS, 4),
                              "streaming_model_bytes": survey,
                              "note": "bytes_read: what this path must read per step (drafted block + verification); "
                                      "streaming_model_bytes: every head weight streamed once per position "
                                      "(W_ih included), for comparison only"},
            "kernels": kernels,
            "recompute_path": recompute,
            "gpu_launches": launches,
            "e2e": {"value": e2e_val, "unit": UNIT, "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
                    "steps": k_e2e, "copies": "pinned host memory; step k + 1's inputs copied on a second "
                                              "stream while step k computes (two device buffers)"},
            "clocks": clk.summary(),
            "cpu_baseline": cpu,
            "oracle_match": match,
            "acceptance": {"tau": float((a + 1).mean()), "rate": rates[:6]},
        }
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def run_sweep(args):
    """dels_combine_argmax over rows = B*n independent rows [rows, V] (long and
    short logits plus the prior) and dels_verify_block over [B, n+1, V] target
    logits, for every (V, dtype, B, n) of the sweep grid. The combination
    weight does not change the bytes a call moves, so the timing runs at
    w = 0.5 (parity over the weights is in the tests). Each launch is timed
    alone with CUDA events after an L2 flush (a 256 MB write)."""
    import torch
    import synth
    import paper_2607_07409_gb300 as dels
    from paper_2607_07409_gb300 import replicas
    world, rank, local = dist_setup(args.gpus)
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    peak, peak_kind = measured_peaks()
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    reps = max(3, min(args.steps, 10))
    seen = set()

    def timed(fn):
        ts = []
        for i in range(reps + 2):
            flush.fill_(i & 0xFF)
            a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
            a.record()
            fn()
            b.record()
            b.synchronize()
            if i >= 2:
                ts.append(a.elapsed_time(b) * 1e-3)
        return statistics.median(ts)

    only = None
    if args.point:
        v_, d_, b_, n_ = args.point.split(",")
        only = (int(v_), d_, int(b_), int(n_))
    points = [only] if only else [(pt["V"], pt["dtype"], pt["B"], pt["n"]) for pt in synth.sweep_points()]
    for key in points:
        if key in seen:
            continue
        seen.add(key)
        V, dt, B, n = key
        es = 4 if dt == "f32" else 2
        rows = B * n
        d = synth.make_combine_inputs(rows, V, dt, seed=B * 131 + n * 7 + V % 97, device=dev)
        prior = dels.dels_prior_from_counts(d["counts"]).to(dev)
        code = dels.dtype_code(d["long"])
        cb = dels.dels_combine_workspace_bytes(rows, V, code)
        cws = torch.zeros(cb, dtype=torch.uint8, device=dev)
        tok = torch.empty(rows, dtype=torch.int32, device=dev)
        lp = torch.empty(rows, dtype=torch.float32, device=dev)
        gap = torch.empty(rows, dtype=torch.float32, device=dev)

        def comb():
            r = dels.dels_combine_argmax(d["long"], d["short"], code, prior, 0.5, 0.5, rows, V, tok, lp, gap, cws, cb)
            if r != 0:
                raise dels.DelsError(r, "dels_combine_argmax")

        t_c = timed(comb)
        c_bytes = 2 * rows * V * es + 4 * V + 12 * rows
        del d
        target = torch.empty(B, n + 1, V, dtype=torch.float32 if dt == "f32" else torch.bfloat16, device=dev)
        target.normal_(0.0, 3.0, generator=torch.Generator(device=dev).manual_seed(B * 17 + n))
        draft = torch.randint(0, V, (B, n), dtype=torch.int32, device=dev)
        vb = dels.dels_verify_workspace_bytes(B, n, V, code)
        vws = torch.zeros(vb, dtype=torch.uint8, device=dev)
        acc = torch.empty(B, dtype=torch.int32, device=dev)
        bonus = torch.empty(B, dtype=torch.int32, device=dev)

        def ver():
            r = dels.dels_verify_block(draft, target, code, B, n, V, acc, bonus, None, vws, vb)
            if r != 0:
                raise dels.DelsError(r, "dels_verify_block")

        t_v = timed(ver)
        v_bytes = B * (n + 1) * V * es
        del target
        if rank == 0:
            print(json.dumps({"sweep": "combine_verify", "V": V, "dtype": dt, "B": B, "n": n,
                              "combine": {"bytes": c_bytes, "us": round(t_c * 1e6, 2),
                                          "gbs": round(c_bytes / t_c / 1e9, 1),
                                          "frac": round(c_bytes / t_c / 1e9 / peak, 4)},
                              "verify": {"bytes": v_bytes, "us": round(t_v * 1e6, 2),
                                         "gbs": round(v_bytes / t_v / 1e9, 1),
                                         "frac": round(v_bytes / t_v / 1e9 / peak, 4)},
                              "peak_gbs": peak, "peak_source": peak_kind, "l2": "flushed before each launch"}),
                  flush=True)
    replicas.barrier()
    return 0


def run_sampled(args):
    """Drafted tokens per second at temperature 1 on the same workload as the
    default step: dels_draft_block_sampled (every position drawn by the
    Gumbel-max rule inside the vocabulary projection's pass) followed by
    dels_verify_block_sampled (acceptance tests, the rejected position's draft
    distribution rebuilt, the residual or p_n bonus draw). A fresh `step`
    every iteration, so every block draws new variates."""
    import torch
    import synth
    import paper_2607_07409_gb300 as dels
    from paper_2607_07409_gb300 import replicas
    world, rank, local = dist_setup(args.gpus)
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    peak, peak_kind = measured_peaks()
    w0 = synth.WORKLOADS[WORKLOAD]
    w = synth.with_sizes(w0, seed=replicas.replica_seed(w0.seed, rank))
    d = synth.make_inputs(w, device=dev)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = dels.dels_prior_from_counts(d["counts"]).to(dev)
    if not args.no_input_table:
        W["input_table"] = dels.gru_input_table(w.head, W, w.V)
    drafter = dels.Drafter(w.head, W, w.B, w.n, w.V)
    a = [w.alpha] * w.n
    b = [w.beta] * w.n
    head = drafter.head
    vbytes = dels.dels_verify_sampled_workspace_bytes(head, w.B, w.n, w.V, dels.DELS_BF16)
    vws = torch.zeros(vbytes, dtype=torch.uint8, device=dev)
    acc = torch.empty(w.B, dtype=torch.int32, device=dev)
    bonus = torch.empty(w.B, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()
    seed = 1234 + rank

    def draft(step):
        return drafter.sample(d["long"], prior, a, b, seed, step, stream)

    def verify(step, tok, lp, state):
        r = dels.dels_verify_block_sampled(head, tok, lp, state, d["long"], dels.DELS_BF16, prior, a, b, d["target"],
                                           dels.DELS_BF16, w.B, w.n, w.V, seed, step, acc, bonus, None, vws, vbytes,
                                           stream)
        if r != 0:
            raise dels.DelsError(r, "dels_verify_block_sampled")

    for i in range(max(3, args.warmup)):
        tok, lp, _, state = draft(i)
        verify(i, tok, lp, state)
    torch.cuda.synchronize()
    if drafter.status() != 0 or dels.dels_read_status(vws) != 0:
        raise RuntimeError("device status set during warm-up")
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(3)]
    replicas.barrier()
    torch.cuda.synchronize()
    t_draft = t_ver = 0.0
    lens = []
    with ClockSampler(local) as clk:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for i in range(args.steps):
            tok, lp, _, state = draft(1000 + i)
            verify(1000 + i, tok, lp, state)
        e1.record(stream)
        torch.cuda.synchronize()
    ms = replicas.max_over_ranks(e0.elapsed_time(e1) / args.steps)
    # the two halves, timed apart on a few more steps
    for i in range(min(args.steps, 20)):
        ev[0].record(stream)
        tok, lp, _, state = draft(5000 + i)
        ev[1].record(stream)
        verify(5000 + i, tok, lp, state)
        ev[2].record(stream)
        torch.cuda.synchronize()
        t_draft += ev[0].elapsed_time(ev[1])
        t_ver += ev[1].elapsed_time(ev[2])
        lens.append(acc.cpu().numpy().copy())
    k = min(args.steps, 20)
    # the sampled vocabulary kernel, event-timed by the library's profiler
    dels.dels_profile_reset()
    dels.dels_profile_enable(True)
    for i in range(3):
        draft(9000 + i)
    torch.cuda.synchronize()
    n_v, ms_v = dels.dels_profile_read(dels.KCLASS["vocab_combine"])
    dels.dels_profile_enable(False)
    us_v = 1e3 * ms_v / max(n_v, 1)
    vbytes_alg = algorithmic_vocab_bytes(w)
    import numpy as np
    tau = float(np.mean(np.concatenate(lens)) + 1.0)
    if rank == 0:
        print(json.dumps({
            "metric": "drafted tokens/sec at temperature 1 (Gumbel-max draft + speculative-sampling verify)",
            "value": world * w.B * w.n / (ms * 1e-3), "unit": "drafted tokens/s", "n_gpus": world,
            "steps": args.steps, "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True,
            "scaling": "weak", "vs_baseline": None, "dtype": "bf16 weights/logits, f32 accumulate", "data": "synthetic",
            "config": {"workload": f"{WORKLOAD} B={w.B} n={w.n} V={w.V} GRU 4096/1024/256, temperature 1",
                       "l2": "inputs larger than L2"},
            "draft_ms": t_draft / k, "verify_ms": t_ver / k, "tau": tau,
            "roofline": {"bound": "hbm", "kernel": "k_tc_gemm<sample> (vocab projection + Gumbel-max)",
                         "achieved": vbytes_alg / (us_v * 1e-6) / 1e9, "peak": peak, "unit": "GB/s",
                         "frac": vbytes_alg / (us_v * 1e-6) / 1e9 / peak, "peak_source": peak_kind,
                         "us_per_launch": us_v, "algorithmic_bytes_per_launch": vbytes_alg,
                         "traffic": ncu_traffic("vocab_sample_qwen3_8b_batched.md")},
            "clocks": clk.summary()}), flush=True)
    replicas.barrier()
    return 0


def run_wide(args):
    """The wide-projection row: every position projects a 4096-wide state
    (r = E[x_{j-1}], E [V, 4096]) onto the vocabulary through W [V, 4096]
    (1.24 GB bf16 streamed per position, no recurrence), fused with the
    combine; then the greedy verification. Same B, n, V and logits as the
    default step."""
    import torch
    import synth
    import paper_2607_07409_gb300 as dels
    from paper_2607_07409_gb300 import replicas
    world, rank, local = dist_setup(args.gpus)
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    peak, peak_kind = measured_peaks()
    w0 = synth.WORKLOADS[WORKLOAD]
    w = synth.Workload("qwen3_8b_wide", B=w0.B, n=w0.n, V=w0.V, logit_dtype=w0.logit_dtype,
                       head=synth.HeadSpec("markov", "bf16", 0, 0, 4096), weight=w0.weight,
                       seed=replicas.replica_seed(w0.seed, rank), zipf=w0.zipf, long_std=w0.long_std,
                       target_noise=w0.target_noise)
    d = synth.make_inputs(w, device=dev)
    W = {k[5:]: v for k, v in d.items() if k.startswith("head.")}
    prior = dels.dels_prior_from_counts(d["counts"]).to(dev)
    drafter = dels.Drafter(w.head, W, w.B, w.n, w.V)
    vbytes = dels.dels_verify_workspace_bytes(w.B, w.n, w.V, dels.DELS_BF16)
    vws = torch.zeros(vbytes, dtype=torch.uint8, device=dev)
    acc = torch.empty(w.B, dtype=torch.int32, device=dev)
    bonus = torch.empty(w.B, dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()

    def step():
        tok, lp, gap = drafter(d["long"], prior, w.alpha, w.beta, stream)
        r = dels.dels_verify_block(tok, d["target"], dels.DELS_BF16, w.B, w.n, w.V, acc, bonus, None, vws, vbytes,
                                   stream)
        if r != 0:
            raise dels.DelsError(r, "dels_verify_block")

    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()
    if drafter.status() != 0:
        raise RuntimeError("device status set during warm-up")
    steps = max(1, min(args.steps, 30))
    replicas.barrier()
    torch.cuda.synchronize()
    with ClockSampler(local) as clk:
        e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(steps):
            step()
        e1.record(stream)
        torch.cuda.synchronize()
    ms = replicas.max_over_ranks(e0.elapsed_time(e1) / steps)
    dels.dels_profile_reset()
    dels.dels_profile_enable(True)
    step()
    torch.cuda.synchronize()
    n_v, ms_v = dels.dels_profile_read(dels.KCLASS["vocab_combine"])
    dels.dels_profile_enable(False)
    us_v = 1e3 * ms_v / max(n_v, 1)
    R = w.head.d_rank
    vb = w.V * R * 2 + w.B * w.V * 2 + w.V * 4 + w.B * R * 2
    if rank == 0:
        print(json.dumps({
            "metric": "drafted tokens/sec, wide vocabulary projection (W [V, 4096] per position) + verify",
            "value": world * w.B * w.n / (ms * 1e-3), "unit": "drafted tokens/s", "n_gpus": world, "steps": steps,
            "warmup": args.warmup, "ms_per_step": ms, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
            "config": {"workload": f"B={w.B} n={w.n} V={w.V}, 4096-wide state, W [V, 4096] bf16",
                       "l2": "inputs larger than L2"},
            "roofline": {"bound": "hbm", "kernel": "k_tc_gemm<1> (K = 4096)", "achieved": vb / (us_v * 1e-6) / 1e9,
                         "peak": peak, "unit": "GB/s", "frac": vb / (us_v * 1e-6) / 1e9 / peak,
                         "peak_source": peak_kind, "us_per_launch": us_v, "algorithmic_bytes": vb},
            "clocks": clk.summary()}), flush=True)
    replicas.barrier()
    return 0


def run_prior(args):
    """Corpus positions per second of dels_prior_estimate (zero the counts,
    count the loss-masked ids, write l_P) over the 2^28-position synthetic
    corpus of synth.make_corpus (V = 151936). The corpus (1.34 GB) is larger
    than L2, so no flush is needed between steps. The count kernel is also
    timed alone (dels_prior_count, one launch) for the roofline: it reads
    4 bytes of id and 1 byte of mask per position."""
    import torch
    import numpy as np
    import synth
    import paper_2607_07409_gb300 as dels
    from paper_2607_07409_gb300 import replicas
    world, rank, local = dist_setup(args.gpus)
    dev = torch.device(f"cuda:{local}")
    torch.cuda.set_device(dev)
    peak, peak_kind = measured_peaks()
    w = synth.WORKLOADS[WORKLOAD]
    V, N = w.V, synth.CORPUS_TOKENS
    tok, mask = synth.make_corpus(V, N, replicas.replica_seed(w.seed, rank), device=dev)
    nbytes = dels.dels_prior_workspace_bytes(V, N)
    ws = torch.zeros(nbytes, dtype=torch.uint8, device=dev)
    out = torch.empty(V, dtype=torch.float32, device=dev)
    counts = torch.empty(V, dtype=torch.int64, device=dev)
    tally = torch.empty(2, dtype=torch.int64, device=dev)

    def estimate():
        r = dels.dels_prior_estimate(tok, mask, N, V, 1.0, out, counts, tally, ws, nbytes)
        if r != 0:
            raise dels.DelsError(r, "dels_prior_estimate")

    acc = torch.zeros(V, dtype=torch.int64, device=dev)

    def count_only():
        r = dels.dels_prior_count(tok, mask, N, V, acc, None, ws, nbytes)
        if r != 0:
            raise dels.DelsError(r, "dels_prior_count")

    def timed(fn, k):
        a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        torch.cuda.synchronize()
        a.record()
        for _ in range(k):
            fn()
        b.record()
        b.synchronize()
        return a.elapsed_time(b) * 1e-3 / k

    for _ in range(args.warmup):
        estimate()
        count_only()
    torch.cuda.synchronize()
    replicas.barrier()
    clk = ClockSampler(local)
    with clk:
        t_est = replicas.max_over_ranks(timed(estimate, args.steps))
        t_cnt = replicas.max_over_ranks(timed(count_only, args.steps))
    st = dels.dels_read_status(ws)
    c = counts.cpu().numpy()
    t = tally.cpu().numpy()
    masked = int(mask.sum(dtype=torch.int64).item())
    props = bool(st == 0 and t[0] == masked and t[1] == 0 and c.sum() == masked
                 and np.isclose(np.exp(out.double().cpu().numpy()).sum(), 1.0, atol=1e-5))
    # oracle on a bounded sample of the same corpus, on the host cores
    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        import oracle
        n_s = 1 << 25
        ts, ms = tok[:n_s].cpu().numpy(), mask[:n_s].cpu().numpy()
        t0 = time.perf_counter()
        c_s, _, _ = oracle.count_masked_tokens(ts, ms, V)
        oracle.log_prior(c_s)
        dt = time.perf_counter() - t0
        cpu = {"value": n_s / dt, "unit": "corpus positions/s", "cores": 1, "kind": "oracle",
               "sample": f"first {n_s} positions of the corpus (count + log prior)"}
    cnt_bytes = 5 * N
    if rank == 0:
        print(json.dumps({
            "metric": "unigram prior estimation: corpus positions/s (masked histogram + smoothing + log)",
            "value": world * N / t_est, "unit": "corpus positions/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": t_est * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "int32 ids, u8 mask, u64 counts, f64 log", "data": "synthetic",
            "config": {"workload": f"chat corpus N={N} V={V} Zipf(1.1) ids, ~75% loss-masked",
                       "l2": "inputs larger than L2"},
            "roofline": {"bound": "hbm", "kernel": "k_prior_count", "achieved": cnt_bytes / t_cnt / 1e9,
                         "peak": peak, "unit": "GB/s", "frac": cnt_bytes / t_cnt / 1e9 / peak,
                         "peak_source": peak_kind, "us_per_launch": t_cnt * 1e6, "algorithmic_bytes": cnt_bytes},
            "gpu_launches": 2 * args.steps + args.steps,
            "properties_ok": props, "clocks": clk.summary(), "cpu_baseline": cpu}), flush=True)
    replicas.barrier()
    return 0


def main():
    args = parse_args()
    if args.oracle_single_thread:
        return oracle_single_thread(args)
    if args.impl == "reference":
        return run_reference(args)
    if args.sweep:
        return run_sweep(args)
    if args.prior:
        return run_prior(args)
    if args.temperature == 1:
        return run_sampled(args)
    if args.variant == "wide":
        return run_wide(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
