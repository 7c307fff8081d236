"""Benchmark of the SpecFLASH verification step on GB300.

One step = one pass of the whole hot path over one batch: verification
attention for every layer of the workload (one sf_verify_attention call per
layer, separate KV caches) followed by the acceptance rule (sf_accept).
Default workload: the image-LMM 7B shape (B1, 32 layers, 32/32 heads, d128,
prefix 3008 = 5x576 visual + 128 text, k=5 drafts, V=32000, sampling at
tau=1): 1.58 GB of KV per step, far larger than the 129 MB L2, so every step
streams the caches from HBM.

Prints ONE JSON line (rank 0).  `value` is draft tokens verified per second
over the whole job; `e2e` repeats the measurement through host buffers
(pinned host -> device copies of the step's inputs and a device -> host read
of its results inside the timed region).  The step is captured once into
CUDA graphs (the C-ABI calls are asynchronous and allocation-free) and
replayed, as a serving loop would; `--eager` launches every call from Python
instead (then the host, not the GPU, sets the pace).

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME]
  python bench.py --impl reference ...   # the CPU oracle, same metric
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

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

METRIC = ("verify-step latency (µs) and KV-cache HBM GB/s vs GB300 peak; "
          "draft tokens verified/sec")
UNIT = "draft tokens/s"
NOMINAL_HBM_GBS = 8000.0


# --------------------------------------------------------------------------- #
# distributed plumbing (one process per GPU, launched by torchrun)            #
# --------------------------------------------------------------------------- #
def dist_env():
    rank = int(os.environ.get("RANK", "0"))
    world = int(os.environ.get("WORLD_SIZE", "1"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return rank, world, local


def init_dist(world: int, backend: str):
    import torch.distributed as dist
    if world > 1 and not dist.is_initialized():
        dist.init_process_group(backend=backend)
    return dist


def barrier(world: int):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int, device=None) -> float:
    """Largest value of x across ranks (the job is as slow as its slowest rank)."""
    if world <= 1:
        return float(x)
    import torch
    import torch.distributed as dist
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# --------------------------------------------------------------------------- #
# clocks during the timed region                                              #
# --------------------------------------------------------------------------- #
class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.proc = None
        self.path = None

    def start(self):
        try:
            fd, self.path = tempfile.mkstemp(suffix=".csv")
            os.close(fd)
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.gpu}", f"--query-gpu={self.QUERY}",
                 "--format=csv,noheader,nounits", "-lms", "200"],
                stdout=open(self.path, "w"), stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        rows = []
        with open(self.path) as f:
            for line in f:
                parts = [p.strip() for p in line.split(",")]
                if len(parts) >= 9:
                    rows.append(parts)
        os.unlink(self.path)
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["no samples"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        smax = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({names[i] for r in rows for i in range(4) if r[5 + i] == "Active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(smax) if smax else None, "reasons": reasons,
                "samples": len(rows)}


# --------------------------------------------------------------------------- #
# workload bookkeeping                                                        #
# --------------------------------------------------------------------------- #
def attention_bytes_per_layer(wl, seq_lens) -> int:
    """Algorithmic HBM bytes of one verification-attention launch: every
    visible K and V row once, Q in, O out (bf16), LSE out (fp32)."""
    kv = int(np.sum(seq_lens.astype(np.int64))) * wl.H_kv * wl.d * 2 * 2
    qo = wl.B * wl.rows * wl.H_q * wl.d * 2 * 2
    return kv + qo + wl.B * wl.rows * wl.H_q * 4


def accept_bytes(wl, mode_sampling_rows: int) -> int:
    """Algorithmic bytes of acceptance: all (k+1) logits rows once, plus row j
    of q for each sampled sequence's draw.  The draw's second read of row j
    of the logits (usually still in L2) is implementation overhead, reported
    separately (accept_reread_bytes)."""
    return wl.B * (wl.k + 1) * wl.V * 4 + mode_sampling_rows * wl.V * 4


# Sources whose code (comments and layout removed) a committed ncu summary
# was taken on, per attention kernel, and the summary of each workload.
KERNEL_SOURCES = {
    "verify_attention_kernel": ["paper_2505_12728_gb300/csrc/verify_attention.cu",
                                "paper_2505_12728_gb300/csrc/attn_common.cuh",
                                "paper_2505_12728_gb300/csrc/sf_device.cuh"],
    "verify_attention_tc_kernel": ["paper_2505_12728_gb300/csrc/verify_attention_tc.cu",
                                   "paper_2505_12728_gb300/csrc/attn_common.cuh",
                                   "paper_2505_12728_gb300/csrc/sf_device.cuh"],
    "lm_head_kernel": ["paper_2505_12728_gb300/csrc/draft_tail.cu",
                       "paper_2505_12728_gb300/csrc/ff_math.cuh",
                       "paper_2505_12728_gb300/csrc/sf_device.cuh"],
}
PROFILES = {"image7b": "profiles/verify_attention_image7b.md",
            "video": "profiles/verify_attention_tc_video.md"}
LM_HEAD_PROFILES = {"image7b": "profiles/lm_head_image7b.md",
                    "long": "profiles/lm_head_long.md"}


def attention_kernel(wl):
    """The kernel the library runs for a workload: the tcgen05 kernel when a
    KV head has more than 16 query rows, else the mma.sync kernel."""
    return "verify_attention_tc_kernel" if wl.rows * (wl.H_q // wl.H_kv) > 16 \
        else "verify_attention_kernel"


def tc_merge_partial_bytes(wl, seq_lens, sm_count):
    """Bytes of the tcgen05 kernel's split partials (fp32 O, max and sum per
    row of each key-split copy of each piece of a split segment, written once
    and read once by the merge kernel), from the partition rule the kernel applies on the device
    with one CTA per SM: the segment-aligned partition when its piece length
    is within 3 tiles of the balanced share, else the balanced one.  None for
    shapes of the mma.sync kernel (at most 16 rows per KV head), which merges
    through distributed shared memory or a last-CTA merge."""
    R = wl.rows * (wl.H_q // wl.H_kv)
    if R <= 16:
        return None
    tiles = [(int(t) + 63) // 64 for t in seq_lens]
    Tot = wl.H_kv * sum(tiles)
    G = min(Tot, sm_count)
    S = wl.B * wl.H_kv
    pieces = None
    if sm_count > S:
        Ta = -(-Tot // (sm_count - S))
        Tmin = -(-Tot // sm_count)
        if Ta <= Tmin + 3:
            for cand in range(Tmin, Ta):
                if wl.H_kv * sum(-(-t // cand) for t in tiles) <= sm_count:
                    Ta = cand
                    break
            pieces = [-(-t // Ta) for t in tiles for _ in range(wl.H_kv)]
    if pieces is None:
        q, r = divmod(Tot, G)
        start = lambda c: c * q + (c * r) // G
        def owner(t):
            lo, hi = 0, G - 1
            while lo < hi:
                mid = (lo + hi + 1) // 2
                if start(mid) <= t:
                    lo = mid
                else:
                    hi = mid - 1
            return lo
        pieces, base = [], 0
        for t in tiles:
            for h in range(wl.H_kv):
                first = base + h * t
                pieces.append(owner(first + t - 1) - owner(first) + 1)
            base += wl.H_kv * t
    # a split piece writes one partial per key-split copy of its rows
    copies = 4 if R <= 32 else (2 if R <= 64 else 1)
    per_piece = copies * (R * wl.d + 2 * R) * 4
    return 2 * per_piece * sum(n for n in pieces if n > 1)


def profiled_traffic(kernel_sources, profile):
    """DRAM bytes per launch from a committed ncu summary, or None when the
    kernel's sources changed since the counters were taken."""
    import hashlib
    import re
    try:
        h = hashlib.sha256()
        for f in kernel_sources:
            with open(os.path.join(ROOT, f)) as fh:
                code = fh.read()
            # the code only: comments and layout do not change the kernel
            code = re.sub(r"/\*.*?\*/", "", code, flags=re.S)
            code = re.sub(r"//[^\n]*", "", code)
            h.update("".join(code.split()).encode())
        with open(os.path.join(ROOT, profile)) as fh:
            text = fh.read()
    except OSError:
        return None
    fields = dict(line.split(":", 1) for line in text.splitlines()
                  if line.startswith(("kernel_source_sha256_16:", "traffic_bytes_per_launch:")))
    if fields.get("kernel_source_sha256_16", "").strip() != h.hexdigest()[:16]:
        return None
    try:
        return int(fields["traffic_bytes_per_launch"])
    except (KeyError, ValueError):
        return None


def measured_peaks():
    try:
        with open(os.path.join(ROOT, "MEASURED_PEAKS.json")) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return 6800.0, "fallback"


# --------------------------------------------------------------------------- #
# CPU oracle timing (the reported baseline; never the product path)           #
# --------------------------------------------------------------------------- #
def time_oracle_step_sample(wl, att, acc, layer: int):
    """Oracle time of one layer of attention and of the acceptance, in s."""
    from oracle import oracle
    t0 = time.perf_counter()
    oracle.verify_attention(att.q[layer], att.k_cache[layer], att.v_cache[layer],
                            att.block_table[layer], att.seq_lens, H_kv=att.H_kv)
    t1 = time.perf_counter()
    oracle.accept(acc.target_logits, acc.draft_probs, acc.draft_tokens, acc.uniforms,
                  acc.temperature)
    t2 = time.perf_counter()
    return t1 - t0, t2 - t1


def oracle_cores() -> int:
    n = os.environ.get("OMP_NUM_THREADS")
    return int(n) if n and n.isdigit() else (os.cpu_count() or 1)


def cpu_baseline(wl, att, acc, budget_s=12.0):
    from oracle import oracle
    oracle.build()
    layers_done, t_att, t_acc, n_acc = 0, 0.0, 0.0, 0
    start = time.perf_counter()
    while True:
        a, c = time_oracle_step_sample(wl, att, acc, layers_done % att.layers)
        t_att += a
        t_acc += c
        layers_done += 1
        n_acc += 1
        if time.perf_counter() - start > budget_s or layers_done >= att.layers:
            break
    step_s = wl.layers * (t_att / layers_done) + t_acc / n_acc
    # the same oracle on one thread: one attention layer and one acceptance
    oracle.set_threads(1)
    try:
        a1, c1 = time_oracle_step_sample(wl, att, acc, 0)
    finally:
        oracle.set_threads(0)
    step1_s = wl.layers * a1 + c1
    return {"value": wl.B * wl.k / step_s, "unit": UNIT, "cores": oracle_cores(),
            "kind": "oracle",
            "sample": f"fp64 C oracle on the host: {layers_done} of {wl.layers} attention layers "
                      f"and {n_acc} acceptance passes of the {wl.name} workload, scaled to one "
                      f"full step ({step_s * 1e3:.1f} ms)",
            "step_ms": step_s * 1e3,
            "value_1thread": wl.B * wl.k / step1_s, "step_ms_1thread": step1_s * 1e3,
            "cpu_model": cpu_model()}


def cpu_model() -> str:
    """The host CPU's name as /proc/cpuinfo gives it (model name on x86,
    implementer and part on Arm), with the machine type."""
    import platform
    fields = {}
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                if ":" in line:
                    k, v = line.split(":", 1)
                    fields.setdefault(k.strip(), v.strip())
    except OSError:
        pass
    name = fields.get("model name") or " ".join(
        f"{k} {fields[k]}" for k in ("CPU implementer", "CPU part") if k in fields)
    return f"{name or platform.processor() or 'unknown'} ({platform.machine()}, {os.cpu_count()} cores)"


def run_reference(args):
    rank, world, _ = dist_env()
    if rank != 0:
        return 0
    from paper_2505_12728_gb300.workloads import (make_accept_inputs, make_attention_inputs,
                                                  workload)
    from oracle import oracle
    oracle.build()
    wl = workload(args.workload, **({"layers": args.layers} if args.layers else {}))
    att = make_attention_inputs(wl, layers=min(wl.layers, 2))
    acc = make_accept_inputs(wl)

    def layer(l):
        # the inputs of two generated layers, used in turn (the oracle's time
        # does not depend on the values)
        oracle.verify_attention(att.q[l % att.layers], att.k_cache[l % att.layers],
                                att.v_cache[l % att.layers], att.block_table[l % att.layers],
                                att.seq_lens, H_kv=att.H_kv)

    def accept():
        oracle.accept(acc.target_logits, acc.draft_probs, acc.draft_tokens, acc.uniforms,
                      acc.temperature)

    # Each step is a bounded sample of the workload: as many of its layers as
    # let all W + K steps end within the wall-clock budget (all of them when
    # they fit), then the acceptance.  Layer and acceptance times are
    # measured apart, so that a sampled step's attention time can be scaled
    # to the workload's layer count.
    t = time.perf_counter()
    layer(0)
    t_layer = time.perf_counter() - t
    t = time.perf_counter()
    accept()
    t_acc = time.perf_counter() - t
    n_steps = args.warmup + args.steps
    per_step = args.reference_budget / n_steps
    n_layers = int(min(wl.layers, max(1, (per_step - t_acc) // max(t_layer, 1e-9))))

    def step():
        t = time.perf_counter()
        for l in range(n_layers):
            layer(l)
        t_att = time.perf_counter() - t
        accept()
        return t_att

    for _ in range(args.warmup):
        step()
    att_s = 0.0
    t0 = time.perf_counter()
    for _ in range(args.steps):
        att_s += step()
    step_s = (time.perf_counter() - t0) / args.steps
    att_step_s = att_s / args.steps
    # the workload's full step: the attention of all its layers (scaled from
    # the sampled ones when fewer ran) plus the measured acceptance
    full_step_s = att_step_s * wl.layers / n_layers + (step_s - att_step_s)
    value = wl.B * wl.k / full_step_s
    if n_layers == wl.layers:
        sample = (f"each step: the fp64 C oracle on all {wl.layers} attention layers plus the "
                  f"acceptance of the {wl.name} workload, measured (no extrapolation)")
    else:
        sample = (f"each step: the fp64 C oracle on {n_layers} of the {wl.name} workload's "
                  f"{wl.layers} attention layers plus its acceptance (so that {n_steps} steps "
                  f"fit {args.reference_budget:.0f} s); ms_per_step is that measured step, and "
                  f"value is draft tokens per full step with the attention time scaled by "
                  f"{wl.layers}/{n_layers}")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": UNIT,
            "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic",
            "config": workload_config(wl, att.seq_lens),
            "layers_per_step": n_layers,
            "ms_per_full_step": full_step_s * 1e3,
            "cpu_baseline": {"value": value, "unit": UNIT, "cores": oracle_cores(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": UNIT, "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def time_draft_tail(wl, dev, stream, capture):
    """Device time of sf_draft_sample (projection + sampling) and of
    sf_lm_head alone for the workload's B*k draft rows over a random bf16 LM
    head of the target's shape (V x hidden), each replayed from a CUDA graph
    of 10 calls; the weights (262 MB-1.09 GB) exceed L2, so every call
    streams them from HBM."""
    import torch
    from paper_2505_12728_gb300 import specflash_verify as sfv
    from paper_2505_12728_gb300.workloads import make_draft_tail_inputs
    case = make_draft_tail_inputs(wl)
    R, Hd, V = case.shape
    bf = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(
        torch.bfloat16)
    h, w = bf(case.hidden), bf(case.weight)
    u = torch.from_numpy(case.uniforms).to(dev)
    t = torch.from_numpy(case.temperature).to(dev)
    logits = torch.empty((R, V), dtype=torch.float32, device=dev)
    probs = torch.empty_like(logits)
    tokens = torch.empty(R, dtype=torch.int32, device=dev)
    ws = sfv.new_workspace(sfv.draft_tail_workspace_size(R, V), dev)
    fused = lambda: sfv.draft_sample(h, w, u, t, logits=logits, probs=probs, tokens=tokens,
                                     workspace=ws, stream=stream)
    proj = lambda: sfv.lm_head(h, w, logits=logits, workspace=ws, stream=stream)

    def per_call_us(fn, calls=10, reps=5):
        fn()
        g = capture(lambda: [fn() for _ in range(calls)])
        g.replay()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) * 1e3 / (calls * reps)

    fused_us = per_call_us(fused)
    proj_us = per_call_us(proj)
    status = sfv.read_device_status(ws)
    ok = bool(torch.isfinite(probs).all().item()) and \
        float((probs.double().sum(1) - 1).abs().max().item()) < 1e-5
    peak, kind = measured_peaks()
    alg = V * Hd * 2 + R * Hd * 2 + R * V * 4  # weights + hidden states + logits
    gbs = alg / (proj_us * 1e-6) / 1e9
    del w
    return {"rows": R, "hidden": Hd, "vocab": V, "draft_sample_us": fused_us,
            "lm_head_us": proj_us, "sampling_us": fused_us - proj_us,
            "lm_head_gbs": gbs, "lm_head_frac": gbs / peak,
            "lm_head_algorithmic_bytes": alg,
            "lm_head_traffic": (profiled_traffic(KERNEL_SOURCES["lm_head_kernel"],
                                                 LM_HEAD_PROFILES[wl.name])
                                if wl.name in LM_HEAD_PROFILES else None),
            "peak_gbs": peak, "peak_source": kind,
            "kernels": ["lm_head_kernel", "sample_finish_kernel"],
            "probs_sum_to_one": ok, "device_status": status}


def time_visual_compress(wl, dev, stream, capture):
    """Device time of sf_visual_compress (the draft model's Eq. 3 compressor)
    over the workload's frames, and of its score projection alone
    (sf_lm_head with the queries as rows and the features as the weight
    matrix), each replayed from a CUDA graph of 10 calls."""
    import torch
    from paper_2505_12728_gb300 import specflash_verify as sfv
    from paper_2505_12728_gb300.workloads import COMPRESS_SHAPES, make_compress_inputs
    if wl.name not in COMPRESS_SHAPES:
        return None
    F, N, C, d = COMPRESS_SHAPES[wl.name]
    qb, fb = make_compress_inputs(wl)
    bf = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(
        torch.bfloat16)
    q, f = bf(qb), bf(fb)
    out = torch.empty((F, C, d), dtype=torch.bfloat16, device=dev)
    ws = sfv.new_workspace(sfv.visual_compress_workspace_size(F, N, C, d), dev)
    scores = torch.empty((C, F * N), dtype=torch.float32, device=dev)
    ws2 = sfv.new_workspace(sfv.draft_tail_workspace_size(C, F * N), dev)
    full = lambda: sfv.visual_compress(q, f, out=out, workspace=ws, stream=stream)
    proj = lambda: sfv.lm_head(q, f.view(F * N, d), logits=scores, workspace=ws2, stream=stream)

    def per_call_us(fn, calls=10, reps=5):
        fn()
        g = capture(lambda: [fn() for _ in range(calls)])
        g.replay()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) * 1e3 / (calls * reps)

    full_us = per_call_us(full)
    proj_us = per_call_us(proj)
    peak, kind = measured_peaks()
    alg = F * N * d * 2 + C * d * 2 + F * C * d * 2  # features once, queries, output
    flops = 4.0 * F * C * N * d
    return {"frames": F, "tokens_per_frame": N, "queries": C, "hidden": d,
            "visual_compress_us": full_us, "scores_projection_us": proj_us,
            "gbs": alg / (full_us * 1e-6) / 1e9, "frac": alg / (full_us * 1e-6) / 1e9 / peak,
            "tflops": flops / (full_us * 1e-6) / 1e12, "algorithmic_bytes": alg,
            "peak_gbs": peak, "peak_source": kind,
            "kernels": ["lm_head_kernel", "compress_apply_kernel"],
            "device_status": sfv.read_device_status(ws)}


def time_fused_acceptance(wl, dev, stream, capture):
    """The target LM head of the B*(k+1) verified positions fused with the
    acceptance (sf_verify_lm_head_accept) against the two calls it replaces
    (sf_lm_head, then sf_accept on its logits), over a random bf16 LM head
    of the target's shape; graphs of 10 calls."""
    import torch
    from paper_2505_12728_gb300 import specflash_verify as sfv
    from paper_2505_12728_gb300.workloads import make_accept_inputs, make_draft_tail_case
    if wl.B * (wl.k + 1) > 256:
        return None
    from paper_2505_12728_gb300.workloads import HIDDEN_SIZES
    R, d, V = wl.B * (wl.k + 1), HIDDEN_SIZES[wl.V], wl.V
    case = make_draft_tail_case(R, d, V, seed=[wl.seed, 0xF05E], logit_std=wl.logit_std)
    acc = make_accept_inputs(wl)
    bf = lambda bits: torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(
        torch.bfloat16)
    h, w = bf(case.hidden).view(wl.B, wl.k + 1, d), bf(case.weight)
    q = torch.from_numpy(acc.draft_probs).to(dev)
    t = torch.from_numpy(acc.draft_tokens).to(dev)
    u = torch.from_numpy(acc.uniforms).to(dev)
    tau = torch.from_numpy(acc.temperature).to(dev)
    logits = torch.empty((wl.B, wl.k + 1, V), dtype=torch.float32, device=dev)
    n = torch.empty(wl.B, dtype=torch.int32, device=dev)
    toks = torch.empty((wl.B, wl.k + 1), dtype=torch.int32, device=dev)
    ratio = torch.empty((wl.B, wl.k), dtype=torch.float32, device=dev)
    ws_f = sfv.new_workspace(sfv.verify_lm_head_accept_workspace_size(wl.B, wl.k, V), dev)
    ws_l = sfv.new_workspace(sfv.draft_tail_workspace_size(R, V), dev)
    ws_a = sfv.new_workspace(sfv.accept_workspace_size(wl.B, wl.k, V), dev)
    fused = lambda: sfv.verify_lm_head_accept(h, w, q, t, u, tau, logits=logits, num_accepted=n,
                                              out_tokens=toks, accept_ratio=ratio, workspace=ws_f,
                                              stream=stream)

    def unfused():
        sfv.lm_head(h.view(R, d), w, logits=logits.view(R, V), workspace=ws_l, stream=stream)
        sfv.accept(logits, q, t, u, tau, num_accepted=n, out_tokens=toks, accept_ratio=ratio,
                   workspace=ws_a, stream=stream)

    def per_call_us(fn, calls=10, reps=5):
        fn()
        g = capture(lambda: [fn() for _ in range(calls)])
        g.replay()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(reps):
            g.replay()
        b.record(stream)
        torch.cuda.synchronize()
        return a.elapsed_time(b) * 1e3 / (calls * reps)

    fused_us = per_call_us(fused)
    n_f = n.clone()
    unfused_us = per_call_us(unfused)
    return {"rows": R, "hidden": d, "vocab": V, "fused_us": fused_us, "unfused_us": unfused_us,
            "same_num_accepted": bool(torch.equal(n_f, n)),
            "device_status": sfv.read_device_status(ws_f)}


def device_attention_layers(wl, n_layers, seed):
    """Verification-attention inputs of `n_layers` independent layers of a
    workload, built on the device for timing: sequence lengths follow the
    workload's prefix recipe (seeded numpy draw, as workloads.py draws them);
    every layer's page order in its pool is a seeded random permutation; Q, K
    and V are N(0, 1) from a seeded torch generator, rounded to bf16.  (Parity
    at these shapes is the GPU tests' job; here only the timing matters.)"""
    import torch
    from paper_2505_12728_gb300.workloads import prefix_lengths
    rng = np.random.default_rng([seed, 0xA77])
    seq_lens = (prefix_lengths(wl, rng) + wl.rows).astype(np.int32)
    pages = (seq_lens.astype(np.int64) + 15) // 16
    num_pages, max_pages = int(pages.sum()), int(pages.max())
    gen = torch.Generator(device="cuda").manual_seed(int(seed) * 7919 + 17)
    dev = torch.device("cuda", torch.cuda.current_device())
    layers = []
    for l in range(n_layers):
        perm = rng.permutation(num_pages).astype(np.int32)
        bt = np.full((wl.B, max_pages), -1, np.int32)
        off = 0
        for b in range(wl.B):
            bt[b, :pages[b]] = perm[off:off + pages[b]]
            off += int(pages[b])
        randn = lambda *shape: torch.randn(*shape, generator=gen, device=dev).to(torch.bfloat16)
        layers.append(dict(q=randn(wl.B, wl.rows, wl.H_q, wl.d),
                           k_cache=randn(num_pages, wl.H_kv, 16, wl.d),
                           v_cache=randn(num_pages, wl.H_kv, 16, wl.d),
                           block_table=torch.from_numpy(bt).to(dev)))
    return seq_lens, torch.from_numpy(seq_lens).to(dev), layers


def l2_bytes():
    import torch
    try:
        return int(torch.cuda.get_device_properties(torch.cuda.current_device()).L2_cache_size)
    except (AttributeError, RuntimeError):
        return 129 << 20


def time_workload(name, dev, stream, capture, peak, min_calls=200):
    """Attention and acceptance of one more workload, each replayed from a
    CUDA graph that rotates over enough distinct inputs (independent layers
    of KV; copies of the acceptance inputs) to exceed twice the L2, so every
    call streams from HBM, for at least min_calls calls after warm-up.
    Reports per-call device times (CUDA events on the launching stream: the
    mean, and p10 / median / p90 over the replays), algorithmic GB/s and the
    fractions of the measured copy bandwidth and of the nominal 8 TB/s."""
    import torch
    from paper_2505_12728_gb300 import specflash_verify as sfv
    from paper_2505_12728_gb300.workloads import make_accept_inputs, workload
    wl = workload(name)
    rng = np.random.default_rng([wl.seed, 0xA77])
    from paper_2505_12728_gb300.workloads import prefix_lengths
    lens0 = prefix_lengths(wl, rng) + wl.rows
    per_layer = attention_bytes_per_layer(wl, lens0)
    n_layers = max(2, -(-2 * l2_bytes() // per_layer))
    seq_np, sl, layers = device_attention_layers(wl, n_layers, wl.seed)
    bytes_layer = attention_bytes_per_layer(wl, seq_np)
    max_pages = layers[0]["block_table"].shape[1]
    ws = sfv.new_workspace(sfv.verify_attention_workspace_size(
        wl.B, wl.rows, wl.H_q, wl.H_kv, wl.d, max_pages), dev)
    outs = [torch.empty_like(x["q"]) for x in layers]
    lses = [torch.empty((wl.B, wl.rows, wl.H_q), dtype=torch.float32, device=dev) for _ in layers]

    def attn_all():
        for x, o, e in zip(layers, outs, lses):
            sfv.verify_attention(x["q"], x["k_cache"], x["v_cache"], x["block_table"], sl, out=o,
                                 lse=e, workspace=ws, stream=stream)

    def timed(fn, calls):
        """Mean per-call µs over the replays, and {p10, median, p90} of the
        per-replay means (an event between replays)."""
        fn()
        g = capture(fn)
        for _ in range(3):
            g.replay()
        reps = max(20, -(-min_calls // calls))
        ev = [torch.cuda.Event(enable_timing=True) for _ in range(reps + 1)]
        torch.cuda.synchronize()
        ev[0].record(stream)
        for i in range(reps):
            g.replay()
            ev[i + 1].record(stream)
        torch.cuda.synchronize()
        per = np.array([ev[i].elapsed_time(ev[i + 1]) * 1e3 / calls for i in range(reps)])
        dist = {"p10": float(np.percentile(per, 10)), "median": float(np.median(per)),
                "p90": float(np.percentile(per, 90)), "calls": calls * reps}
        return ev[0].elapsed_time(ev[reps]) * 1e3 / (calls * reps), dist

    att_us, att_dist = timed(attn_all, n_layers)
    att_status = sfv.read_device_status(ws)
    finite = all(bool(torch.isfinite(e).all().item()) for e in lses)
    del layers, outs
    # acceptance over rotating copies of the workload's inputs
    acc = make_accept_inputs(wl)
    base = [torch.from_numpy(a).to(dev) for a in (acc.target_logits, acc.draft_probs,
                                                 acc.draft_tokens, acc.uniforms, acc.temperature)]
    per_copy = base[0].numel() * 4 + base[1].numel() * 4
    n_copies = max(2, -(-2 * l2_bytes() // per_copy))
    copies = [base] + [[t.clone() for t in base] for _ in range(n_copies - 1)]
    ws_a = sfv.new_workspace(sfv.accept_workspace_size(wl.B, wl.k, wl.V), dev)
    n_acc = torch.empty(wl.B, dtype=torch.int32, device=dev)
    toks = torch.empty((wl.B, wl.k + 1), dtype=torch.int32, device=dev)
    ratio = torch.empty((wl.B, wl.k), dtype=torch.float32, device=dev)

    def acc_all():
        for c in copies:
            sfv.accept(*c, num_accepted=n_acc, out_tokens=toks, accept_ratio=ratio,
                       workspace=ws_a, stream=stream)

    acc_us, acc_dist = timed(acc_all, n_copies)
    sampling_rows = int(np.sum(acc.temperature > 0))
    acc_bytes = accept_bytes(wl, sampling_rows)
    # the data-dependent minimum: the logits rows 0..min(j, k) of each
    # sequence, and row j of q where a sampled sequence rejected draft j
    j = n_acc.cpu().numpy().astype(np.int64)
    sampled = acc.temperature > 0
    acc_min_bytes = int((np.minimum(j, wl.k) + 1).sum() * wl.V * 4
                        + np.sum(sampled & (j < wl.k)) * wl.V * 4)
    kv_gbs = bytes_layer / (att_us * 1e-6) / 1e9
    acc_gbs = acc_bytes / (acc_us * 1e-6) / 1e9
    return {"description": wl.description, "context_tokens": [int(x) for x in seq_np],
            "attention_kernel": attention_kernel(wl),
            "attention_launches_per_call": sfv.verify_attention_kernel_launches(
                wl.B, wl.rows, wl.H_q, wl.H_kv, wl.d, max_pages),
            "attention_us": att_us, "attention_us_distribution": att_dist,
            "attention_algorithmic_bytes": bytes_layer,
            "kv_gbs": kv_gbs, "frac": kv_gbs / peak, "frac_of_nominal_8tbs": kv_gbs / 8000.0,
            "layers_rotated": n_layers, "attention_finite": finite,
            "accept_kernels": (["accept_cluster_kernel"] if sfv.accept_kernel_launches(
                wl.B, wl.k, wl.V) == 1 else ["accept_chunks_kernel", "accept_draw_kernel"]),
            "accept_us": acc_us, "accept_us_distribution": acc_dist,
            "accept_algorithmic_bytes": acc_bytes, "accept_gbs": acc_gbs,
            "accept_reread_bytes": sampling_rows * wl.V * 4,
            "accept_min_bytes": acc_min_bytes, "accept_min_gbs": acc_min_bytes / (acc_us * 1e-6) / 1e9,
            "merge_partial_bytes": tc_merge_partial_bytes(
                wl, seq_np, torch.cuda.get_device_properties(dev).multi_processor_count),
            "accept_frac": acc_gbs / peak, "accept_frac_of_nominal_8tbs": acc_gbs / 8000.0,
            "accept_input_copies_rotated": n_copies,
            "mean_accepted": float(n_acc.float().mean().item()),
            "device_status": att_status | sfv.read_device_status(ws_a)}


def workload_config(wl, seq_lens):
    return {"workload": wl.name, "description": wl.description, "batch": wl.B,
            "layers": wl.layers, "H_q": wl.H_q, "H_kv": wl.H_kv, "head_dim": wl.d,
            "draft_k": wl.k, "query_rows": wl.rows, "vocab": wl.V,
            "prefix_tokens": [int(x) - wl.rows for x in seq_lens],
            "page_size": 16, "acceptance": wl.mode,
            "l2": "inputs larger than L2: every step streams "
                  f"{wl.layers} separate KV caches"}


# --------------------------------------------------------------------------- #
# the GPU path                                                                #
# --------------------------------------------------------------------------- #
def run_ours(args):
    import torch

    rank, world, local = dist_env()
    dist = init_dist(world, "nccl")
    torch.cuda.set_device(local)
    dev = torch.device("cuda", local)

    from paper_2505_12728_gb300 import build_lib
    from paper_2505_12728_gb300 import specflash_verify as sfv
    from paper_2505_12728_gb300.workloads import (make_accept_inputs, make_attention_inputs,
                                                  workload)
    build_lib.build()
    sfv.load_library()
    wl = workload(args.workload, **({"layers": args.layers} if args.layers else {}))
    att = make_attention_inputs(wl)
    acc = make_accept_inputs(wl)

    # CPU oracle baseline first (rank 0, N = 1 only), before any GPU work
    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(wl, att, acc, budget_s=args.cpu_budget)

    def bf16(bits):
        return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).to(dev).view(
            torch.bfloat16)

    L = att.layers
    q = bf16(att.q)                      # [L][B][n_q][H_q][d]
    kc = [bf16(att.k_cache[l]) for l in range(L)]
    vc = [bf16(att.v_cache[l]) for l in range(L)]
    bt = torch.from_numpy(att.block_table).to(dev)
    sl = torch.from_numpy(att.seq_lens).to(dev)
    logits = torch.from_numpy(acc.target_logits).to(dev)
    qprob = torch.from_numpy(acc.draft_probs).to(dev)
    toks = torch.from_numpy(acc.draft_tokens).to(dev)
    uni = torch.from_numpy(acc.uniforms).to(dev)
    temp = torch.from_numpy(acc.temperature).to(dev)
    out = torch.empty_like(q)
    lse = torch.empty((L, wl.B, wl.rows, wl.H_q), dtype=torch.float32, device=dev)
    n_acc = torch.empty(wl.B, dtype=torch.int32, device=dev)
    out_toks = torch.empty((wl.B, wl.k + 1), dtype=torch.int32, device=dev)
    ratio = torch.empty((wl.B, wl.k), dtype=torch.float32, device=dev)
    ws_att = sfv.new_workspace(sfv.verify_attention_workspace_size(
        wl.B, wl.rows, wl.H_q, wl.H_kv, wl.d, att.block_table.shape[2]), dev)
    ws_acc = sfv.new_workspace(sfv.accept_workspace_size(wl.B, wl.k, wl.V), dev)
    torch.cuda.synchronize()
    stream = torch.cuda.Stream()          # a non-default stream (graphs are captured on it)
    torch.cuda.set_stream(stream)

    def attention_layers(qsrc):
        for l in range(L):
            sfv.verify_attention(qsrc[l], kc[l], vc[l], bt[l], sl, out=out[l], lse=lse[l],
                                 workspace=ws_att, stream=stream)

    def acceptance(lg, qp, tk, un, tp):
        sfv.accept(lg, qp, tk, un, tp, num_accepted=n_acc, out_tokens=out_toks,
                   accept_ratio=ratio, workspace=ws_acc, stream=stream)

    def step():
        attention_layers(q)
        acceptance(logits, qprob, toks, uni, temp)

    for _ in range(args.warmup):
        step()
    torch.cuda.synchronize()

    # ---- eager timing (Python launches every call; host-bound, for reference) ----
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize()
    eager_ms = e0.elapsed_time(e1) / args.steps

    # ---- the step as CUDA graphs: all attention layers, then the acceptance ----
    def capture(fn):
        g = torch.cuda.CUDAGraph()
        with torch.cuda.graph(g, stream=stream):
            fn()
        return g

    use_graph = not args.eager
    if use_graph:
        # the step as one graph (the timed quantity), and its two parts as
        # separate graphs for the per-part breakdown
        g_step = capture(step)
        g_att = capture(lambda: attention_layers(q))
        g_acc = capture(lambda: acceptance(logits, qprob, toks, uni, temp))
        run_step, run_att, run_acc = g_step.replay, g_att.replay, g_acc.replay
    else:
        run_step = step
        run_att = lambda: attention_layers(q)
        run_acc = lambda: acceptance(logits, qprob, toks, uni, temp)
    # clocks are sampled from the warm-up through the end of the timed region
    clocks = ClockSampler(local)
    clocks.start()
    for _ in range(args.warmup):
        run_step()
    torch.cuda.synchronize()

    # ---- device-resident timing: K steps back to back ----
    barrier(world)
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record(stream)
    for _ in range(args.steps):
        run_step()
    t_end.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    clk = clocks.stop()
    total_ms = max_over_ranks(t_start.elapsed_time(t_end), world, dev)

    # ---- per-part breakdown (the two parts as separate launches, with
    # events between them; the part boundary costs a launch here) ----
    ev = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    for s in range(args.steps):
        ev[s][0].record(stream)
        run_att()
        ev[s][1].record(stream)
        run_acc()
        ev[s][2].record(stream)
    torch.cuda.synchronize()
    att_ms = [ev[s][0].elapsed_time(ev[s][1]) for s in range(args.steps)]
    acc_ms = [ev[s][1].elapsed_time(ev[s][2]) for s in range(args.steps)]

    # ---- per-step distribution: a second pass of the step, an event after
    # every step (the timed region above has none between steps) ----
    evs = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    evs[0].record(stream)
    for s in range(args.steps):
        run_step()
        evs[s + 1].record(stream)
    torch.cuda.synchronize()
    per_step = sorted(evs[s].elapsed_time(evs[s + 1]) * 1e3 for s in range(args.steps))
    pick = lambda fr: per_step[min(len(per_step) - 1, int(round(fr * (len(per_step) - 1))))]
    step_dist = {"p10": pick(0.1), "median": pick(0.5), "p90": pick(0.9), "unit": "us",
                 "steps": args.steps}
    ms_per_step = total_ms / args.steps
    tokens = wl.B * wl.k * world * args.steps
    value = tokens / (total_ms / 1e3)

    # ---- KV commit after acceptance (outside the step: it changes the cache
    # state).  Timed in a steady state on a copy of layer 0's table: a = 0
    # keeps one verified row and the next step verifies n_q - 1 rows, so every
    # length and page stays put; 100 commits replayed as one graph.
    commit_us = None
    if wl.rows >= 2:
        c_sl, c_bt = sl.clone(), bt[0].clone()
        c_fp = torch.zeros(16, dtype=torch.int32, device=dev)
        c_fc = torch.zeros(1, dtype=torch.int32, device=dev)
        c_acc = torch.zeros(wl.B, dtype=torch.int32, device=dev)
        c_ws = sfv.new_workspace(sfv.kv_commit_workspace_size(), dev)
        commit_once = lambda: sfv.kv_commit(c_sl, c_bt, c_fp, c_fc, c_acc, wl.rows, wl.rows - 1,
                                            workspace=c_ws, stream=stream)
        commit_once()
        g_com = capture(lambda: [commit_once() for _ in range(100)])
        g_com.replay()
        c0 = torch.cuda.Event(enable_timing=True)
        c1 = torch.cuda.Event(enable_timing=True)
        c0.record(stream)
        for _ in range(5):
            g_com.replay()
        c1.record(stream)
        torch.cuda.synchronize()
        commit_us = c0.elapsed_time(c1) * 1e3 / 500
        assert sfv.read_device_status(c_ws) == 0 and torch.equal(c_sl, sl)

    # ---- draft-distribution tail (the LM head, softmax and sampling of the
    # B*k draft rows that produce q and T'; outside the verification step)
    dt = time_draft_tail(wl, dev, stream, capture) if not args.no_draft_tail else None
    vcomp = time_visual_compress(wl, dev, stream, capture) if not args.no_draft_tail else None
    fused_acc = time_fused_acceptance(wl, dev, stream, capture) if not args.no_draft_tail else None
    # ---- the other workloads of the paper's image- and video-LMM settings,
    # attention and acceptance at their own shapes (>= 4K-token contexts:
    # video and long) ----
    peak_gbs = measured_peaks()[0]
    others = {}
    # the step's own workload first: its acceptance back to back over
    # rotating input copies (the in-step figure below carries a graph
    # launch at the part boundary)
    for name in [wl.name] + [w for w in args.also.split(",") if w and w != wl.name]:
        others[name] = time_workload(name, dev, stream, capture, peak_gbs)
        torch.cuda.empty_cache()

    # ---- end to end through host buffers: each step's inputs are packed in
    # one pinned staging buffer and copied to the device in one host-to-device
    # copy, and its results come back in one device-to-host copy.  The copy
    # of step s + 1's inputs runs on a side stream while step s computes (two
    # pinned and two device staging buffers, alternating), and each step
    # joins it at its end ----
    inputs = [att.q.view(np.int16), acc.target_logits, acc.draft_probs, acc.draft_tokens,
              acc.uniforms, acc.temperature]
    offs, total = [], 0
    for a in inputs:
        offs.append(total)
        total += (a.nbytes + 255) // 256 * 256
    h_stages = [torch.empty(total, dtype=torch.uint8).pin_memory() for _ in range(2)]
    for h_stage in h_stages:
        for a, o in zip(inputs, offs):
            h_stage[o:o + a.nbytes].copy_(torch.from_numpy(np.ascontiguousarray(a).view(np.uint8).reshape(-1)))
    d_stages = [torch.empty(total, dtype=torch.uint8, device=dev) for _ in range(2)]

    def staged(d_stage, i, dtype, shape):
        n = inputs[i].nbytes
        return d_stage[offs[i]:offs[i] + n].view(dtype).view(shape)

    views = [(staged(d, 0, torch.bfloat16, tuple(q.shape)), staged(d, 1, torch.float32, tuple(logits.shape)),
              staged(d, 2, torch.float32, tuple(qprob.shape)), staged(d, 3, torch.int32, tuple(toks.shape)),
              staged(d, 4, torch.float32, tuple(uni.shape)), staged(d, 5, torch.float32, tuple(temp.shape)))
             for d in d_stages]
    copy_stream = torch.cuda.Stream(device=dev)
    d_res = torch.empty(wl.B * (wl.k + 2), dtype=torch.int32, device=dev)
    e_n, e_out = d_res[:wl.B], d_res[wl.B:].view(wl.B, wl.k + 1)
    h_res = torch.empty(wl.B * (wl.k + 2), dtype=torch.int32).pin_memory()
    h_n, h_out = h_res[:wl.B], h_res[wl.B:].view(wl.B, wl.k + 1)
    h2d = h_stages[0].numel()  # one step's packed inputs (each padded to 256 bytes)
    d2h = h_res.numel() * 4

    def e2e_step(par):
        # this step's inputs are in d_stages[par]; the next step's are copied
        # into the other buffer (free once the previous step is done) meanwhile
        copy_stream.wait_stream(stream)
        with torch.cuda.stream(copy_stream):
            d_stages[1 - par].copy_(h_stages[1 - par], non_blocking=True)
        d_q, d_logits, d_qprob, d_toks, d_uni, d_temp = views[par]
        attention_layers(d_q)
        sfv.accept(d_logits, d_qprob, d_toks, d_uni, d_temp, num_accepted=e_n, out_tokens=e_out,
                   accept_ratio=ratio, workspace=ws_acc, stream=stream)
        h_res.copy_(d_res, non_blocking=True)
        stream.wait_stream(copy_stream)

    d_stages[0].copy_(h_stages[0], non_blocking=True)  # the first step's inputs
    for i in range(args.warmup):
        e2e_step(i % 2)
    torch.cuda.synchronize()
    if use_graph:
        g_par = [capture(lambda: e2e_step(0)), capture(lambda: e2e_step(1))]
        run_e2e = lambda i: g_par[i % 2].replay()
    else:
        run_e2e = e2e_step
    # the step counter continues across warm-up and the timed steps, so that
    # every step reads the buffer the previous one filled
    step_i = 0
    d_stages[0].copy_(h_stages[0], non_blocking=True)
    for _ in range(args.warmup):
        run_e2e(step_i % 2)
        step_i += 1
    torch.cuda.synchronize()
    barrier(world)
    e0.record(stream)
    for _ in range(args.steps):
        run_e2e(step_i % 2)
        step_i += 1
    e1.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    e2e_ms = max_over_ranks(e0.elapsed_time(e1), world, dev)
    e2e_value = tokens / (e2e_ms / 1e3)
    h_ok = bool(np.array_equal(h_n.numpy(), n_acc.cpu().numpy()))

    # ---- roofline of the dominant kernel (verification attention) ----
    peak, peak_kind = measured_peaks()
    bytes_layer = attention_bytes_per_layer(wl, att.seq_lens)
    att_launch_ms = sum(att_ms) / (args.steps * L)
    achieved = bytes_layer / (att_launch_ms / 1e3) / 1e9
    sampling_rows = int(np.sum(acc.temperature > 0))
    acc_launch_ms = sum(acc_ms) / args.steps
    status = sfv.read_device_status(ws_att) | sfv.read_device_status(ws_acc)

    kernel = attention_kernel(wl)
    line = {
        "metric": METRIC, "value": value, "unit": UNIT, "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_per_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": workload_config(wl, att.seq_lens),
        "verify_step_us": ms_per_step * 1e3,
        "verify_step_us_distribution": step_dist,
        "attention_us_per_layer": att_launch_ms * 1e3,
        "accept_us": others[wl.name]["accept_us"],
        "accept_us_in_step": acc_launch_ms * 1e3,
        "kv_gbs": achieved,
        "kv_frac_of_nominal_8tbs": achieved / NOMINAL_HBM_GBS,
        "accept_gbs": others[wl.name]["accept_gbs"],
        "accept_frac": others[wl.name]["accept_frac"],
        "kv_commit_us": commit_us,
        "draft_tail": dt,
        "visual_compress": vcomp,
        "lm_head_accept": fused_acc,
        "workloads": others,
        "mean_accepted": float(n_acc.float().mean().item()),
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak,
                     "traffic": (profiled_traffic(KERNEL_SOURCES[kernel], PROFILES[wl.name])
                                 if wl.name in PROFILES else None),
                     "algorithmic_bytes": bytes_layer,
                     "kernel": kernel,
                     "peak_source": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)"},
        "e2e": {"value": e2e_value, "unit": UNIT, "h2d_bytes_per_step": h2d,
                "d2h_bytes_per_step": d2h, "ms_per_step": e2e_ms / args.steps,
                "host_result_matches_device": h_ok},
        "launch": "cuda_graph" if use_graph else "eager",
        "eager_ms_per_step": eager_ms,
        # per step: each layer's attention launches, then the acceptance's, as
        # the library reports them for these shapes on this device
        "gpu_launches": args.steps * (
            L * sfv.verify_attention_kernel_launches(wl.B, wl.rows, wl.H_q, wl.H_kv, wl.d,
                                                     att.block_table.shape[2])
            + sfv.accept_kernel_launches(wl.B, wl.k, wl.V)),
        "clocks": clk,
        "device_status": status,
    }
    if cpu is not None:
        line["cpu_baseline"] = {k: cpu[k] for k in ("value", "unit", "cores", "kind", "sample",
                                                    "value_1thread", "cpu_model")}
    if rank == 0:
        print(json.dumps(line), flush=True)
    if world > 1:
        dist.destroy_process_group()
    return 0


def main(argv=None):
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=400)
    ap.add_argument("--warmup", type=int, default=50)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="image7b")
    ap.add_argument("--layers", type=int, default=0,
                    help="independent attention layers per step (default: the workload's)")
    ap.add_argument("--cpu-budget", type=float, default=12.0,
                    help="seconds of oracle work for the cpu_baseline sample")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--reference-budget", type=float, default=150.0,
                    help="--impl reference: wall-clock seconds for all warm-up and timed steps; "
                         "each step runs as many of the workload's layers as fit")
    ap.add_argument("--no-draft-tail", action="store_true",
                    help="skip the draft-side and LM-head timings (draft tail, visual compressor, "
                         "fused target LM head + acceptance)")
    ap.add_argument("--also", default="video,gqa,long",
                    help="comma-separated workloads whose attention and acceptance are timed "
                         "too (field `workloads`); empty for none")
    ap.add_argument("--eager", action="store_true",
                    help="launch every call from Python instead of replaying CUDA graphs")
    args = ap.parse_args(argv)
    args.warmup = max(3, args.warmup)   # at least 3 untimed warm-up steps
    if args.impl == "reference":
        return run_reference(args)
    return run_ours(args)


if __name__ == "__main__":
    sys.exit(main())
