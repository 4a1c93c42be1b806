"""Benchmark of the artifact-KV read path on GB300.

One step = one pass of the whole path over one batch: adapted Q projection
(LoRA, RMSNorm, RoPE) and attention over the assembled artifact blocks plus
the suffix KV (split-KV combine included).  Headline workload: the long
assembled context of the Qwen3-8B layer geometry (hidden 4096, 32/8 heads,
d 128, r 16; 64 artifacts of 2048 tokens = 131,072 cached keys plus a
2048-token suffix, batch 1), with the same kernel timed on full causal
attention over all 133,120 tokens beside it.  The Qwen3-4B prefill layer,
the Qwen3-8B layer with 4 requests and the 64-request decode step follow as
sub-objects of the same line, each with its own roofline.  Inputs are seeded
synthetic tensors of those shapes.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--workload NAME] [--no-configs]
  python bench.py --impl reference ...   # the fp64 CPU oracle, timed on host cores

Prints ONE JSON line (rank 0).  value = algorithmic attention FLOPs (or KV
bytes for the decode workload) per step / device time per step, with the
inputs resident in HBM; e2e = the same metric through the public API with
the step's inputs copied from pinned host memory and its output copied back.
The headline numbers are computed first; a later sub-object that fails
records {"error": ...} in the line and the run exits non-zero.
"""

from __future__ import annotations

import argparse
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

METRIC = "artifact-KV attention TFLOP/s (prefill) & KV GB/s (decode), % of roofline"
L2_FLUSH_BYTES = 512 << 20
HEADLINE = "qwen3_8b_long_131k"
SUB_CONFIGS = ("qwen3_4b_prefill", "qwen3_8b_prefill_4req", "qwen3_8b_decode_64req")


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return dict(hbm=d["hbm_gbs"], bf16=d["bf16_tflops"], bf16_sus=d["bf16_tflops_sustained"], src="measured")
    return dict(hbm=6800.0, bf16=1900.0, bf16_sus=1700.0, src="fallback")


# ---------------------------------------------------------------------------
# work accounting (algorithmic, per step)
# ---------------------------------------------------------------------------
def max_over_ranks(x: float, world: int, device="cpu") -> float:
    """The largest of every rank's value (the job is as slow as its slowest
    replica); the identity on one rank.  `device` is where the collective's
    buffer lives: the GPU under NCCL, the CPU under gloo."""
    if world <= 1:
        return x
    import torch
    t = torch.tensor([x], device=device, dtype=torch.float64)
    torch.distributed.all_reduce(t, op=torch.distributed.ReduceOp.MAX)
    return float(t.item())


def job_throughput(work_per_rank_step: float, world: int, steps: int, seconds: float) -> float:
    """Whole-job throughput: the work all ranks did over the slowest rank's time."""
    return work_per_rank_step * world * steps / seconds


def attention_flops(wl) -> float:
    """4 d Hq per visible (query, key) pair: 2d for q.k and 2d for p.v."""
    g = wl.geom
    pairs = 0
    for r in range(wl.n_req):
        t = wl.t_art(r)
        pairs += wl.S * t + wl.S * (wl.S_kv - wl.S) + wl.S * (wl.S + 1) // 2
    return 4.0 * g.head_dim * g.n_q_heads * pairs


def qproj_flops(wl) -> float:
    g = wl.geom
    M = wl.n_req * wl.S
    return 2.0 * M * g.hidden * g.d_q + 2.0 * M * g.hidden * g.rank + 2.0 * M * g.rank * g.d_q


def kv_bytes(wl) -> float:
    """Each request reads its assembled K and V once: (T_art + S_kv) * 2 * Hkv * d * 2 bytes."""
    g = wl.geom
    return float(sum((wl.t_art(r) + wl.S_kv) * 2 * g.n_kv_heads * g.head_dim * 2 for r in range(wl.n_req)))


def kv_distinct_bytes(wl) -> float:
    """The distinct K/V a step needs: every artifact the requests use, once, and
    every request's own suffix rows.  Requests that share an artifact need its
    bytes once, so a kernel that reads shared blocks once (or from L2) moves
    fewer DRAM bytes than kv_bytes counts."""
    g = wl.geom
    used = {a for r in wl.requests for a in r}
    tokens = sum(wl.art_lengths[a] for a in used) + wl.n_req * wl.S_kv
    return float(tokens * 2 * g.n_kv_heads * g.head_dim * 2)


def is_decode(wl) -> bool:
    return wl.S * wl.geom.group <= 16


# ---------------------------------------------------------------------------
# clocks sampled during the timed region
# ---------------------------------------------------------------------------
class ClockSampler:
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, device_index: int):
        self.proc = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits", "-lms", "200",
                 "-i", str(device_index)], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        return parse_clocks(out)


def parse_clocks(out: str):
    """Median SM clock under load, the largest max clock and every throttle
    reason seen in `nvidia-smi --query-gpu=<ClockSampler.FIELDS>` CSV lines
    (noheader, nounits); None without a readable sample."""
    sm, mx, reasons = [], [], set()
    names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
    for line in out.strip().splitlines():
        parts = [p.strip() for p in line.split(",")]
        if len(parts) < 9:
            continue
        try:
            sm.append(float(parts[1]))
            mx.append(float(parts[2]))
        except ValueError:
            continue
        for n, v in zip(names, parts[5:9]):
            if v.lower().startswith("active"):
                reasons.add(n)
    if not sm:
        return None
    load = [s for s in sm if s > 0.5 * max(sm)] or sm
    return {"sm_mhz": statistics.median(load), "sm_max_mhz": max(mx), "reasons": sorted(reasons),
            "samples": len(sm)}


# ---------------------------------------------------------------------------
# the oracle timed on host cores (cpu_baseline and the reference arm)
# ---------------------------------------------------------------------------
def _oracle_inputs(wl, req):
    import oracle
    f = oracle.bf16_to_f64
    g = wl.geom
    ids = wl.requests[req]
    return dict(x=f(wl.x[req]), w_q=f(wl.w_q), a=None if wl.lora_a is None else f(wl.lora_a),
                b=None if wl.lora_b is None else f(wl.lora_b), s=g.scale, q_norm_w=f(wl.q_norm_w),
                eps=g.rms_eps, theta=g.rope_theta, art_k=[f(wl.art_k[i]) for i in ids],
                art_v=[f(wl.art_v[i]) for i in ids], suffix_k=f(wl.suffix_k[req]),
                suffix_v=f(wl.suffix_v[req]), n_q_heads=g.n_q_heads)


def oracle_sample(wl, inputs, tokens, decode: bool):
    """Run the oracle on every head of the given suffix tokens of request 0.
    Returns (seconds, work) with work in FLOPs (prefill) or bytes (decode)."""
    import oracle
    g = wl.geom
    pairs = [(i, h) for i in tokens for h in range(g.n_q_heads)]
    t0 = time.perf_counter()
    oracle.request_forward(**inputs, pairs=pairs)
    dt = time.perf_counter() - t0
    t_art = wl.t_art(0)
    vis = sum(t_art + (wl.S_kv - wl.S) + i + 1 for i in tokens)
    if decode:
        # every KV head's keys and values of the request are read once per token
        work = float(vis * 2 * g.n_kv_heads * g.head_dim * 2)
    else:
        work = 4.0 * g.head_dim * g.n_q_heads * vis
    return dt, work


def host_threads_env():
    """Let the oracle's BLAS use every host core: set before numpy loads."""
    n = str(os.cpu_count() or 1)
    for k in ("OMP_NUM_THREADS", "OPENBLAS_NUM_THREADS", "MKL_NUM_THREADS", "BLIS_NUM_THREADS"):
        os.environ[k] = n


def blas_threads() -> int:
    """Threads numpy's BLAS actually runs with (read from the loaded library),
    else the thread count the environment asked for."""
    try:
        import threadpoolctl
        info = [d for d in threadpoolctl.threadpool_info() if d.get("user_api") == "blas"]
        if info:
            return int(info[0]["num_threads"])
    except Exception:
        pass
    try:
        import ctypes
        with open("/proc/self/maps") as f:
            libs = sorted({ln.split()[-1] for ln in f
                           if "openblas" in ln.split()[-1].lower() and ".so" in ln.split()[-1]})
        for path in libs:
            lib = ctypes.CDLL(path)
            for sym in ("scipy_openblas_get_num_threads64_", "openblas_get_num_threads64_",
                        "openblas_get_num_threads"):
                fn = getattr(lib, sym, None)
                if fn is not None:
                    fn.restype = ctypes.c_int
                    return int(fn())
    except Exception:
        pass
    return int(os.environ.get("OPENBLAS_NUM_THREADS", "1"))


def cpu_baseline(wl, budget_s: float = 12.0, seed: int = 0):
    """The oracle on a bounded sample of request 0's suffix tokens (all q
    heads), multithreaded BLAS on every host core; the metric is the sample's
    work over its time, and the full step is extrapolated linearly by work."""
    import numpy as np
    decode = is_decode(wl)
    inputs = _oracle_inputs(wl, 0)
    rng = np.random.default_rng(seed)
    tokens_all = list(range(wl.S))
    done_t, done_w, n_tok = 0.0, 0.0, 0
    chunk = max(1, min(8, wl.S))
    while done_t < budget_s and n_tok < wl.S:
        toks = sorted(rng.choice(tokens_all, size=min(chunk, wl.S), replace=False).tolist())
        dt, w = oracle_sample(wl, inputs, toks, decode)
        done_t += dt
        done_w += w
        n_tok += len(toks)
    scale = 1e9 if decode else 1e12
    full = kv_bytes(wl) if decode else attention_flops(wl)
    threads = blas_threads()
    return {"value": done_w / done_t / scale, "unit": "GB/s" if decode else "TFLOP/s",
            "cores": threads, "host_cpus": os.cpu_count(), "kind": "oracle",
            "sample": f"request 0, {n_tok} random suffix tokens x all {wl.geom.n_q_heads} q heads of "
                      f"{wl.n_req * wl.S} query tokens (fp64 numpy oracle, BLAS on {threads} threads), "
                      f"{done_t:.1f} s of CPU work; the full step ({full / scale:.4g} "
                      f"{'GB' if decode else 'TFLOP'}) extrapolated linearly by work: "
                      f"{full * done_t / done_w:.4g} s"}


# ---------------------------------------------------------------------------
# our arm
# ---------------------------------------------------------------------------
class Bed:
    """One workload loaded into a library context: registered artifacts, the
    assembled plan and the step's output buffers, all resident on the GPU."""

    def __init__(self, name, dev, local_rank):
        import torch
        import paper_2609_36722_gb300 as pkg
        from gen import make_workload
        self.name = name
        self.dev = dev
        self.wl = wl = make_workload(name, device=dev)
        self.g = g = wl.geom
        self.decode = is_decode(wl)
        self.ctx = pkg.Context.for_geometry(g, pool_blocks=sum(-(-L // 64) for L in wl.art_lengths) + 1,
                                            device=local_rank)
        for k, v in zip(wl.art_k, wl.art_v):
            self.ctx.register_artifact(k, v)
        self.plan = self.ctx.assemble(wl.requests)
        self.out = torch.empty(wl.n_req, wl.S, g.n_q_heads, g.head_dim, dtype=torch.bfloat16, device=dev)
        self.lse = torch.empty(wl.n_req, wl.S, g.n_q_heads, dtype=torch.float32, device=dev)
        self.q = torch.empty_like(self.out)
        self.work = kv_bytes(wl) if self.decode else attention_flops(wl)
        self.scale = 1e9 if self.decode else 1e12
        self.unit = "GB/s" if self.decode else "TFLOP/s"

    def close(self):
        import torch
        self.plan.free()
        self.ctx.close()
        del self.wl, self.out, self.lse, self.q
        torch.cuda.empty_cache()


class Timer:
    """Times callables on the device.  By default the calls are captured once
    into a CUDA graph and every timed run replays it, with events recorded as
    nodes inside the graph; with eager=True (for profilers, which step through
    graph replays very slowly) the same calls are launched directly."""

    def __init__(self, eager, flush):
        self.eager = eager
        self.flush = flush

    def event(self):
        import torch
        # an event that a captured graph records as a node of its own
        return torch.cuda.Event(enable_timing=True, external=not self.eager)

    def graphed(self, fn):
        import torch
        e0, e1 = self.event(), self.event()
        if self.eager:
            class Eager:
                def replay(_):
                    e0.record()
                    fn()
                    e1.record()
            return Eager(), e0, e1
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr):
            e0.record()
            fn()
            e1.record()
        torch.cuda.synchronize()
        return gr, e0, e1

    def time(self, fn, steps):
        """ms of each of `steps` runs of fn, L2 flushed before each (outside the events)."""
        gr, e0, e1 = self.graphed(fn)
        ms = []
        for _ in range(steps):
            self.flush.zero_()
            gr.replay()
            e1.synchronize()
            ms.append(e0.elapsed_time(e1))
        return ms


def measure_core(bed, args, world, timer, with_clocks=False, local_rank=0):
    """Device-resident timing of one workload: the step (Q projection +
    attention) for the value, and the same step with events around the
    attention call for the roofline."""
    import torch
    wl, g, ctx, plan = bed.wl, bed.g, bed.ctx, bed.plan
    ev_q, ev_a, ev_b = timer.event(), timer.event(), timer.event()

    def step(attn_events=False):
        # attn_events: bracket the attention call with events (for the roofline).
        # An event recorded between the two calls keeps the attention kernel
        # from starting while the projection finishes (programmatic dependent
        # launch needs kernel after kernel), so the step timing runs without.
        if attn_events:
            ev_q.record()
        ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=wl.S_kv, out=bed.q)
        n1 = ctx.last_launch_count()
        if attn_events:
            ev_a.record()
        ctx.attend(plan, bed.q, wl.suffix_k, wl.suffix_v, out=bed.out, lse=bed.lse)
        if attn_events:
            ev_b.record()
        return n1 + ctx.last_launch_count()

    launches_per_step = 0
    for _ in range(args.warmup):
        launches_per_step = step()
    torch.cuda.synchronize()
    if ctx.sync_status() != 0:
        raise RuntimeError(f"{bed.name}: device status after the warm-up steps")
    g_step, ev_s, ev_e = timer.graphed(step)
    g_parts, _, _ = timer.graphed(lambda: step(attn_events=True))
    sampler = ClockSampler(local_rank) if with_clocks else None
    # keep the GPU busy ~1 s before timing so the clock samples describe the timed region
    t_end = time.perf_counter() + (1.0 if with_clocks else 0.0)
    while time.perf_counter() < t_end:
        g_step.replay()
        torch.cuda.synchronize()
    if world > 1:
        torch.distributed.barrier()
    torch.cuda.synchronize()
    step_ms = []
    for _ in range(args.steps):
        timer.flush.zero_()                                   # L2 flush between steps, outside the events
        g_step.replay()
        ev_e.synchronize()
        step_ms.append(ev_s.elapsed_time(ev_e))
    torch.cuda.synchronize()
    total_ms = max_over_ranks(sum(step_ms), world, bed.dev)
    clocks = sampler.stop() if sampler else None
    # the same steps again with events around the attention call: its launch
    # duration for the roofline
    attn_ms, qproj_ms = [], []
    for _ in range(args.steps):
        timer.flush.zero_()
        g_parts.replay()
        ev_b.synchronize()
        attn_ms.append(ev_a.elapsed_time(ev_b))
        qproj_ms.append(ev_q.elapsed_time(ev_a))
    torch.cuda.synchronize()
    st = ctx.sync_status()
    if st != 0:
        raise RuntimeError(f"{bed.name}: device status {st} after the timed region")
    del g_step, g_parts
    peaks = _peaks()
    attn_avg = statistics.mean(attn_ms)
    achieved = bed.work / (attn_avg * 1e-3) / bed.scale
    peak = peaks["hbm"] if bed.decode else peaks["bf16"]
    qp_avg = statistics.mean(qproj_ms)
    qp_tf = qproj_flops(wl) / (qp_avg * 1e-3) / 1e12
    # the Q projection's own bound: its FLOPs at the bf16 peak, or its
    # operand bytes (x, W_q, A, B, q_norm weight, Q out) at the copy bandwidth
    qp_bytes = 2.0 * (wl.n_req * wl.S * g.hidden + g.d_q * g.hidden + g.rank * g.hidden + g.d_q * g.rank + g.head_dim
                      + wl.n_req * wl.S * g.d_q)
    qp_bound_ms = max(qproj_flops(wl) / (peaks["bf16"] * 1e12), qp_bytes / (peaks["hbm"] * 1e9)) * 1e3
    return {
        "value": round(job_throughput(bed.work, world, args.steps, total_ms * 1e-3) / bed.scale, 3),
        "unit": bed.unit,
        "ms_per_step": round(total_ms / args.steps, 5),
        "roofline": {"bound": "hbm" if bed.decode else "tensor", "achieved": round(achieved, 3), "peak": peak,
                     "unit": bed.unit, "frac": round(achieved / peak, 4), "traffic": load_traffic(bed.name),
                     "kernel": ("attn_mma_kernel (split-KV chunks merged inside it)" if bed.decode
                                else "attn_tc_kernel (split-KV chunks merged inside it)"),
                     "work_per_launch": bed.work,
                     "work_unit": "bytes (each request's assembled K and V read once)" if bed.decode
                                  else "FLOP (4 d Hq per visible query-key pair)",
                     "peak_source": f"{peaks['src']} ({'hbm_gbs' if bed.decode else 'bf16_tflops burst'})",
                     "avg_launch_ms": round(attn_avg, 5),
                     **(decode_read_fracs(wl, attn_avg, peak, load_traffic(bed.name)) if bed.decode else {})},
        "qproj": {"avg_call_ms": round(qp_avg, 5), "tflops": round(qp_tf, 3),
                  "frac_of_bf16_peak": round(qp_tf / peaks["bf16"], 4),
                  "bound_ms": round(qp_bound_ms, 5), "frac_of_bound": round(qp_bound_ms / qp_avg, 4)},
        "path_work": {"attention_flops": attention_flops(wl), "qproj_flops": qproj_flops(wl),
                      "kv_bytes": kv_bytes(wl)},
        "gpu_launches": launches_per_step * args.steps,
        "clocks": clocks,
        "workload": {"hidden": g.hidden, "n_q_heads": g.n_q_heads, "n_kv_heads": g.n_kv_heads,
                     "head_dim": g.head_dim, "lora_rank": g.rank, "s": g.scale, "n_req": wl.n_req, "S": wl.S,
                     "S_kv": wl.S_kv, "t_art": [wl.t_art(r) for r in range(wl.n_req)][:8],
                     "artifacts_per_req": [len(r) for r in wl.requests][:8]},
    }


class HostInputs:
    """A step's inputs and output in pinned host memory, and the device suffix
    K/V buffers they update: the new tokens' hidden states and their own
    suffix K/V rows (the last S of each request's S_kv rows).  A decode step's
    earlier suffix rows are the request's resident cache, written by earlier
    steps: they stay on the device, as the artifact pool does."""

    def __init__(self, bed):
        import torch
        wl = bed.wl
        self.S_old = S_old = wl.S_kv - wl.S
        self.x_h = wl.x.cpu().pin_memory()
        self.sk_h = wl.suffix_k[:, S_old:].cpu().contiguous().pin_memory()
        self.sv_h = wl.suffix_v[:, S_old:].cpu().contiguous().pin_memory()
        self.out_h = torch.empty(bed.out.shape, dtype=bed.out.dtype, pin_memory=True)
        self.x_d = torch.empty_like(wl.x)
        self.sk_d = wl.suffix_k.clone()
        self.sv_d = wl.suffix_v.clone()
        self.h2d_bytes = (self.x_h.numel() + self.sk_h.numel() + self.sv_h.numel()) * 2
        self.d2h_bytes = self.out_h.numel() * 2

    def copy_in(self):
        """The inputs' H2D copies as separate calls (the warm-cache step, whose
        Q projection runs apart from the attention)."""
        self.x_d.copy_(self.x_h, non_blocking=True)
        self.sk_d[:, self.S_old:].copy_(self.sk_h, non_blocking=True)
        self.sv_d[:, self.S_old:].copy_(self.sv_h, non_blocking=True)


L2_BYTES = 129 << 20
E2E_DEPTH = 3   # steps in flight in the end-to-end loop


def working_set_bytes(bed) -> int:
    """Bytes a step reads: the registered artifacts' K/V, the weights, the inputs."""
    wl, g = bed.wl, bed.g
    pool = sum(wl.art_lengths) * 2 * g.n_kv_heads * g.head_dim * 2
    weights = (g.d_q * g.hidden + g.rank * g.hidden + g.d_q * g.rank) * 2
    inputs = (wl.x.numel() + wl.suffix_k.numel() + wl.suffix_v.numel()) * 2
    return pool + weights + inputs


def measure_e2e(bed, args, world, flush, local_rank=0):
    """The same metric through the public API with host buffers, as a serving
    loop.  Every step assembles its plan (attuner_assemble) and makes one
    attuner_query_attend_host call, which copies the step's new inputs from
    pinned host memory (the new tokens' hidden states and their own suffix K/V
    rows; a decode step's earlier suffix rows are the request's resident cache,
    like the artifact pool), runs the projection and the attention, and copies
    O back to pinned host memory, all on the step's stream; a step counts as
    done once its output is on the host.  Steps i+1 and i+2 are assembled and
    enqueued, on other streams, while step i runs (three sets of buffers per
    context), so host work and copies overlap device work as in a server.  No flush runs
    inside the loop: a workload whose working set fits in L2 alternates between
    enough identical, separately loaded contexts that every step reads data the
    others have evicted."""
    import torch
    n_sets = max(1, -(-2 * L2_BYTES // working_set_bytes(bed)))
    beds = [bed] + [Bed(bed.name, bed.dev, local_rank) for _ in range(n_sets - 1)]
    try:
        # (bed, host buffers and device suffix K/V, stream, output-on-host event)
        # interleaved, so that consecutive steps use different contexts
        units = []
        for _ in range(E2E_DEPTH):
            for b in beds:
                units.append((b, HostInputs(b), torch.cuda.Stream(device=bed.dev), torch.cuda.Event()))
        n_units = len(units)

        def enqueue(i, plan):
            # each unit's buffers are reused only after the step that last used
            # them was waited for (E2E_DEPTH steps in flight at most)
            b, io, stream, done = units[i % n_units]
            wl, g = b.wl, b.g
            b.ctx.query_attend_host(plan, io.x_h, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, io.sk_d,
                                    io.sv_d, io.sk_h, io.sv_h, out_host=io.out_h, stream=stream)
            done.record(stream)

        def assemble(i):
            b = units[i % n_units][0]
            return b.ctx.assemble(b.wl.requests)

        def run(n):
            plans = {}
            for i in range(min(E2E_DEPTH - 1, n)):
                plans[i] = assemble(i)
                enqueue(i, plans[i])
            for i in range(n):
                nxt = i + E2E_DEPTH - 1
                if nxt < n:
                    plans[nxt] = assemble(nxt)         # a later step, while step i runs
                    enqueue(nxt, plans[nxt])
                units[i % n_units][3].synchronize()    # step i's output is on the host
                plans.pop(i).free()

        run(max(3, args.warmup))
        flush.zero_()
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        run(args.steps)
        e2e_s = max_over_ranks(time.perf_counter() - t0, world, bed.dev)
        for b in beds:
            if b.ctx.sync_status() != 0:
                raise RuntimeError(f"{bed.name}: device status after the end-to-end steps")
        io = units[0][1]
        return {"value": round(job_throughput(bed.work, world, args.steps, e2e_s) / bed.scale, 3), "unit": bed.unit,
                "h2d_bytes_per_step": io.h2d_bytes, "d2h_bytes_per_step": io.d2h_bytes,
                "ms_per_step": round(e2e_s * 1e3 / args.steps, 4),
                "l2": (f"no flush in the loop; {n_sets} separately loaded contexts alternate so each step's "
                       f"{working_set_bytes(bed) / 1e6:.0f} MB working set is evicted before its next use"
                       if n_sets > 1 else f"no flush in the loop; the {working_set_bytes(bed) / 1e6:.0f} MB working "
                                          "set of a step exceeds L2"),
                "includes": "per step: assemble (host block table + upload) and one attuner_query_attend_host call "
                            "(H2D of the step's new tokens - x and their own suffix K/V rows; a decode step's earlier "
                            "suffix rows stay resident - the Q projection, the attention and the D2H of O, on the "
                            "step's stream) and a wait for the output; steps i+1 and i+2 assembled and enqueued on "
                            "other streams while step i runs"}
    finally:
        for b in beds[1:]:
            b.close()


def measure_full_causal(bed, reps=5):
    """The 131k-key layer's analogue of the paper's reuse-vs-full-prefill
    speedup: the same attention kernel on full causal attention over the
    whole assembled sequence (an empty plan: every token a query), i.e. the
    prefill the cached artifacts avoid."""
    import torch
    wl, g, ctx = bed.wl, bed.g, bed.ctx
    n_full = wl.t_art(0) + wl.S_kv
    gen = torch.Generator(device=bed.dev).manual_seed(4)
    qf = torch.randn(1, n_full, g.n_q_heads, g.head_dim, device=bed.dev, dtype=torch.bfloat16, generator=gen)
    kf = torch.randn(1, n_full, g.n_kv_heads, g.head_dim, device=bed.dev, dtype=torch.bfloat16, generator=gen)
    vf = torch.randn(1, n_full, g.n_kv_heads, g.head_dim, device=bed.dev, dtype=torch.bfloat16, generator=gen)
    of = torch.empty_like(qf)
    fplan = ctx.assemble([[]])
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    ms = []
    for i in range(reps):
        e0.record()
        ctx.attend(fplan, qf, kf, vf, out=of, want_lse=False)
        e1.record()
        e1.synchronize()
        if i >= 2:
            ms.append(e0.elapsed_time(e1))
    fplan.free()
    if ctx.sync_status() != 0:
        raise RuntimeError("device status after the full causal analogue")
    flops = 4.0 * g.head_dim * g.n_q_heads * n_full * (n_full + 1) / 2
    return n_full, statistics.mean(ms), flops


def measure_kv_project(bed, args, timer):
    """The suffix tokens' K/V projection: same x, base k_proj / v_proj weights
    of the geometry, into scratch suffix buffers."""
    from gen import make_kv_weights
    wl, g, ctx = bed.wl, bed.g, bed.ctx
    wk, wv, kn = make_kv_weights(g, 0, device=bed.dev)
    sk_s, sv_s = wl.suffix_k.clone(), wl.suffix_v.clone()
    ms = timer.time(lambda: ctx.kv_project(bed.plan, wl.x, wk, wv, kn, sk_s, sv_s), args.steps)
    flops = 2.0 * wl.n_req * wl.S * g.hidden * 2 * g.n_kv_heads * g.head_dim
    if ctx.sync_status() != 0:
        raise RuntimeError("device status after kv_project")
    return {"avg_call_ms": round(statistics.mean(ms), 5),
            "tflops": round(flops / (statistics.mean(ms) * 1e-3) / 1e12, 3)}


def measure_layout(bed, args, timer):
    """The paper's skills layout: a 16-token online system span, 5-token
    online separators between the artifacts, the rest of the online rows (the
    task) last; every online row is a query (S = S_kv)."""
    wl, g, ctx = bed.wl, bed.g, bed.ctx
    if wl.S != wl.S_kv:
        return None
    layouts = []
    for r in wl.requests:
        lay = [-16]
        for k, a in enumerate(r):
            lay += ([a] if k == 0 else [-5, a])
        layouts.append(lay)
    if not all(16 + 5 * (len(r) - 1) <= wl.S_kv for r in wl.requests):
        return None
    lplan = ctx.assemble_layout(layouts)
    flops = 0.0
    for lay in layouts:
        at, online_pos = 0, []
        for it in lay:
            if it >= 0:
                at += wl.art_lengths[it]
            else:
                online_pos += list(range(at, at - it))
                at += -it
        online_pos += list(range(at, at + wl.S_kv - len(online_pos)))
        flops += 4.0 * g.head_dim * g.n_q_heads * sum(p_ + 1 for p_ in online_pos[wl.S_kv - wl.S:])
    ms = timer.time(lambda: ctx.attend(lplan, bed.q, wl.suffix_k, wl.suffix_v, out=bed.out, lse=bed.lse),
                    args.steps)
    lplan.free()
    if ctx.sync_status() != 0:
        raise RuntimeError("device status after the layout attention")
    return {"avg_call_ms": round(statistics.mean(ms), 5),
            "tflops": round(flops / (statistics.mean(ms) * 1e-3) / 1e12, 3),
            "layout": "online system span 16, artifacts with 5-token online separators, task last"}


def measure_warm_cache(bed, args, world, flush, local_rank):
    """Warm-cache end to end: the request's artifacts start in pinned host
    memory (the paper's CPU RAM cache) and are loaded into an emptied pool in
    every step, on a second stream that overlaps the Q projection."""
    import torch
    import paper_2609_36722_gb300 as pkg
    wl, g = bed.wl, bed.g
    stream = torch.cuda.current_stream()
    used = sorted({a for r in wl.requests for a in r})
    remap = {a: i for i, a in enumerate(used)}
    reqs_w = [[remap[a] for a in r] for r in wl.requests]
    ak_h = [wl.art_k[a].cpu().pin_memory() for a in used]
    av_h = [wl.art_v[a].cpu().pin_memory() for a in used]
    art_bytes = sum(t.numel() * 2 for t in ak_h) * 2
    io = HostInputs(bed)
    wctx = pkg.Context.for_geometry(g, pool_blocks=sum(-(-wl.art_lengths[a] // 64) for a in used) + 1,
                                    device=local_rank)
    side = torch.cuda.Stream(device=bed.dev)
    q_w = torch.empty_like(bed.q)
    ev_l0 = torch.cuda.Event(enable_timing=True)
    ev_l1 = torch.cuda.Event(enable_timing=True)

    def warm_step():
        wctx.pool_reset()
        side.wait_stream(stream)
        ev_l0.record(side)
        for i in range(0, len(used), 64):
            wctx.register_artifacts_host(ak_h[i:i + 64], av_h[i:i + 64], stream=side)
        ev_l1.record(side)
        p = wctx.assemble(reqs_w)
        io.copy_in()
        wctx.q_project(p, io.x_d, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=wl.S_kv, out=q_w)
        stream.wait_stream(side)
        wctx.attend(p, q_w, io.sk_d, io.sv_d, out=bed.out, want_lse=False)
        io.out_h.copy_(bed.out, non_blocking=True)
        torch.cuda.synchronize()
        p.free()

    try:
        for _ in range(max(3, args.warmup)):
            warm_step()
        times, load_ms = [], []
        for _ in range(args.steps):
            flush.zero_()
            torch.cuda.synchronize()
            t0 = time.perf_counter()
            warm_step()
            times.append(time.perf_counter() - t0)
            load_ms.append(ev_l0.elapsed_time(ev_l1))
        if wctx.sync_status() != 0:
            raise RuntimeError("device status after the warm-cache steps")
    finally:
        wctx.close()
    warm_s = max_over_ranks(sum(times), world, bed.dev)
    return {"value": round(job_throughput(bed.work, world, args.steps, warm_s) / bed.scale, 3), "unit": bed.unit,
            "h2d_bytes_per_step": io.h2d_bytes + art_bytes, "d2h_bytes_per_step": io.d2h_bytes,
            "artifact_load_ms": round(statistics.mean(load_ms), 4),
            "artifact_load_gbs": round(art_bytes / (statistics.mean(load_ms) * 1e-3) / 1e9, 1),
            "includes": "pool reset, load of the requests' artifact K/V from pinned host memory (one kernel "
                        "over the CPU-GPU link, second stream, overlapping the Q projection), assemble, H2D of "
                        "the step's new tokens (x and their own suffix K/V rows), Q projection, attention, D2H of O"}


def measure_variants(bed, args, timer):
    """The two read variants of the paper's training-free baselines (App.
    C.2) on the same layer: APE's separate context (temperature 0.9) and
    online attention with the calibrated combine (scale 0.9), and EPIC's keys
    stored before RoPE and rotated to their assembled positions at assembly
    (the rotation kernel, then the attention over the rotated keys).  Both
    count the same visible (query, key) pairs as the plain read."""
    import torch
    wl, ctx = bed.wl, bed.ctx
    flops = attention_flops(wl)
    ms = timer.time(lambda: ctx.attend_ape(bed.plan, bed.q, wl.suffix_k, wl.suffix_v, 0.9, 0.9, out=bed.out,
                                           lse=bed.lse), args.steps)
    ape_launches = ctx.last_launch_count()
    ape = {"avg_call_ms": round(statistics.mean(ms), 5),
           "tflops": round(flops / (statistics.mean(ms) * 1e-3) / 1e12, 3), "launches": ape_launches,
           "temperature": 0.9, "scale": 0.9}
    rplan = ctx.assemble(wl.requests)
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    rot_ms = []
    for i in range(max(3, min(args.steps, 10))):
        timer.flush.zero_()
        e0.record()
        ctx.rotate_keys(rplan)
        e1.record()
        e1.synchronize()
        if i >= 1:
            rot_ms.append(e0.elapsed_time(e1))
    g = bed.g
    n_slots = sum(-(-wl.art_lengths[a] // 64) for r in wl.requests for a in r)
    # the artifact tokens' keys read once, every slot's rows written once
    rot_bytes = (sum(wl.t_art(r) for r in range(wl.n_req)) + n_slots * 64) * g.n_kv_heads * g.head_dim * 2
    ms = timer.time(lambda: ctx.attend(rplan, bed.q, wl.suffix_k, wl.suffix_v, out=bed.out, lse=bed.lse),
                    args.steps)
    rplan.free()
    if ctx.sync_status() != 0:
        raise RuntimeError("device status after the read variants")
    peaks = _peaks()
    rot_gbs = rot_bytes / (statistics.mean(rot_ms) * 1e-3) / 1e9 if rot_ms else None
    epic = {"rotate_ms": round(statistics.mean(rot_ms), 5) if rot_ms else None,
            "rotate_gbs": round(rot_gbs, 1) if rot_gbs else None,
            "rotate_frac_of_hbm": round(rot_gbs / peaks["hbm"], 4) if rot_gbs else None,
            "attention_ms": round(statistics.mean(ms), 5),
            "tflops": round(flops / (statistics.mean(ms) * 1e-3) / 1e12, 3)}
    return {"ape": ape, "epic_rotated_keys": epic}


def _guarded(fn, errors, label):
    """Run an optional part of the line; a failure is recorded, not raised."""
    import traceback
    try:
        return fn()
    except Exception as e:  # noqa: BLE001 - reported in the line, and the run exits non-zero
        traceback.print_exc()
        errors.append(label)
        return {"error": f"{type(e).__name__}: {e}"}


def run_ours(args, rank, world, local_rank):
    import torch
    dev = torch.device("cuda", local_rank)
    torch.cuda.set_device(dev)
    flush = torch.empty(L2_FLUSH_BYTES // 4, dtype=torch.float32, device=dev)
    timer = Timer(args.eager, flush)
    errors = []

    # ---- the headline: computed first, and a failure here fails the run
    bed = Bed(args.workload, dev, local_rank)
    core = measure_core(bed, args, world, timer, with_clocks=(rank == 0), local_rank=local_rank)
    e2e = measure_e2e(bed, args, world, flush, local_rank)
    full = None
    if args.workload == HEADLINE:
        n_full, full_ms, full_flops = measure_full_causal(bed)
        full = {"tokens": n_full, "avg_call_ms": round(full_ms, 3),
                "tflops": round(full_flops / (full_ms * 1e-3) / 1e12, 3),
                "frac_of_bf16_peak": round(full_flops / (full_ms * 1e-3) / 1e12 / _peaks()["bf16"], 4),
                "flops": full_flops,
                "work_ratio_full_over_cached": round(full_flops / bed.work, 2),
                "wall_ratio_full_over_cached": round(full_ms / core["roofline"]["avg_launch_ms"], 2)}
    result = {
        "metric": METRIC, "value": core["value"], "unit": core["unit"], "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": core["ms_per_step"], "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "bf16", "data": "synthetic",
        "config": {"workload": args.workload, **core["workload"],
                   "parallelism": f"replicas x{world}",
                   "l2": f"flushed between timed steps ({L2_FLUSH_BYTES >> 20} MiB write, outside the events)",
                   "attention_kernel": "split-KV warp-MMA (attn_mma)" if bed.decode else "tcgen05 (attn_tc)",
                   "launch": "eager calls" if args.eager else "CUDA graph replay of the calls"},
        "roofline": core["roofline"],
        "e2e": e2e,
        "gpu_launches": core["gpu_launches"],
        "clocks": core["clocks"],
        "qproj": core["qproj"],
        "path_work": core["path_work"],
        "full_causal_analogue": full,
    }
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(bed.wl)

    # ---- optional parts: each failure is recorded in the line
    def extras(b):
        out = {}
        if args.sub_lines:
            out["kv_project"] = _guarded(lambda: measure_kv_project(b, args, timer), errors, f"{b.name}.kv_project")
            out["layout_attention"] = _guarded(lambda: measure_layout(b, args, timer), errors,
                                               f"{b.name}.layout_attention")
            out["e2e_warm_cache"] = _guarded(lambda: measure_warm_cache(b, args, world, flush, local_rank), errors,
                                             f"{b.name}.e2e_warm_cache")
            out["read_variants"] = _guarded(lambda: measure_variants(b, args, timer), errors,
                                            f"{b.name}.read_variants")
        return out

    result.update(extras(bed))
    bed.close()
    del bed
    configs = {}
    if not args.no_configs:
        for name in SUB_CONFIGS:
            if name == args.workload:
                continue

            def one(name=name):
                b = Bed(name, dev, local_rank)
                try:
                    c = measure_core(b, args, world, timer, local_rank=local_rank)
                    d = {"value": c["value"], "unit": c["unit"], "ms_per_step": c["ms_per_step"],
                         "roofline": c["roofline"], "qproj": c["qproj"], "gpu_launches": c["gpu_launches"],
                         "config": c["workload"], "path_work": c["path_work"]}
                    d["e2e"] = _guarded(lambda: measure_e2e(b, args, world, flush, local_rank), errors, f"{name}.e2e")
                    d.update(extras(b))
                    return d
                finally:
                    b.close()
            configs[name] = _guarded(one, errors, name)
    result["configs"] = configs
    if errors:
        result["errors"] = errors
    return result, (1 if errors else 0)


def decode_read_fracs(wl, attn_ms, peak_gbs, traffic):
    """The decode roofline counted in the bytes the launch must move: the distinct
    K/V (each shared artifact once) and, when an ncu capture of the current
    kernel exists, the DRAM bytes it did move, each per second against the peak."""
    d = kv_distinct_bytes(wl)
    out = {"distinct_bytes": d, "distinct_frac": round(d / (attn_ms * 1e-3) / 1e9 / peak_gbs, 4)}
    if traffic:
        out["dram_frac"] = round(traffic / (attn_ms * 1e-3) / 1e9 / peak_gbs, 4)
    return out


def load_traffic(workload):
    """DRAM bytes per launch of the dominant kernel from the committed ncu summary,
    or None when there is none or the kernel source changed since it was taken."""
    import hashlib
    p = os.path.join(ROOT, "profiles", "traffic.json")
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f).get(workload)
    if not d:
        return None
    src = os.path.join(ROOT, d["source"])
    if not os.path.exists(src):
        return None
    with open(src, "rb") as f:
        if hashlib.sha256(f.read()).hexdigest()[:16] != d["sha256_16"]:
            return None
    return d["bytes_per_launch"]


# ---------------------------------------------------------------------------
# reference arm: the fp64 oracle on host cores
# ---------------------------------------------------------------------------
def run_reference(args):
    import numpy as np
    import torch
    from gen import make_workload
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    wl = make_workload(args.workload, device=dev).to("cpu")
    decode = is_decode(wl)
    inputs = _oracle_inputs(wl, 0)
    rng = np.random.default_rng(0)
    # a bounded sample per step: fewer tokens where every query row sees more keys
    toks_per_step = max(1, min(4, wl.S, int(4 * 16384 / max(1, wl.t_art(0) + wl.S_kv)) or 1))
    for _ in range(args.warmup):
        oracle_sample(wl, inputs, sorted(rng.choice(wl.S, size=toks_per_step, replace=False).tolist()), decode)
    tot_t, tot_w = 0.0, 0.0
    for _ in range(args.steps):
        dt, w = oracle_sample(wl, inputs, sorted(rng.choice(wl.S, size=toks_per_step, replace=False).tolist()),
                              decode)
        tot_t += dt
        tot_w += w
    scale = 1e9 if decode else 1e12
    unit = "GB/s" if decode else "TFLOP/s"
    value = tot_w / tot_t / scale
    threads = blas_threads()
    full = kv_bytes(wl) if decode else attention_flops(wl)
    sample = (f"per step: request 0, {toks_per_step} random suffix tokens x all {wl.geom.n_q_heads} q heads of "
              f"{wl.n_req * wl.S} query tokens (fp64 numpy oracle, BLAS on {threads} threads); the full step "
              f"extrapolated linearly by work: {full * tot_t / tot_w:.4g} s")
    return {"metric": METRIC, "value": value, "unit": unit, "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": tot_t * 1e3 / args.steps, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": args.workload, "parallelism": "host cores"},
            "cpu_baseline": {"value": value, "unit": unit, "cores": threads, "host_cpus": os.cpu_count(),
                             "kind": "oracle", "sample": sample},
            "e2e": {"value": value, "unit": unit, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", default="ours", choices=["ours", "reference"])
    ap.add_argument("--workload", default=HEADLINE)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-configs", action="store_true",
                    help="time the headline workload only (no per-config sub-objects)")
    ap.add_argument("--no-sub-lines", dest="sub_lines", action="store_false",
                    help="skip the kv_project, layout_attention, e2e_warm_cache and read_variants sub-lines")
    ap.add_argument("--eager", action="store_true",
                    help="launch the timed calls directly instead of replaying CUDA graphs (for profilers)")
    args = ap.parse_args()
    if args.warmup < 3:
        args.warmup = 3

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local_rank = int(os.environ.get("LOCAL_RANK", "0"))

    host_threads_env()
    if args.impl == "reference":
        if rank != 0:
            return
        print(json.dumps(run_reference(args)))
        return

    if world > 1:
        import datetime

        import torch
        torch.cuda.set_device(local_rank)
        # a rank whose part failed must not hold the others at a collective for long
        torch.distributed.init_process_group("nccl", device_id=torch.device("cuda", local_rank),
                                             timeout=datetime.timedelta(minutes=5))
    res, rc = run_ours(args, rank, world, local_rank)
    if rank == 0:
        print(json.dumps(res))
    if world > 1:
        import torch
        torch.distributed.barrier()
        torch.distributed.destroy_process_group()
    if rc:
        sys.exit(rc)


if __name__ == "__main__":
    main()
