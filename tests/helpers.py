"""Shared helpers of the GPU parity tests: load a seeded workload into a
library context and evaluate the oracle on the same inputs."""

from __future__ import annotations

import numpy as np
import torch

import oracle
from gen import make_custom, make_workload


# Tolerances of the parity bar, fixed by the path's precision: bf16 inputs
# and outputs, Q rounded to bf16 once after RoPE, P rounded to bf16 before
# the PV product, fp32 accumulation everywhere.
O_MAX_ABS = 2e-2
O_MEAN_ABS = 2e-3
LSE_MAX_ABS = 1e-2
# Q: one bf16 rounding of values of magnitude up to ~4 (unit-RMS heads)
# gives |dq| <= 2^-8 * 4 = 1.6e-2; fp32 accumulation order adds ~1e-5.
Q_MAX_ABS = 2e-2


def load_context(wl, pool_blocks=None, device=0):
    import paper_2609_36722_gb300 as pkg
    if pool_blocks is None:
        pool_blocks = sum(-(-L // 64) for L in wl.art_lengths) + 1
    ctx = pkg.Context.for_geometry(wl.geom, pool_blocks=pool_blocks, device=device)
    for i, (k, v) in enumerate(zip(wl.art_k, wl.art_v)):
        aid = ctx.register_artifact(k, v)
        assert aid == i
    plan = ctx.assemble(wl.requests)
    return ctx, plan


def run_path(ctx, plan, wl, want_lse=True):
    g = wl.geom
    out, lse = ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w,
                                wl.suffix_k, wl.suffix_v, want_lse=want_lse)
    st = ctx.sync_status()
    assert st == 0, f"device status {st}"
    return out, lse


def compare(o_gpu: np.ndarray, o_ref: np.ndarray, lse_gpu=None, lse_ref=None, label=""):
    err = np.abs(o_gpu - o_ref)
    rel = np.linalg.norm(o_gpu - o_ref) / max(np.linalg.norm(o_ref), 1e-30)
    msg = f"{label}: max|dO|={err.max():.3e} mean|dO|={err.mean():.3e} relF={rel:.3e}"
    ok = err.max() <= O_MAX_ABS and err.mean() <= O_MEAN_ABS and np.all(np.isfinite(o_gpu))
    if lse_gpu is not None:
        lerr = np.abs(lse_gpu - lse_ref)
        msg += f" max|dLSE|={lerr.max():.3e}"
        ok = ok and lerr.max() <= LSE_MAX_ABS
    print(msg)
    assert ok, msg
    assert rel <= 2e-2, msg
    return err.max(), err.mean(), rel


def sample_pairs(wl, n=256, seed=1234):
    """(request, token, head) triples: first and last suffix rows of every
    request, every row of one full head of request 0, plus random ones."""
    rng = np.random.default_rng(seed)
    Hq = wl.geom.n_q_heads
    trip = set()
    for r in range(wl.n_req):
        for h in (0, Hq - 1):
            trip.add((r, 0, h))
            trip.add((r, wl.S - 1, h))
    h0 = int(rng.integers(Hq))
    for i in range(wl.S):
        trip.add((0, i, h0))
    while len(trip) < n + 4 * wl.n_req + wl.S:
        trip.add((int(rng.integers(wl.n_req)), int(rng.integers(wl.S)), int(rng.integers(Hq))))
    return sorted(trip)
