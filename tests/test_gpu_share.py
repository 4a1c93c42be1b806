"""Shared artifact reads of the decode kernel against the fp64 oracle.

When several requests of one call use the same artifact, the warp-MMA kernel
can read each chunk of it once for a group of those requests (up to 16 packed
query rows per CTA) and merge every request's partial results afterwards by
their log-sum-exp (the split-KV identity of the attention over the assembled
keys).  These cases force the mode on and off on plans with repeated
artifacts (across requests and within one request), requests without
artifacts, chunked artifacts and online chunks, every group size and both
head sizes, and compare each with the oracle.
"""

import numpy as np
import pytest
import torch

import oracle
from gen import Geometry, make_custom
from helpers import compare, load_context, run_path

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None

LENGTHS = [300, 77, 640, 64, 1, 129, 1000]
REQS = [[2, 0], [1], [3, 1, 0, 2], [], [6, 2, 2], [5, 4, 6, 0], [0, 2, 6], [4]]


def _reference(wl):
    outs, lses = [], []
    for r in range(wl.n_req):
        o, l = oracle.workload_reference(wl, r)
        outs.append(o)
        lses.append(l)
    return np.stack(outs), np.stack(lses)


def _np(t):
    return t.double().cpu().numpy()


def _case(G, D, S, S_kv, seed):
    geom = Geometry(hidden=256, n_q_heads=2 * G, n_kv_heads=2, head_dim=D, rank=8)
    return make_custom("share", geom, seed, LENGTHS, REQS, S, S_kv, device=DEV)


@pytest.mark.parametrize("G,D,S", [(1, 128, 1), (2, 128, 1), (4, 128, 1), (8, 128, 1), (4, 64, 1), (4, 128, 2),
                                   (2, 64, 4)])
@pytest.mark.parametrize("share,split", [(1, 0), (2, 0), (2, 3), (2, 16)])
def test_shared_reads_match_oracle(G, D, S, share, split):
    import paper_2609_36722_gb300 as pkg
    wl = _case(G, D, S, 200 + S, seed=31 + G + D + S)
    o_ref, lse_ref = _reference(wl)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, 2)
    ctx.set_option(pkg.OPT_SHARE_READS, share)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label=f"share={share} split={split} G={G} D={D} S={S}")


def test_shared_reads_are_deterministic():
    import paper_2609_36722_gb300 as pkg
    wl = _case(4, 128, 1, 129, seed=3)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_SHARE_READS, 2)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, 4)
    o1, l1 = run_path(ctx, plan, wl)
    o2, l2 = run_path(ctx, plan, wl)
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    assert torch.equal(l1, l2)


def test_shared_and_per_request_reads_agree():
    # the two decompositions merge the same keys in different chunks: equal up
    # to the rounding of the merge (bf16 outputs)
    import paper_2609_36722_gb300 as pkg
    wl = _case(4, 128, 1, 129, seed=5)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_SHARE_READS, 1)
    o1, l1 = run_path(ctx, plan, wl)
    ctx.set_option(pkg.OPT_SHARE_READS, 2)
    o2, l2 = run_path(ctx, plan, wl)
    assert (o1.float() - o2.float()).abs().max().item() <= 1.6e-2
    assert (l1 - l2).abs().max().item() <= 1e-4


def test_static_scratch_takes_a_64_request_shared_decode():
    # 64 decode requests over a 32-artifact pool (the bench's decode recipe,
    # smaller hidden size): the shared-read partials (S G rows per record) fit
    # the allocation-free entry point's fixed scratch, and its result is the
    # pool-backed call's, bit for bit (same decomposition, same arithmetic)
    import paper_2609_36722_gb300 as pkg
    rng = np.random.default_rng(61)
    lengths = rng.integers(256, 2049, size=32).tolist()
    reqs = [rng.choice(32, size=int(rng.integers(4, 13)), replace=False).tolist() for _ in range(64)]
    geom = Geometry(hidden=256, n_q_heads=32, n_kv_heads=8, head_dim=128, rank=16)
    wl = make_custom("dec64", geom, 61, lengths, reqs, 1, 129, device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_SHARE_READS, 2)
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, geom.scale, wl.q_norm_w, S_kv=wl.S_kv)
    o1, l1 = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    o2, l2 = ctx.attend_static_scratch(plan, q, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    assert torch.equal(o1.view(torch.int16), o2.view(torch.int16))
    assert torch.equal(l1, l2)
    # and both against the oracle on a sample of requests
    for r in (0, 17, 63):
        o_ref, lse_ref = oracle.workload_reference(wl, r)
        compare(_np(o1[r:r + 1]), o_ref[None], _np(l1[r:r + 1]), lse_ref[None], label=f"dec64 request {r}")


@pytest.mark.parametrize("seed", range(6))
def test_random_decode_plans_both_decompositions(seed):
    # random plans: artifacts repeated across and within requests, empty
    # requests, lengths across block boundaries, random group size, head size,
    # rows per request (S G <= 16) and chunk size; shared reads forced on and off
    import paper_2609_36722_gb300 as pkg
    rng = np.random.default_rng(100 + seed)
    G = int(rng.choice([1, 2, 4, 8]))
    D = int(rng.choice([64, 128]))
    S = int(rng.choice([s for s in (1, 2, 3, 4) if s * G <= 16]))
    n_kv = int(rng.choice([1, 2, 4]))
    geom = Geometry(hidden=256, n_q_heads=G * n_kv, n_kv_heads=n_kv, head_dim=D, rank=8)
    lengths = [int(x) for x in rng.integers(1, 400, size=int(rng.integers(2, 9)))]
    n_req = int(rng.integers(1, 13))
    reqs = [[int(a) for a in rng.integers(0, len(lengths), size=int(rng.integers(0, 6)))] for _ in range(n_req)]
    S_kv = S + int(rng.integers(0, 150))
    wl = make_custom(f"rand{seed}", geom, 200 + seed, lengths, reqs, S, S_kv, device=DEV)
    o_ref, lse_ref = _reference(wl)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, 2)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, int(rng.choice([0, 1, 2, 5])))
    for share in (1, 2):
        ctx.set_option(pkg.OPT_SHARE_READS, share)
        out, lse = run_path(ctx, plan, wl)
        compare(_np(out), o_ref, _np(lse), lse_ref,
                label=f"seed={seed} share={share} G={G} D={D} S={S} n_req={n_req} S_kv={S_kv}")
