"""attuner_attend_static_scratch: the attention entry point for callers that
cannot allocate GPU memory (a serving engine that owns the whole device, a
runtime that bars other libraries from allocating because an allocation can
synchronise the device).  Its split-KV partial results live in a fixed
device array of the library instead of a stream-ordered pool.

The test calls it through the C ABI twice in a row on a layout that splits
the KV (so the fixed array is really used, and the second call finds the
first call's contents there) and compares each result with attuner_attend
on the same inputs, and checks that a call takes no device memory: on a
context whose pool has never been drawn from, the GPU's free memory is the
same before and after the calls (while attuner_attend on the same layout
does draw from that pool).  It must pass alone in a fresh process and after
every other test; pytest collects this file last."""

import numpy as np
import pytest
import torch

from gen import Geometry, make_custom
from helpers import LSE_MAX_ABS, O_MAX_ABS, O_MEAN_ABS, load_context

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None


def _close(a, b):
    d = (a.double() - b.double()).abs()
    return d.max().item() <= O_MAX_ABS and d.mean().item() <= O_MEAN_ABS


@pytest.mark.parametrize("kernel,split,S,S_kv", [(1, 4, 96, 96), (2, 0, 1, 129)])
def test_static_scratch_matches_attend_twice(kernel, split, S, S_kv):
    import paper_2609_36722_gb300 as pkg
    geom = Geometry(hidden=256, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)
    wl = make_custom("noalloc", geom, 41, [700, 333, 1200, 64], [[2, 0, 3], [1, 3], [0, 1, 2, 3]], S, S_kv,
                     device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    g = wl.geom
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=S_kv)
    ref_o, ref_l = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    # the KV must split so that the partial results go through the scratch:
    # chunks of `split` blocks for the tcgen05 kernel, of at least 16 blocks
    # (the decode chunk at this size) for the warp-MMA kernel; either kernel
    # merges its chunks itself (one launch)
    n_blocks = [sum(-(-wl.art_lengths[a] // 64) for a in req) + -(-S_kv // 64) for req in wl.requests]
    if kernel == 1:
        assert min(n_blocks) > split
    else:
        assert max(n_blocks) > 16
    launches = 1
    assert ctx.last_launch_count() == launches
    for _ in range(2):
        out, lse = ctx.attend_static_scratch(plan, q, wl.suffix_k, wl.suffix_v)
        assert ctx.sync_status() == 0
        assert ctx.last_launch_count() == launches
        assert _close(out, ref_o)
        assert (lse - ref_l).abs().max().item() <= LSE_MAX_ABS


@pytest.mark.parametrize("split", [4, 24])
def test_static_scratch_cluster_merge(split):
    # split-KV chunks merged inside thread-block clusters (4 and 2 CTAs): no
    # partial results in any scratch, the output leaves by the kernel's tensor
    # store; the result equals attuner_attend's
    import paper_2609_36722_gb300 as pkg
    geom = Geometry(hidden=256, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)
    wl = make_custom("noalloc_cl", geom, 43, [700, 333, 1200, 64], [[2, 0, 3], [1, 3], [0, 1, 2, 3]], 96, 96,
                     device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, 1)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    ctx.set_option(pkg.OPT_SPLIT_MERGE, 2)
    g = wl.geom
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=96)
    ref_o, ref_l = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0 and ctx.last_launch_count() == 1
    out, lse = ctx.attend_static_scratch(plan, q, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0 and ctx.last_launch_count() == 1
    assert torch.equal(out, ref_o) and torch.equal(lse, ref_l)


@pytest.mark.parametrize("kernel,split,S,S_kv", [(1, 4, 96, 96), (2, 0, 1, 129)])
def test_static_scratch_takes_no_device_memory(kernel, split, S, S_kv):
    import paper_2609_36722_gb300 as pkg
    geom = Geometry(hidden=256, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)
    wl = make_custom("noalloc_mem", geom, 47, [700, 333, 1200, 64], [[2, 0, 3], [1, 3], [0, 1, 2, 3]], S, S_kv,
                     device=DEV)
    g = wl.geom

    def configured(c):
        c.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
        c.set_option(pkg.OPT_SPLIT_BLOCKS, split)
        return c

    # a first context: the Q rows, and one call that loads the kernels and
    # sets up the fixed array's address (module loading may take memory)
    ctx_a, plan_a = load_context(wl)
    configured(ctx_a)
    q = ctx_a.q_project(plan_a, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=S_kv)
    ref_o, ref_l = ctx_a.attend_static_scratch(plan_a, q, wl.suffix_k, wl.suffix_v)
    assert ctx_a.sync_status() == 0
    # a fresh context: its stream-ordered pool has never been drawn from, so
    # any allocation from it (or any cudaMalloc) takes free device memory
    ctx_b, plan_b = load_context(wl)
    configured(ctx_b)
    out = torch.empty_like(q)
    lse = torch.empty(q.shape[:3], dtype=torch.float32, device=DEV)
    torch.cuda.synchronize()
    free0 = torch.cuda.mem_get_info(DEV)[0]
    for _ in range(2):
        ctx_b.attend_static_scratch(plan_b, q, wl.suffix_k, wl.suffix_v, out=out, lse=lse)
        assert ctx_b.sync_status() == 0
    torch.cuda.synchronize()
    free1 = torch.cuda.mem_get_info(DEV)[0]
    assert free1 == free0, f"free device memory {free0} -> {free1}"
    assert _close(out, ref_o) and (lse - ref_l).abs().max().item() <= LSE_MAX_ABS
    # the check can see an allocation: attuner_attend on the same split layout
    # draws its partial results from the pool
    ctx_b.attend(plan_b, q, wl.suffix_k, wl.suffix_v, out=out, lse=lse)
    assert ctx_b.sync_status() == 0
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info(DEV)[0] < free1


def test_static_scratch_rejects_calls_beyond_its_size():
    import paper_2609_36722_gb300 as pkg
    geom = Geometry(hidden=256, n_q_heads=32, n_kv_heads=8, head_dim=128, rank=16)
    # 8 KV heads x 64 row tiles x 8 splits of 128-row fp32 partials is far over 32 MiB
    wl = make_custom("big", geom, 43, [4096], [[0]], 2048, 2048, device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, 16)
    q = torch.zeros(1, 2048, 32, 128, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(pkg.AttunerError) as e:
        ctx.attend_static_scratch(plan, q, wl.suffix_k, wl.suffix_v)
    assert e.value.status == pkg.attuner.ERR_INVALID_ARG
    assert "32" in str(e.value) or "bytes" in str(e.value)
