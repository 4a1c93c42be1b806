"""Properties the paper fixes, checked on the GPU path through the C ABI:
B = 0 gives base PIC (App. A.5: the update starts at zero), merged equals
unmerged (App. A.5 Deployment), artifact order does not change the output
(keys pre-rotated at local positions, every artifact visible: Sec. 2, App.
C.1), and stored artifact KV never changes (Sec. 3, App. A.3)."""

import numpy as np
import pytest
import torch

from gen import Geometry, make_custom
from helpers import O_MAX_ABS, O_MEAN_ABS, load_context, run_path

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
GEOM = Geometry(hidden=512, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)


def _wl(seed=21, reqs=((3, 0, 2, 1),), S=40, S_kv=48):
    return make_custom("inv", GEOM, seed, [150, 64, 333, 20], [list(r) for r in reqs], S, S_kv, device=DEV)


def test_b_zero_is_base_pic_bit_exact():
    wl = _wl()
    ctx, plan = load_context(wl)
    g = wl.geom
    zero_b = torch.zeros_like(wl.lora_b)
    o1, l1 = ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, zero_b, g.scale, wl.q_norm_w, wl.suffix_k, wl.suffix_v)
    o2, l2 = ctx.query_attend(plan, wl.x, wl.w_q, None, None, g.scale, wl.q_norm_w, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    assert torch.equal(o1, o2) and torch.equal(l1, l2)


def test_merged_equals_unmerged():
    wl = _wl()
    ctx, plan = load_context(wl)
    g = wl.geom
    merged = (wl.w_q.float() + g.scale * (wl.lora_b.float() @ wl.lora_a.float())).to(torch.bfloat16)
    o1, _ = ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, wl.suffix_k, wl.suffix_v)
    o2, _ = ctx.query_attend(plan, wl.x, merged, None, None, g.scale, wl.q_norm_w, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    d = (o1.double() - o2.double()).abs()
    assert d.max().item() <= O_MAX_ABS and d.mean().item() <= O_MEAN_ABS, (d.max().item(), d.mean().item())


def test_artifact_order_invariance_and_index_maps():
    perms = [(3, 0, 2, 1), (0, 1, 2, 3), (2, 3, 1, 0)]
    wl = _wl(reqs=perms)
    # identical suffix inputs for every request
    wl.x[1:] = wl.x[0]
    wl.suffix_k[1:] = wl.suffix_k[0]
    wl.suffix_v[1:] = wl.suffix_v[0]
    ctx, plan = load_context(wl)
    out, lse = run_path(ctx, plan, wl)
    for r in (1, 2):
        d = (out[r].double() - out[0].double()).abs()
        assert d.max().item() <= O_MAX_ABS / 4 and d.mean().item() <= O_MEAN_ABS / 4
        assert (lse[r] - lse[0]).abs().max().item() <= 1e-3
    # the index maps are the same tokens in permuted order
    ex = plan.export()
    T = wl.t_art(0)
    maps = [ex["index_map"][r * T:(r + 1) * T] for r in range(3)]
    arts = [ex["token_art"][r * T:(r + 1) * T] for r in range(3)]
    offs = [ex["token_off"][r * T:(r + 1) * T] for r in range(3)]
    keyset = [sorted(zip(a.tolist(), o.tolist(), m.tolist())) for a, o, m in zip(arts, offs, maps)]
    assert keyset[0] == keyset[1] == keyset[2]


def test_artifact_kv_unchanged_by_calls():
    wl = _wl()
    ctx, plan = load_context(wl)
    kp, vp, used = ctx.pool_tensors()
    k0 = kp[:used].clone()
    v0 = vp[:used].clone()
    for _ in range(3):
        run_path(ctx, plan, wl)
    torch.cuda.synchronize()
    assert torch.equal(kp[:used].view(torch.int16), k0.view(torch.int16))
    assert torch.equal(vp[:used].view(torch.int16), v0.view(torch.int16))


def test_duplicate_artifact_counts_twice():
    wl = make_custom("dup", GEOM, 23, [100, 70], [[0, 0, 1]], 12, 12, device=DEV)
    import oracle
    ctx, plan = load_context(wl)
    out, lse = run_path(ctx, plan, wl)
    o_ref, l_ref = oracle.workload_reference(wl, 0)
    d = np.abs(out[0].double().cpu().numpy() - o_ref)
    assert d.max() <= O_MAX_ABS and d.mean() <= O_MEAN_ABS
    assert plan.t_art() == [270]


def test_error_paths_leave_context_usable():
    import paper_2609_36722_gb300 as pkg
    wl = _wl()
    ctx, plan = load_context(wl)
    with pytest.raises(pkg.AttunerError) as e:
        ctx.assemble([[0, 99]])
    assert e.value.status == pkg.attuner.ERR_UNKNOWN_ARTIFACT
    with pytest.raises(pkg.AttunerError) as e:
        ctx.register_artifact(torch.zeros(2000, 4, 128, dtype=torch.bfloat16, device=DEV),
                              torch.zeros(2000, 4, 128, dtype=torch.bfloat16, device=DEV))
    assert e.value.status == pkg.attuner.ERR_OOM
    with pytest.raises(ValueError):
        ctx.attend(plan, wl.x, wl.suffix_k, wl.suffix_v)   # wrong shapes / dtypes are caught in the binding
    out, _ = run_path(ctx, plan, wl)
    assert torch.isfinite(out.float()).all()


def test_plans_serve_only_their_context_and_pool_generation():
    import paper_2609_36722_gb300 as pkg
    wl = _wl()
    ctx, plan = load_context(wl)
    other, other_plan = load_context(wl)
    # a plan of another context (same geometry, same pool) is refused before any launch
    with pytest.raises(pkg.AttunerError) as e:
        run_path(other, plan, wl)
    assert e.value.status == pkg.attuner.ERR_INVALID_ARG
    # after a reset the old plan is refused; one assembled afterwards works
    ctx.pool_reset()
    for k, v in zip(wl.art_k, wl.art_v):
        ctx.register_artifact(k, v)
    with pytest.raises(pkg.AttunerError) as e:
        run_path(ctx, plan, wl)
    assert e.value.status == pkg.attuner.ERR_INVALID_ARG
    fresh = ctx.assemble(wl.requests)
    out_a, _ = run_path(ctx, fresh, wl)
    out_b, _ = run_path(other, other_plan, wl)
    assert torch.equal(out_a.view(torch.int16), out_b.view(torch.int16))


@pytest.mark.parametrize("merge", [1, 2])
@pytest.mark.parametrize("S,S_kv", [(1, 129), (40, 48), (300, 300)])
def test_repeated_calls_are_bit_identical(S, S_kv, merge):
    # split-K partial sums and split-KV partials are combined in a fixed order,
    # whichever CTA finishes last and whichever merge path runs
    import paper_2609_36722_gb300 as pkg
    wl = make_custom("det", GEOM, 27, [150, 64, 333, 20], [[3, 0, 2, 1], [1, 2]], S, S_kv, device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, 4)
    ctx.set_option(pkg.OPT_SPLIT_MERGE, merge)
    o1, l1 = run_path(ctx, plan, wl)
    o2, l2 = run_path(ctx, plan, wl)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)


def test_plan_buffers_reused_and_plans_freed_after_their_context():
    # freed plans hand their device buffers back to the context, which reuses
    # them for later assemblies of other sizes: results stay bit-identical to
    # a first assembly; a plan freed after its context releases its own buffer
    import paper_2609_36722_gb300 as pkg
    wl = make_custom("reuse", GEOM, 29, [150, 64, 333, 20, 900], [[3, 0, 2, 1], [1, 2, 4]], 40, 48, device=DEV)
    ctx, plan = load_context(wl)
    o1, l1 = run_path(ctx, plan, wl)
    plan.free()
    for reqs in ([[4, 4, 4, 4], [0]], [[1]], [[0, 1, 2, 3, 4], [4, 3, 2, 1, 0]]):
        ctx.assemble(reqs).free()
    again = ctx.assemble(wl.requests)
    o2, l2 = run_path(ctx, again, wl)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    late = ctx.assemble(wl.requests)
    again.free()
    ctx.close()
    late.free()   # after the context: must not touch it
