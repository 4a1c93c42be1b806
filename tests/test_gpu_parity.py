"""GPU parity of the CUDA path against the fp64 oracle on the same seeded
inputs.  Every call goes through the C ABI (ctypes binding).

Bar: block table, valid lengths, index map and gathered K/V bytes are
bit-exact; O (bf16) within max-abs 2e-2 and mean-abs 2e-3; LSE within 1e-2.
"""

import numpy as np
import pytest
import torch

import oracle
from gen import Geometry, make_custom, make_workload
from helpers import (Q_MAX_ABS, compare, load_context, run_path)

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None

G128 = Geometry(hidden=512, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)


def _full_reference(wl):
    outs, lses = [], []
    for r in range(wl.n_req):
        o, l = oracle.workload_reference(wl, r)
        outs.append(o)
        lses.append(l)
    return np.stack(outs), np.stack(lses)


def _np(t):
    return t.double().cpu().numpy()


@pytest.fixture(scope="module")
def tiny():
    wl = make_workload("tiny", device=DEV)
    return wl, _full_reference(wl)


def test_assemble_bit_exact_tiny(tiny):
    wl, _ = tiny
    ctx, plan = load_context(wl)
    ex = plan.export()
    ref = oracle.assemble(wl.art_lengths, wl.requests[0])
    for key in ("block_table", "valid_len", "index_map", "token_art", "token_off"):
        np.testing.assert_array_equal(ex[key], ref[key], err_msg=key)
    assert plan.t_art() == [201]
    # the gathered K/V bytes are the registered artifacts, bit for bit
    kp, vp, used = ctx.pool_tensors()
    assert used == ref["total_blocks"]
    idx = torch.as_tensor(ex["index_map"], device=DEV, dtype=torch.long)
    k_tok = kp.permute(0, 2, 1, 3).reshape(-1, wl.geom.n_kv_heads, wl.geom.head_dim)[idx]
    v_tok = vp.permute(0, 2, 1, 3).reshape(-1, wl.geom.n_kv_heads, wl.geom.head_dim)[idx]
    k_cat = torch.cat([wl.art_k[a] for a in wl.requests[0]])
    v_cat = torch.cat([wl.art_v[a] for a in wl.requests[0]])
    assert torch.equal(k_tok.view(torch.int16), k_cat.view(torch.int16))
    assert torch.equal(v_tok.view(torch.int16), v_cat.view(torch.int16))


@pytest.mark.parametrize("split_k", [1, 2])
def test_q_project_tiny(tiny, split_k):
    import paper_2609_36722_gb300 as pkg
    wl, _ = tiny
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_QPROJ_SPLIT_K, split_k)
    g = wl.geom
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=wl.S_kv)
    assert ctx.sync_status() == 0
    q_ref = oracle.workload_reference(wl, 0, q_only=True)
    err = np.abs(_np(q[0]) - q_ref)
    print(f"q: max|dq|={err.max():.3e} mean={err.mean():.3e} max|q|={np.abs(q_ref).max():.2f}")
    assert err.max() <= Q_MAX_ABS


@pytest.mark.parametrize("kernel", [2, 1])
def test_query_attend_tiny(tiny, kernel):
    import paper_2609_36722_gb300 as pkg
    wl, (o_ref, lse_ref) = tiny
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label=f"tiny kernel={kernel}")


def _ragged(seed=7, n_req=2, S=50, S_kv=70, geom=G128, lengths=(37, 200, 64, 1, 129), reqs=None):
    reqs = reqs if reqs is not None else [[1, 0, 3], [4, 2, 2, 0]][:n_req]
    return make_custom("ragged", geom, seed, list(lengths), reqs, S, S_kv, device=DEV)


@pytest.mark.parametrize("kernel", [2, 1])
@pytest.mark.parametrize("split", [0, 2, 4])
def test_ragged_multi_request(kernel, split):
    import paper_2609_36722_gb300 as pkg
    wl = _ragged()
    o_ref, lse_ref = _full_reference(wl)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label=f"ragged kernel={kernel} split={split}")


@pytest.mark.parametrize("merge", [1, 2])
@pytest.mark.parametrize("split,S,S_kv", [(2, 50, 70), (4, 300, 300), (6, 130, 200), (0, 300, 300)])
def test_split_merge_modes(merge, split, S, S_kv):
    # tcgen05 kernel, split-KV chunks merged through global memory (1) or inside
    # one thread-block cluster per row tile (2); 300 suffix tokens x G = 4 give
    # ragged 256-row tiles; clusters of 2 or 4 chunks per row tile (each CTA
    # producing whole column blocks), global mode with up to 6 chunks
    import paper_2609_36722_gb300 as pkg
    wl = _ragged(seed=17, S=S, S_kv=S_kv, lengths=(37, 700, 64, 1, 1290))
    o_ref, lse_ref = _full_reference(wl)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, 1)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    ctx.set_option(pkg.OPT_SPLIT_MERGE, merge)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label=f"merge={merge} split={split} S={S}")


G64 = Geometry(hidden=256, n_q_heads=8, n_kv_heads=2, head_dim=64, rank=8)


@pytest.mark.parametrize("merge", [1, 2])
@pytest.mark.parametrize("split,S,S_kv", [(4, 300, 300), (16, 130, 200)])
def test_split_merge_modes_head_dim_64(merge, split, S, S_kv):
    # head_dim 64: clusters of 4 (16 output columns per CTA, a 32-byte row of
    # the output tile) and of 2 (32 columns, 64-byte rows), and the global mode
    import paper_2609_36722_gb300 as pkg
    wl = _ragged(seed=19, S=S, S_kv=S_kv, geom=G64, lengths=(37, 700, 64, 1, 1290))
    o_ref, lse_ref = _full_reference(wl)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, 1)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    ctx.set_option(pkg.OPT_SPLIT_MERGE, merge)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label=f"d=64 merge={merge} split={split} S={S}")


@pytest.mark.parametrize("G", [1, 2, 8])
def test_group_sizes(G):
    geom = Geometry(hidden=256, n_q_heads=4 * G, n_kv_heads=4, head_dim=128, rank=8)
    wl = make_custom("groups", geom, 11, [100, 300], [[1, 0]], 33, 40, device=DEV)
    o_ref, lse_ref = _full_reference(wl)
    ctx, plan = load_context(wl)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label=f"G={G}")


def test_no_artifacts_is_causal_self_attention():
    wl = make_custom("suffix_only", G128, 3, [64], [[]], 200, 200, device=DEV)
    o_ref, lse_ref = _full_reference(wl)
    ctx, plan = load_context(wl)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label="suffix only")


def test_decode_shape():
    # one query token per request, S_kv = prior + 1
    wl = make_custom("decode", G128, 5, [300, 77, 640, 64], [[2, 0], [1], [3, 1, 0, 2]], 1, 129, device=DEV)
    o_ref, lse_ref = _full_reference(wl)
    ctx, plan = load_context(wl)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label="decode")


@pytest.mark.parametrize("kernel,S,S_kv", [(2, 1, 9), (1, 8, 12)])
def test_most_requests_per_call(kernel, S, S_kv):
    # 512 requests, as many as one call takes (the kernels' per-request tables);
    # ragged artifact lists, some empty, every request its own suffix
    import paper_2609_36722_gb300 as pkg
    rng = np.random.default_rng(29)
    lengths = rng.integers(1, 200, size=16).tolist()
    reqs = [rng.choice(16, size=int(rng.integers(0, 4)), replace=False).tolist() for _ in range(512)]
    wl = make_custom("max_req", G128, 29, lengths, reqs, S, S_kv, device=DEV)
    # the oracle per request, the shared weights and artifacts widened once
    f, g = oracle.bf16_to_f64, wl.geom
    w_q, a, b, qn = f(wl.w_q), f(wl.lora_a), f(wl.lora_b), f(wl.q_norm_w)
    ak, av = [f(t) for t in wl.art_k], [f(t) for t in wl.art_v]
    x, sk, sv = f(wl.x), f(wl.suffix_k), f(wl.suffix_v)
    refs = [oracle.request_forward(x[r], w_q, a, b, g.scale, qn, g.rms_eps, g.rope_theta, [ak[i] for i in ids],
                                   [av[i] for i in ids], sk[r], sv[r], g.n_q_heads) for r, ids in enumerate(reqs)]
    o_ref, lse_ref = np.stack([o for o, _ in refs]), np.stack([l for _, l in refs])
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref, label=f"512 requests kernel={kernel}")
    with pytest.raises(pkg.AttunerError):
        ctx.assemble(reqs + [[0]])


G64P = Geometry(hidden=512, n_q_heads=4, n_kv_heads=2, head_dim=64, rank=8)


def _q_shape_case(geom, rank, rows, split, seed=13):
    """Q projection with the kernel shape pinned (rows per CTA, K slices per
    tile): two requests of 150 suffix tokens (M = 300: row tiles of 128 end
    in a ragged 44-row tile, of 256 in a tile whose second accumulator holds
    no row), against the oracle row by row."""
    import paper_2609_36722_gb300 as pkg
    g = Geometry(hidden=geom.hidden, n_q_heads=geom.n_q_heads, n_kv_heads=geom.n_kv_heads,
                 head_dim=geom.head_dim, rank=rank)
    wl = make_custom("qshape", g, seed, [100, 37], [[0], [1, 0]], 150, 150, device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_QPROJ_ROWS, rows)
    ctx.set_option(pkg.OPT_QPROJ_SPLIT_K, split)
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=wl.S_kv)
    assert ctx.sync_status() == 0
    for r in range(wl.n_req):
        q_ref = oracle.workload_reference(wl, r, q_only=True)
        err = np.abs(_np(q[r]) - q_ref)
        assert err.max() <= Q_MAX_ABS, (rows, split, r, err.max())
    return ctx, plan, wl, q


@pytest.mark.parametrize("rows", [128, 256])
@pytest.mark.parametrize("split", [1, 2, 4, 8])
def test_q_project_shapes_match_oracle(rows, split):
    _q_shape_case(G128, 16, rows, split)


@pytest.mark.parametrize("rows,split", [(128, 1), (128, 4), (256, 1), (128, 8)])
def test_q_project_shapes_rank64(rows, split):
    # LoRA rank 64: the widest partial rows (D + 64 columns) the exchange carries
    # (256-row tiles with a K split do not fit this width in shared memory)
    _q_shape_case(G128, 64, rows, split, seed=17)


@pytest.mark.parametrize("rows,split", [(128, 1), (128, 2), (128, 4), (256, 1), (256, 2), (256, 8)])
def test_q_project_shapes_head64(rows, split):
    _q_shape_case(G64P, 8, rows, split, seed=19)


def test_q_project_shapes_are_deterministic():
    # the K slices are summed in slice order: two calls give the same bytes
    ctx, plan, wl, q1 = _q_shape_case(G128, 16, 256, 4)
    g = wl.geom
    q2 = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=wl.S_kv)
    assert ctx.sync_status() == 0
    assert torch.equal(q1.view(torch.int16), q2.view(torch.int16))


def test_q_project_unsupported_shape_refused():
    # head size 64 with 8 K slices of 128-row tiles would leave 4 columns per
    # thread: no kernel shape, so the call is refused before any launch
    import paper_2609_36722_gb300 as pkg
    wl = make_custom("qbad", G64P, 23, [40], [[0]], 16, 16, device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_QPROJ_ROWS, 128)
    ctx.set_option(pkg.OPT_QPROJ_SPLIT_K, 8)
    g = wl.geom
    with pytest.raises(pkg.AttunerError):
        ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=wl.S_kv)
    with pytest.raises(pkg.AttunerError):
        ctx.set_option(pkg.OPT_QPROJ_SPLIT_K, 3)
    with pytest.raises(pkg.AttunerError):
        ctx.set_option(pkg.OPT_QPROJ_ROWS, 64)


@pytest.mark.parametrize("seed", range(6))
def test_random_prefill_plans(seed):
    # random plans for the tcgen05 kernel: artifacts repeated across and within
    # requests, empty requests, lengths across block boundaries, ragged row
    # tiles, random group size and head size; the split merge mode and split
    # size forced at random
    import paper_2609_36722_gb300 as pkg
    rng = np.random.default_rng(300 + seed)
    G = int(rng.choice([1, 2, 4, 8]))
    D = int(rng.choice([64, 128]))
    n_kv = int(rng.choice([1, 2, 4]))
    geom = Geometry(hidden=256, n_q_heads=G * n_kv, n_kv_heads=n_kv, head_dim=D, rank=8)
    lengths = [int(x) for x in rng.integers(1, 900, size=int(rng.integers(2, 7)))]
    n_req = int(rng.integers(1, 4))
    reqs = [[int(a) for a in rng.integers(0, len(lengths), size=int(rng.integers(0, 5)))] for _ in range(n_req)]
    S = int(rng.integers(17, 260))
    S_kv = S + int(rng.integers(0, 100))
    wl = make_custom(f"randp{seed}", geom, 400 + seed, lengths, reqs, S, S_kv, device=DEV)
    o_ref, lse_ref = _full_reference(wl)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, 1)
    merge, split = int(rng.choice([0, 1, 2])), int(rng.choice([0, 2, 4, 6]))
    ctx.set_option(pkg.OPT_SPLIT_MERGE, merge)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    out, lse = run_path(ctx, plan, wl)
    compare(_np(out), o_ref, _np(lse), lse_ref,
            label=f"seed={seed} G={G} D={D} S={S} S_kv={S_kv} n_req={n_req} merge={merge} split={split}")
