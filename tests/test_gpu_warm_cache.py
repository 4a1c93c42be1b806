"""Warm-cache load of artifact KV from pinned host memory (the "CPU RAM cache
lookup and GPU transfer" stage of the paper's time-to-first-token, Sec. 5 and
App. A.3): attuner_register_artifacts_host and attuner_pool_reset, through the
C ABI.

Bar: the pool a host load writes is byte-identical to the one device
registration writes (zeroed tails of partial blocks included); attention over
host-loaded artifacts matches the oracle within the usual tolerance, also
after a pool reset with different artifacts and when the load runs on a second
stream that overlaps the Q projection."""

import ctypes

import numpy as np
import pytest
import torch

import oracle
from gen import Geometry, make_custom
from helpers import compare, load_context, run_path

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
GEOM = Geometry(hidden=512, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)


def _wl(seed=31, lengths=(37, 700, 64, 1, 129), reqs=([1, 0, 3], [4, 2, 2, 0]), S=50, S_kv=70):
    return make_custom("warm", GEOM, seed, list(lengths), [list(r) for r in reqs], S, S_kv, device=DEV)


def _pinned(ts):
    return [t.cpu().pin_memory() for t in ts]


def _reference(wl):
    outs, lses = [], []
    for r in range(wl.n_req):
        o, l = oracle.workload_reference(wl, r)
        outs.append(o)
        lses.append(l)
    return np.stack(outs), np.stack(lses)


def _used_pool(ctx):
    kp, vp, used = ctx.pool_tensors()
    return kp[:used].clone(), vp[:used].clone()


def test_host_load_matches_device_registration():
    import paper_2609_36722_gb300 as pkg
    wl = _wl()
    ref_ctx, _ = load_context(wl)
    ctx = pkg.Context.for_geometry(wl.geom, pool_blocks=sum(-(-L // 64) for L in wl.art_lengths) + 1)
    ks, vs = _pinned(wl.art_k), _pinned(wl.art_v)      # alive until the copy has run
    ids = ctx.register_artifacts_host(ks, vs)
    torch.cuda.synchronize()
    assert ids == list(range(len(wl.art_lengths)))
    k1, v1 = _used_pool(ref_ctx)
    k2, v2 = _used_pool(ctx)
    assert torch.equal(k1.view(torch.int16), k2.view(torch.int16))
    assert torch.equal(v1.view(torch.int16), v2.view(torch.int16))


def test_attention_over_host_loaded_artifacts():
    import paper_2609_36722_gb300 as pkg
    wl = _wl()
    o_ref, lse_ref = _reference(wl)
    ctx = pkg.Context.for_geometry(wl.geom, pool_blocks=sum(-(-L // 64) for L in wl.art_lengths) + 1)
    ks, vs = _pinned(wl.art_k), _pinned(wl.art_v)
    ctx.register_artifacts_host(ks, vs)
    plan = ctx.assemble(wl.requests)
    out, lse = run_path(ctx, plan, wl)
    compare(out.double().cpu().numpy(), o_ref, lse.double().cpu().numpy(), lse_ref, label="host-loaded")


def test_reset_then_reload_other_artifacts():
    # a first set fills the pool with other data (its tails included); after a
    # reset, a second set with different lengths must read exactly as a fresh
    # pool holding only the second set
    import paper_2609_36722_gb300 as pkg
    first = _wl(seed=41, lengths=(1000, 130, 17))
    second = _wl(seed=43, lengths=(37, 700, 64, 1, 129))
    ctx = pkg.Context.for_geometry(GEOM, pool_blocks=40)
    for k, v in zip(first.art_k, first.art_v):
        ctx.register_artifact(k, v)
    ctx.pool_reset()
    ks, vs = _pinned(second.art_k), _pinned(second.art_v)
    ids = ctx.register_artifacts_host(ks, vs)
    assert ids == list(range(5))
    torch.cuda.synchronize()
    fresh, _ = load_context(second, pool_blocks=40)
    k1, v1 = _used_pool(fresh)
    k2, v2 = _used_pool(ctx)
    assert torch.equal(k1.view(torch.int16), k2.view(torch.int16))
    assert torch.equal(v1.view(torch.int16), v2.view(torch.int16))
    o_ref, lse_ref = _reference(second)
    plan = ctx.assemble(second.requests)
    out, lse = run_path(ctx, plan, second)
    compare(out.double().cpu().numpy(), o_ref, lse.double().cpu().numpy(), lse_ref, label="after reset")


def test_load_on_second_stream_overlapping_q_projection():
    import paper_2609_36722_gb300 as pkg
    wl = _wl(seed=47)
    o_ref, lse_ref = _reference(wl)
    g = wl.geom
    ctx = pkg.Context.for_geometry(g, pool_blocks=sum(-(-L // 64) for L in wl.art_lengths) + 1)
    ks, vs = _pinned(wl.art_k), _pinned(wl.art_v)
    main, side = torch.cuda.current_stream(), torch.cuda.Stream()
    side.wait_stream(main)
    ctx.register_artifacts_host(ks, vs, stream=side)       # block ids are known on the host at once
    plan = ctx.assemble(wl.requests)
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=wl.S_kv)
    main.wait_stream(side)
    out, lse = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    compare(out.double().cpu().numpy(), o_ref, lse.double().cpu().numpy(), lse_ref, label="second stream")


def test_rejections():
    import paper_2609_36722_gb300 as pkg
    from paper_2609_36722_gb300 import attuner as A
    wl = _wl()
    ctx = pkg.Context.for_geometry(wl.geom, pool_blocks=20)
    k_page = wl.art_k[0].cpu()                           # pageable, not pinned
    v_page = wl.art_v[0].cpu()
    kp = (ctypes.c_void_p * 1)(k_page.data_ptr())
    vp = (ctypes.c_void_p * 1)(v_page.data_ptr())
    lens = (ctypes.c_int32 * 1)(k_page.shape[0])
    ids = (ctypes.c_int32 * 1)()
    assert A.lib().attuner_register_artifacts_host(ctx.handle, 1, kp, vp, lens, None, ids) == A.ERR_INVALID_ARG
    assert A.lib().attuner_register_artifacts_host(ctx.handle, 0, kp, vp, lens, None, ids) == A.ERR_INVALID_ARG
    # the five artifacts take 1 + 11 + 1 + 1 + 3 = 17 of the 20 blocks; 4 more do not fit,
    # and a load that does not fit registers nothing
    ks, vs = _pinned(wl.art_k), _pinned(wl.art_v)
    ctx.register_artifacts_host(ks, vs)
    big = _pinned([torch.zeros(64 * 4, 4, 128, dtype=torch.bfloat16)])
    with pytest.raises(pkg.AttunerError) as e:
        ctx.register_artifacts_host(big, big)
    assert e.value.status == A.ERR_OOM
    torch.cuda.synchronize()
    _, _, used = ctx.pool_tensors()
    assert used == sum(-(-L // 64) for L in wl.art_lengths)
