"""Failure detection without a GPU fault: one role of the attention kernel
waits on an mbarrier that nothing arrives at.  Its bounded wait runs out,
the kernel drains the copies and MMAs it issued, frees its tensor memory and
returns; the host reads ATTUNER_ERR_TIMEOUT from the status word and the
context stays usable for the next, correct call."""

import pytest
import torch

from gen import Geometry, make_custom
from helpers import load_context, run_path

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None


@pytest.mark.parametrize("kernel", [2, 1])
def test_stuck_wait_reports_timeout_and_recovers(kernel):
    import paper_2609_36722_gb300 as pkg
    geom = Geometry(hidden=256, n_q_heads=8, n_kv_heads=2, head_dim=128, rank=8)
    wl = make_custom("stuck", geom, 31, [500, 300], [[0, 1]], 64, 64, device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
    ref, _ = run_path(ctx, plan, wl)
    ctx.set_option(pkg.OPT_WAIT_LIMIT, 4_000_000)          # ~2 ms
    ctx.set_option(pkg.OPT_TEST_STUCK_WAIT, 1)
    g = wl.geom
    ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == pkg.attuner.ERR_TIMEOUT
    ctx.set_option(pkg.OPT_TEST_STUCK_WAIT, 0)
    ctx.set_option(pkg.OPT_WAIT_LIMIT, 0)
    out, _ = run_path(ctx, plan, wl)
    assert torch.equal(out, ref)


def test_sync_check_option_makes_the_call_report_the_timeout():
    # with ATTUNER_OPT_SYNC_CHECK the compute call itself waits for its stream and
    # returns the device status: a correct call returns OK, a stuck wait TIMEOUT
    import paper_2609_36722_gb300 as pkg
    geom = Geometry(hidden=256, n_q_heads=8, n_kv_heads=2, head_dim=128, rank=8)
    wl = make_custom("stuck_sync", geom, 33, [500, 300], [[1, 0]], 64, 64, device=DEV)
    ctx, plan = load_context(wl)
    ref, _ = run_path(ctx, plan, wl)
    ctx.set_option(pkg.OPT_SYNC_CHECK, 1)
    g = wl.geom
    args = (plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, wl.suffix_k, wl.suffix_v)
    out, _ = ctx.query_attend(*args)
    assert torch.equal(out, ref)
    ctx.set_option(pkg.OPT_WAIT_LIMIT, 4_000_000)          # ~2 ms
    ctx.set_option(pkg.OPT_TEST_STUCK_WAIT, 1)
    with pytest.raises(pkg.AttunerError) as e:
        ctx.query_attend(*args)
    assert e.value.status == pkg.attuner.ERR_TIMEOUT
    ctx.set_option(pkg.OPT_TEST_STUCK_WAIT, 0)
    ctx.set_option(pkg.OPT_WAIT_LIMIT, 0)
    assert ctx.sync_status() == 0                           # the call consumed the status
    out, _ = ctx.query_attend(*args)
    assert torch.equal(out, ref)
