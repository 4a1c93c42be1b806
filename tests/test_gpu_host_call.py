"""attuner_query_attend_host through the C ABI: the step's new inputs (hidden
states, and the new tokens' own K/V rows) and its output in host memory,
copied by the library on the caller's stream.

Bar: bit-identical O and LSE to attuner_query_attend on the same inputs placed
on the device by the caller (the same kernels run on the same bytes); the rows
before the new tokens in the caller's suffix K/V are left as they were; and O
within the oracle's tolerance."""

import numpy as np
import pytest
import torch

import oracle
from gen import Geometry, make_custom
from helpers import compare, load_context

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
G128 = Geometry(hidden=512, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)

f64 = oracle.bf16_to_f64


def _pinned(t):
    return t.cpu().contiguous().pin_memory()


@pytest.mark.parametrize("S,S_kv,reqs", [(150, 150, [[1, 0], [3, 2, 0]]), (40, 70, [[1, 0], [3, 2, 0]]),
                                          (1, 129, [[1, 0], [3, 2, 0]]),
                                          # decode whose requests share most artifacts: shared reads
                                          (1, 129, [[1, 0], [1, 3, 2, 0], [0, 1], [3, 1]])])
def test_host_call_matches_device_call(S, S_kv, reqs):
    wl = make_custom("hostcall", G128, 101, [37, 700, 64, 129], reqs, S, S_kv, device=DEV)
    g = wl.geom
    ctx, plan = load_context(wl)
    stream = torch.cuda.Stream(device=DEV)
    # device reference: the caller's own buffers already hold every row
    out_d, lse_d = ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w,
                                    wl.suffix_k, wl.suffix_v)
    # host call: the new rows come from host memory into a device buffer whose
    # earlier rows are the resident cache (and whose new rows hold garbage)
    sk = wl.suffix_k.clone()
    sv = wl.suffix_v.clone()
    sk[:, S_kv - S:] = 7.0
    sv[:, S_kv - S:] = -7.0
    old_k = sk[:, :S_kv - S].clone()
    x_h = _pinned(wl.x)
    k_h, v_h = _pinned(wl.suffix_k[:, S_kv - S:]), _pinned(wl.suffix_v[:, S_kv - S:])
    out_h = torch.empty(wl.n_req, S, g.n_q_heads, g.head_dim, dtype=torch.bfloat16, pin_memory=True)
    lse_h = torch.empty(wl.n_req, S, g.n_q_heads, dtype=torch.float32, pin_memory=True)
    torch.cuda.synchronize()
    ctx.query_attend_host(plan, x_h, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, sk, sv, k_h, v_h,
                          out_host=out_h, lse_host=lse_h, stream=stream)
    stream.synchronize()
    assert ctx.sync_status(stream=stream) == 0
    assert torch.equal(out_h.view(torch.int16), out_d.cpu().view(torch.int16))
    assert torch.equal(lse_h, lse_d.cpu())
    assert torch.equal(sk[:, S_kv - S:].view(torch.int16), wl.suffix_k[:, S_kv - S:].view(torch.int16))
    assert torch.equal(sv[:, S_kv - S:].view(torch.int16), wl.suffix_v[:, S_kv - S:].view(torch.int16))
    assert torch.equal(sk[:, :S_kv - S].view(torch.int16), old_k.view(torch.int16))
    for r in range(wl.n_req):
        o_ref, l_ref = oracle.workload_reference(wl, r)
        compare(f64(out_h[r]), o_ref, f64(lse_h[r]), l_ref, label=f"host call S={S} S_kv={S_kv} req {r}")


def test_host_call_without_new_rows_and_lse():
    # k_new/v_new omitted: the device suffix buffers already hold the new rows;
    # no LSE requested
    S = S_kv = 64
    wl = make_custom("hostcall2", G128, 103, [300, 5], [[0, 1]], S, S_kv, device=DEV)
    g = wl.geom
    ctx, plan = load_context(wl)
    out_d, _ = ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w,
                                wl.suffix_k, wl.suffix_v, want_lse=False)
    out_h, lse_h = ctx.query_attend_host(plan, _pinned(wl.x), wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w,
                                         wl.suffix_k, wl.suffix_v)
    torch.cuda.synchronize()
    assert lse_h is None
    assert ctx.sync_status() == 0
    assert torch.equal(out_h.view(torch.int16), out_d.cpu().view(torch.int16))
