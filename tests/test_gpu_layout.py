"""Prompt layouts whose online text interleaves with the cached artifacts
(App. "Prompt Construction and Artifact Boundaries": instructions, separators
and the question are online, only artifact spans are cached), through the C
ABI: attuner_assemble_layout, then the Q projection, the K/V projection and
the attention.

Bar: O within max-abs 2e-2 / mean-abs 2e-3 and LSE within 1e-2 of the fp64
oracle (layout_forward) for both attention kernels and both split merges; K
of the online rows rotated at their assembled positions within the Q
tolerance; a layout without online items gives bit-identical results to the
plain plan."""

import numpy as np
import pytest
import torch

import oracle
from gen import Geometry, make_custom, make_kv_weights
from helpers import Q_MAX_ABS, compare, load_context

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
G128 = Geometry(hidden=512, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)
LENGTHS = [37, 700, 64, 1, 129, 300]
# request 0: system text, artifact 1, separator, artifact 0, separator, artifact 3, then the question;
# request 1: artifacts 4 and 2 (twice) around separators, starting with an online span
LAYOUTS = [[-12, 1, -5, 0, -5, 3], [-7, 4, -5, 2, -70, 2, 0]]

f64 = oracle.bf16_to_f64


def _wl(S, S_kv, seed=81):
    reqs = [[a for a in lay if a >= 0] for lay in LAYOUTS]
    return make_custom("layout", G128, seed, LENGTHS, reqs, S, S_kv, device=DEV)


def _reference(wl, layouts):
    g = wl.geom
    arts_k = {i: f64(t) for i, t in enumerate(wl.art_k)}
    arts_v = {i: f64(t) for i, t in enumerate(wl.art_v)}
    outs, lses = [], []
    for r, lay in enumerate(layouts):
        o, l = oracle.layout_forward(f64(wl.x[r]), f64(wl.w_q), f64(wl.lora_a), f64(wl.lora_b), g.scale,
                                     f64(wl.q_norm_w), g.rms_eps, g.rope_theta, lay, arts_k, arts_v,
                                     f64(wl.suffix_k[r]), f64(wl.suffix_v[r]), g.n_q_heads)
        outs.append(o)
        lses.append(l)
    return np.stack(outs), np.stack(lses)


def _run(ctx, plan, wl):
    g = wl.geom
    out, lse = ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w,
                                wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    return out, lse


@pytest.mark.parametrize("kernel,split,merge", [(1, 0, 0), (1, 4, 1), (1, 4, 2), (2, 0, 0), (2, 4, 0)])
def test_layout_prefill_every_online_row_is_a_query(kernel, split, merge):
    import paper_2609_36722_gb300 as pkg
    S = S_kv = 150          # explicit online rows: 22 and 82; the rest is the question
    wl = _wl(S, S_kv)
    ref_o, ref_l = _reference(wl, LAYOUTS)
    ctx, _ = load_context(wl)
    plan = ctx.assemble_layout(LAYOUTS)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    ctx.set_option(pkg.OPT_SPLIT_MERGE, merge)
    out, lse = _run(ctx, plan, wl)
    compare(f64(out), ref_o, f64(lse), ref_l, label=f"layout kernel={kernel} split={split} merge={merge}")


def test_layout_decode_token():
    S, S_kv = 1, 129
    wl = _wl(S, S_kv, seed=83)
    ref_o, ref_l = _reference(wl, LAYOUTS)
    ctx, _ = load_context(wl)
    plan = ctx.assemble_layout(LAYOUTS)
    out, lse = _run(ctx, plan, wl)
    compare(f64(out), ref_o, f64(lse), ref_l, label="layout decode")


def test_layout_without_online_items_is_the_plain_plan():
    S = S_kv = 70
    wl = _wl(S, S_kv, seed=85)
    ctx, plan = load_context(wl)
    o1, l1 = _run(ctx, plan, wl)
    plan2 = ctx.assemble_layout(wl.requests)
    o2, l2 = _run(ctx, plan2, wl)
    assert torch.equal(o1, o2) and torch.equal(l1, l2)
    e1, e2 = plan.export(), plan2.export()
    for key in e1:
        np.testing.assert_array_equal(e1[key], e2[key], err_msg=key)


def test_layout_online_keys_rotated_at_assembled_positions():
    S = S_kv = 150
    wl = _wl(S, S_kv, seed=87)
    wk, wv, kn = make_kv_weights(wl.geom, 87, device=DEV)
    ctx, _ = load_context(wl)
    plan = ctx.assemble_layout(LAYOUTS)
    sk = torch.zeros_like(wl.suffix_k)
    sv = torch.zeros_like(wl.suffix_v)
    ctx.kv_project(plan, wl.x, wk, wv, kn, sk, sv)
    assert ctx.sync_status() == 0
    g = wl.geom
    for r, lay in enumerate(LAYOUTS):
        pos = oracle.layout_online_positions(lay, LENGTHS, S_kv)
        k_ref, v_ref = oracle.kv_projection(f64(wl.x[r]), f64(wk), f64(wv), f64(kn), g.rms_eps, g.rope_theta,
                                            pos, g.n_kv_heads)
        assert np.abs(f64(sk[r]) - k_ref).max() <= Q_MAX_ABS
        assert np.abs(f64(sv[r]) - v_ref).max() <= Q_MAX_ABS


def test_layout_rejects_too_few_online_rows():
    import paper_2609_36722_gb300 as pkg
    wl = _wl(50, 50)
    ctx, _ = load_context(wl)
    plan = ctx.assemble_layout(LAYOUTS)          # request 1 has 82 online rows in its spans
    q = torch.zeros(2, 50, 16, 128, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(pkg.AttunerError) as e:
        ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    assert e.value.status == pkg.attuner.ERR_INVALID_ARG


# Many short online spans (1 to 5 tokens) between many artifacts: the online
# rows are read packed after the artifact slots, so every one of these spans
# shares 64-row chunks with its neighbours.
MANY_LENGTHS = [37, 90, 64, 1, 129, 300, 5, 66, 200, 17, 128, 63]
MANY_LAYOUTS = [
    [-3, 0, -1, 1, -5, 2, -2, 3, -4, 4, -1, 5, -3, 6, -5, 7, -1, 8, -2, 9, -4, 10, -1, 11],
    [4, -1, -2, 6, -5, 0, -3, 3, 3, -4, 11, -1, 7],      # starts with an artifact; adjacent spans; a repeat
    [-5, 8, -1, 2, -2, 9, -5],                             # ends with an explicit span
]


def _many_wl(S, S_kv, seed):
    reqs = [[a for a in lay if a >= 0] for lay in MANY_LAYOUTS]
    return make_custom("layout_many", G128, seed, MANY_LENGTHS, reqs, S, S_kv, device=DEV)


def _many_reference(wl):
    g = wl.geom
    arts_k = {i: f64(t) for i, t in enumerate(wl.art_k)}
    arts_v = {i: f64(t) for i, t in enumerate(wl.art_v)}
    outs, lses = [], []
    for r, lay in enumerate(MANY_LAYOUTS):
        o, l = oracle.layout_forward(f64(wl.x[r]), f64(wl.w_q), f64(wl.lora_a), f64(wl.lora_b), g.scale,
                                     f64(wl.q_norm_w), g.rms_eps, g.rope_theta, lay, arts_k, arts_v,
                                     f64(wl.suffix_k[r]), f64(wl.suffix_v[r]), g.n_q_heads)
        outs.append(o)
        lses.append(l)
    return np.stack(outs), np.stack(lses)


@pytest.mark.parametrize("kernel,split,merge", [(1, 0, 0), (1, 2, 1), (1, 4, 2), (2, 0, 0), (2, 2, 0)])
def test_layout_many_short_spans(kernel, split, merge):
    import paper_2609_36722_gb300 as pkg
    S = S_kv = 140          # explicit online rows: 32, 16 and 13; every online row is a query
    wl = _many_wl(S, S_kv, 91)
    ref_o, ref_l = _many_reference(wl)
    ctx, _ = load_context(wl)
    plan = ctx.assemble_layout(MANY_LAYOUTS)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    ctx.set_option(pkg.OPT_SPLIT_MERGE, merge)
    out, lse = _run(ctx, plan, wl)
    compare(f64(out), ref_o, f64(lse), ref_l, label=f"many spans kernel={kernel} split={split} merge={merge}")


def test_layout_many_short_spans_decode():
    S, S_kv = 1, 129
    wl = _many_wl(S, S_kv, 93)
    ref_o, ref_l = _many_reference(wl)
    ctx, _ = load_context(wl)
    plan = ctx.assemble_layout(MANY_LAYOUTS)
    out, lse = _run(ctx, plan, wl)
    compare(f64(out), ref_o, f64(lse), ref_l, label="many spans decode")


@pytest.mark.parametrize("share", [1, 2])
def test_layout_decode_with_shared_reads(share):
    # four decode tokens whose layouts share artifacts (and online spans before
    # and between them): every query sits in its final span and sees every
    # artifact, so the decode kernel may read each artifact once for all four
    import paper_2609_36722_gb300 as pkg
    layouts = [[-12, 1, -5, 0, -5, 3], [-7, 4, -5, 2, -70, 2, 0], [1, -5, 0], [-3, 3, 1, 0]]
    reqs = [[a for a in lay if a >= 0] for lay in layouts]
    wl = make_custom("layout_share", G128, 87, LENGTHS, reqs, 1, 129, device=DEV)
    ref_o, ref_l = _reference(wl, layouts)
    ctx, _ = load_context(wl)
    plan = ctx.assemble_layout(layouts)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, 2)
    ctx.set_option(pkg.OPT_SHARE_READS, share)
    out, lse = _run(ctx, plan, wl)
    compare(f64(out), ref_o, f64(lse), ref_l, label=f"layout decode share={share}")
