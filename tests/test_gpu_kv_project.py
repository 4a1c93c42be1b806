"""The suffix tokens' own keys and values through the C ABI
(attuner_kv_project): base k_proj / v_proj (the adaptation changes W^Q only,
Sec. 3), key norm and RoPE at the tokens' assembled positions (App. A.5),
written into the last S token rows of each request's suffix K/V.

Bar: K and V within the Q tolerance of the fp64 oracle (one bf16 rounding of
unit-RMS / unit-variance values); every other row of the caller's buffers
unchanged bit for bit; the attention over the produced suffix K/V within the
O tolerance of the oracle fed the oracle's own K/V."""

import numpy as np
import pytest
import torch

import oracle
from gen import Geometry, make_custom, make_kv_weights
from helpers import Q_MAX_ABS, compare, load_context

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
G128 = Geometry(hidden=512, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)
G64 = Geometry(hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=64, rank=8)

f64 = oracle.bf16_to_f64


def _oracle_kv(wl, wk, wv, kn, r):
    g = wl.geom
    pos = oracle.query_positions(wl.t_art(r), wl.S, wl.S_kv)
    return oracle.kv_projection(f64(wl.x[r]), f64(wk), f64(wv), f64(kn), g.rms_eps, g.rope_theta, pos,
                                g.n_kv_heads)


@pytest.mark.parametrize("geom,S,S_kv", [(G128, 50, 70), (G128, 300, 300), (G64, 16, 16), (G128, 1, 129)])
def test_kv_project_matches_oracle(geom, S, S_kv):
    wl = make_custom("kvp", geom, 61, [37, 700, 64, 1, 129], [[1, 0, 3], [4, 2, 2, 0]], S, S_kv, device=DEV)
    wk, wv, kn = make_kv_weights(geom, 61, device=DEV)
    ctx, plan = load_context(wl)
    sk = wl.suffix_k.clone()
    sv = wl.suffix_v.clone()
    ctx.kv_project(plan, wl.x, wk, wv, kn, sk, sv)
    assert ctx.sync_status() == 0
    new = slice(S_kv - S, S_kv)
    for r in range(wl.n_req):
        k_ref, v_ref = _oracle_kv(wl, wk, wv, kn, r)
        dk = np.abs(f64(sk[r, new]) - k_ref).max()
        dv = np.abs(f64(sv[r, new]) - v_ref).max()
        assert dk <= Q_MAX_ABS and dv <= Q_MAX_ABS, (r, dk, dv)
        # rows before the new tokens are the caller's and stay as they were
        assert torch.equal(sk[r, :S_kv - S].view(torch.int16), wl.suffix_k[r, :S_kv - S].view(torch.int16))
        assert torch.equal(sv[r, :S_kv - S].view(torch.int16), wl.suffix_v[r, :S_kv - S].view(torch.int16))


@pytest.mark.parametrize("rows,split", [(128, 1), (256, 2), (128, 8), (256, 4)])
def test_kv_project_shapes_match_oracle(rows, split):
    # the projection kernel's shapes pinned (rows per CTA, K slices per tile)
    import paper_2609_36722_gb300 as pkg
    geom, S, S_kv = G128, 300, 310
    wl = make_custom("kvs", geom, 71, [37, 700], [[1, 0], [0]], S, S_kv, device=DEV)
    wk, wv, kn = make_kv_weights(geom, 71, device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_QPROJ_ROWS, rows)
    ctx.set_option(pkg.OPT_QPROJ_SPLIT_K, split)
    sk = wl.suffix_k.clone()
    sv = wl.suffix_v.clone()
    ctx.kv_project(plan, wl.x, wk, wv, kn, sk, sv)
    assert ctx.sync_status() == 0
    new = slice(S_kv - S, S_kv)
    for r in range(wl.n_req):
        k_ref, v_ref = _oracle_kv(wl, wk, wv, kn, r)
        dk = np.abs(f64(sk[r, new]) - k_ref).max()
        dv = np.abs(f64(sv[r, new]) - v_ref).max()
        assert dk <= Q_MAX_ABS and dv <= Q_MAX_ABS, (r, dk, dv)
        assert torch.equal(sk[r, :S_kv - S].view(torch.int16), wl.suffix_k[r, :S_kv - S].view(torch.int16))


def test_decode_appends_one_token_per_step():
    # one request decoding three tokens into a buffer with room for 132 rows:
    # the prefix of S_kv rows is the call's contiguous [1, S_kv, Hkv, d] view,
    # and step t writes row 128 + t only
    geom = G128
    wl0 = make_custom("kvdec", geom, 67, [300, 77, 640], [[2, 0]], 1, 132, device=DEV)
    wk, wv, kn = make_kv_weights(geom, 67, device=DEV)
    sk = wl0.suffix_k.clone()
    sv = wl0.suffix_v.clone()
    before_k, before_v = sk.clone(), sv.clone()
    for t in range(3):
        S_kv = 129 + t
        wl = make_custom("kvdec", geom, 70 + t, [300, 77, 640], [[2, 0]], 1, S_kv, device=DEV)
        ctx, plan = load_context(wl)
        k_view, v_view = sk[:, :S_kv], sv[:, :S_kv]
        assert k_view.is_contiguous() and k_view.data_ptr() == sk.data_ptr()
        ctx.kv_project(plan, wl.x, wk, wv, kn, k_view, v_view)
        assert ctx.sync_status() == 0
        k_ref, v_ref = _oracle_kv(wl, wk, wv, kn, 0)
        assert np.abs(f64(sk[0, S_kv - 1:S_kv]) - k_ref).max() <= Q_MAX_ABS
        assert np.abs(f64(sv[0, S_kv - 1:S_kv]) - v_ref).max() <= Q_MAX_ABS
    # rows 0..127 never change; the last row (never appended) keeps its bytes
    assert torch.equal(sk[:, :128].view(torch.int16), before_k[:, :128].view(torch.int16))
    assert torch.equal(sv[:, :128].view(torch.int16), before_v[:, :128].view(torch.int16))
    assert torch.equal(sk[:, 131:].view(torch.int16), before_k[:, 131:].view(torch.int16))


def test_layer_with_online_kv_matches_oracle():
    # K/V of the suffix from the library, then the attention over them, against
    # the oracle fed its own fp64 K/V for the new rows
    geom = G128
    S, S_kv = 40, 56
    wl = make_custom("kvlayer", geom, 73, [37, 700, 64, 1, 129], [[1, 0, 3], [4, 2, 2, 0]], S, S_kv, device=DEV)
    wk, wv, kn = make_kv_weights(geom, 73, device=DEV)
    ctx, plan = load_context(wl)
    sk = wl.suffix_k.clone()
    sv = wl.suffix_v.clone()
    ctx.kv_project(plan, wl.x, wk, wv, kn, sk, sv)
    g = wl.geom
    out, lse = ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, sk, sv)
    assert ctx.sync_status() == 0
    outs, lses = [], []
    for r in range(wl.n_req):
        k_ref, v_ref = _oracle_kv(wl, wk, wv, kn, r)
        suf_k = f64(wl.suffix_k[r]).copy()
        suf_v = f64(wl.suffix_v[r]).copy()
        suf_k[S_kv - S:] = k_ref
        suf_v[S_kv - S:] = v_ref
        ids = wl.requests[r]
        o, l = oracle.request_forward(
            f64(wl.x[r]), f64(wl.w_q), f64(wl.lora_a), f64(wl.lora_b), g.scale, f64(wl.q_norm_w), g.rms_eps,
            g.rope_theta, [f64(wl.art_k[i]) for i in ids], [f64(wl.art_v[i]) for i in ids], suf_k, suf_v,
            g.n_q_heads)
        outs.append(o)
        lses.append(l)
    compare(f64(out), np.stack(outs), f64(lse), np.stack(lses), label="online K/V layer")
