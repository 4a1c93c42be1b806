"""Pins of the fp64 oracle against what the paper and the mathematics fix.

None of these tests needs a GPU.  Each oracle function is checked against
something other than itself: hand-derived closed forms (tests/golden/),
invariants the paper states (B = 0 gives base PIC, merged = unmerged, the
artifact order does not matter, one artifact at global positions is full
causal attention), and an fp64 library routine
(torch.nn.functional.scaled_dot_product_attention on the CPU).
"""

import json
import math
import os

import numpy as np
import pytest
import torch

from conftest import GOLDEN
import oracle
from oracle import attuner_oracle as O


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _runs(runs, total):
    out = np.full(total, -1, dtype=np.int64)
    for start, count, first in runs:
        out[start:start + count] = first + np.arange(count)
    return out


def _const_runs(runs, total):
    out = np.full(total, -1, dtype=np.int64)
    for start, count, val in runs:
        out[start:start + count] = val
    return out


# --------------------------------------------------------------------------
# Eq. (query-adaptation) and the merged deployment form
# --------------------------------------------------------------------------
def test_lora_projection_hand_example():
    g = _golden("lora_q_projection_2x2.json")
    w, a, b = (np.array(g[k]) for k in ("w_q", "lora_a", "lora_b"))
    x = np.array(g["x"])
    q = O.lora_q_projection(x, w, a, b, g["s"])
    np.testing.assert_allclose(q, np.array(g["q_raw"]), atol=1e-14)
    np.testing.assert_allclose(O.merged_q_weight(w, a, b, g["s"]), np.array(g["merged_w"]), atol=1e-14)


def test_b_zero_is_base_pic():
    # App. A.5: B starts at zero, so the initial update is zero.
    rng = np.random.default_rng(11)
    x = rng.standard_normal((5, 24))
    w = rng.standard_normal((12, 24))
    a = rng.standard_normal((4, 24))
    b0 = np.zeros((12, 4))
    np.testing.assert_array_equal(O.lora_q_projection(x, w, a, b0, 2.0), O.lora_q_projection(x, w, None, None, 2.0))


def test_merged_equals_unmerged_and_scale_linear():
    rng = np.random.default_rng(12)
    x = rng.standard_normal((7, 32))
    w = rng.standard_normal((16, 32))
    a = rng.standard_normal((4, 32))
    b = rng.standard_normal((16, 4))
    un = O.lora_q_projection(x, w, a, b, 2.0)
    mg = x @ O.merged_q_weight(w, a, b, 2.0).T
    np.testing.assert_allclose(un, mg, rtol=1e-12, atol=1e-12)
    # the update is linear in s: f(2) - f(0) = 2 (f(1) - f(0))
    f0 = O.lora_q_projection(x, w, a, b, 0.0)
    f1 = O.lora_q_projection(x, w, a, b, 1.0)
    np.testing.assert_allclose(un - f0, 2.0 * (f1 - f0), rtol=1e-12, atol=1e-12)
    # superposition over the rows of x: projecting unit vectors gives the columns
    eye = np.eye(32)
    cols = O.lora_q_projection(eye, w, a, b, 2.0)          # [32, 16]
    np.testing.assert_allclose(x @ cols, un, rtol=1e-12, atol=1e-11)


# --------------------------------------------------------------------------
# q RMSNorm
# --------------------------------------------------------------------------
def test_rmsnorm_hand_example():
    g = _golden("rms_norm_d2.json")
    q = np.array(g["q"]).reshape(1, 1, 2)
    for c in g["cases"]:
        out = O.rms_norm_heads(q, np.array(g["w"]), c["eps"])
        np.testing.assert_allclose(out.reshape(-1), c["out"], atol=1e-14)


def test_rmsnorm_invariants():
    rng = np.random.default_rng(13)
    q = rng.standard_normal((6, 3, 16)) * 5
    out = O.rms_norm_heads(q, np.ones(16), 1e-6)
    rms = np.sqrt(np.mean(out ** 2, axis=-1))
    assert np.all(rms <= 1.0) and np.all(rms > 1.0 - 1e-6)
    # scale invariance and per-head independence (a wrong axis breaks one of these)
    np.testing.assert_allclose(O.rms_norm_heads(3.0 * q, np.ones(16), 0.0), O.rms_norm_heads(q, np.ones(16), 0.0), atol=1e-13)
    q2 = q.copy()
    q2[:, 1, :] *= 100.0
    q2[:, 2, :] = rng.standard_normal((6, 16))
    np.testing.assert_array_equal(O.rms_norm_heads(q2, np.ones(16), 1e-6)[:, 0], O.rms_norm_heads(q, np.ones(16), 1e-6)[:, 0])


# --------------------------------------------------------------------------
# RoPE
# --------------------------------------------------------------------------
def test_rope_hand_example():
    g = _golden("rope_d4.json")
    q = np.array(g["q"]).reshape(1, 1, 4)
    out = O.rope_rotate_half(q, np.array([g["pos"]]), g["theta"])
    np.testing.assert_allclose(out.reshape(-1), g["out"], atol=1e-13)


def test_rope_invariants():
    rng = np.random.default_rng(14)
    d, theta = 64, 1.0e6
    q = rng.standard_normal((5, 2, d))
    k = rng.standard_normal((5, 2, d))
    p = np.array([0, 3, 17, 201, 131071])
    # R(0) = I
    np.testing.assert_array_equal(O.rope_rotate_half(q, np.zeros(5, dtype=np.int64), theta), q)
    # norm preserving
    np.testing.assert_allclose(np.linalg.norm(O.rope_rotate_half(q, p, theta), axis=-1), np.linalg.norm(q, axis=-1), rtol=1e-12)
    # relative position: <R(p) q, R(p') k> = <R(p + c) q, R(p' + c) k>
    p2 = np.array([5, 9, 1, 60, 100])
    for c in (1, 37, 4096):
        lhs = np.sum(O.rope_rotate_half(q, p, theta) * O.rope_rotate_half(k, p2, theta), axis=-1)
        rhs = np.sum(O.rope_rotate_half(q, p + c, theta) * O.rope_rotate_half(k, p2 + c, theta), axis=-1)
        np.testing.assert_allclose(lhs, rhs, rtol=1e-9, atol=1e-9)
    # composition R(a) R(b) = R(a + b)
    np.testing.assert_allclose(O.rope_rotate_half(O.rope_rotate_half(q, p, theta), p2, theta),
                               O.rope_rotate_half(q, p + p2, theta), atol=1e-9)


def test_kv_projection_invariants():
    # The suffix tokens' keys and values (base k_proj / v_proj, Sec. 3: only
    # W^Q is adapted), pinned by properties a dropped term, a transposed
    # operand, a wrong axis or a wrong position would break.
    rng = np.random.default_rng(21)
    hkv, d, hidden, theta = 2, 8, 6, 1.0e6
    w_k = rng.standard_normal((hkv * d, hidden))
    w_v = rng.standard_normal((hkv * d, hidden))
    ones = np.ones(d)
    # a basis input selects one column of each weight: V is that column, K its
    # per-head unit-RMS normalisation (position 0: no rotation, eps = 0)
    for i in range(hidden):
        x = np.zeros((1, hidden))
        x[0, i] = 1.0
        k, v = O.kv_projection(x, w_k, w_v, ones, 0.0, theta, np.array([0]), hkv)
        np.testing.assert_allclose(v.reshape(-1), w_v[:, i], rtol=1e-14)
        col = w_k[:, i].reshape(hkv, d)
        np.testing.assert_allclose(k[0], col / np.sqrt(np.mean(col * col, axis=-1, keepdims=True)), rtol=1e-12)
    x = rng.standard_normal((5, hidden))
    pos = np.array([3, 40, 41, 700, 131000])
    k, v = O.kv_projection(x, w_k, w_v, ones, 0.0, theta, pos, hkv)
    # unit RMS per head survives the rotation: |k| = sqrt(d)
    np.testing.assert_allclose(np.linalg.norm(k, axis=-1), np.sqrt(d), rtol=1e-12)
    # V is linear in x and ignores positions and the key weights
    k2, v2 = O.kv_projection(2.0 * x, w_k, w_v, ones, 0.0, theta, pos + 5, hkv)
    np.testing.assert_allclose(v2, 2.0 * v, rtol=1e-13)
    # the key normalisation is scale-invariant (eps = 0), so 2x only moves the rotation:
    # shifting every position by 5 rotates each pair by 5 * inv_freq, preserving <k_t, k_u>
    np.testing.assert_allclose(np.einsum("thd,uhd->thu", k2, k2), np.einsum("thd,uhd->thu", k, k), atol=1e-9)
    # query . key depends only on the position difference (the property RoPE exists for)
    q = rng.standard_normal((5, hkv, d))
    for c in (1, 64, 4096):
        kc, _ = O.kv_projection(x, w_k, w_v, ones, 0.0, theta, pos + c, hkv)
        lhs = np.sum(O.rope_rotate_half(q, pos[::-1], theta) * k, axis=-1)
        rhs = np.sum(O.rope_rotate_half(q, pos[::-1] + c, theta) * kc, axis=-1)
        np.testing.assert_allclose(lhs, rhs, rtol=1e-9, atol=1e-9)
    # the key-norm weight scales each channel after the normalisation
    w = rng.standard_normal(d)
    kw, _ = O.kv_projection(x, w_k, w_v, w, 0.0, theta, np.zeros(5, dtype=np.int64), hkv)
    k0, _ = O.kv_projection(x, w_k, w_v, ones, 0.0, theta, np.zeros(5, dtype=np.int64), hkv)
    np.testing.assert_allclose(kw, k0 * w, rtol=1e-12)


def test_layout_online_positions_hand_example():
    # online 3, artifact of 5, online 2, artifact of 4, then the final online rows
    pos = O.layout_online_positions([-3, 0, -2, 1], [5, 4], 12)
    np.testing.assert_array_equal(pos, [0, 1, 2, 8, 9, 14, 15, 16, 17, 18, 19, 20])


def _layout_case(seed=5, items=(-3, 1, -2, 0, -4, 2), S=9, S_kv=16):
    rng = np.random.default_rng(seed)
    hkv, G, d, hidden, r = 2, 2, 8, 12, 4
    lens = {0: 7, 1: 5, 2: 9}
    art_k = {i: rng.standard_normal((L, hkv, d)) for i, L in lens.items()}
    art_v = {i: rng.standard_normal((L, hkv, d)) for i, L in lens.items()}
    ok, ov = rng.standard_normal((S_kv, hkv, d)), rng.standard_normal((S_kv, hkv, d))
    x = rng.standard_normal((S, hidden))
    w_q = rng.standard_normal((hkv * G * d, hidden)) / math.sqrt(hidden)
    a = rng.standard_normal((r, hidden)) / math.sqrt(hidden)
    b = rng.standard_normal((hkv * G * d, r)) / math.sqrt(r)
    qn = 1.0 + 0.1 * rng.standard_normal(d)
    return dict(x=x, w_q=w_q, a=a, b=b, s=2.0, q_norm_w=qn, eps=1e-6, theta=1.0e4, items=list(items),
                art_k=art_k, art_v=art_v, online_k=ok, online_v=ov, n_q_heads=hkv * G)


def test_layout_without_online_items_is_the_classic_layout():
    c = _layout_case(items=(1, 0, 2))
    o1, l1 = O.layout_forward(**c)
    o2, l2 = O.request_forward(c["x"], c["w_q"], c["a"], c["b"], c["s"], c["q_norm_w"], c["eps"], c["theta"],
                               [c["art_k"][i] for i in (1, 0, 2)], [c["art_v"][i] for i in (1, 0, 2)],
                               c["online_k"], c["online_v"], c["n_q_heads"])
    np.testing.assert_allclose(o1, o2, rtol=1e-13, atol=1e-13)
    np.testing.assert_allclose(l1, l2, rtol=1e-13, atol=1e-13)


def test_layout_against_sdpa_over_the_assembled_sequence():
    # the assembled sequence built token by token, queries rotated at their
    # positions, and fp64 SDPA with an explicit boolean mask key <= query
    c = _layout_case()
    S, S_kv = c["x"].shape[0], c["online_k"].shape[0]
    seq_k, seq_v, online_pos = [], [], []
    row = 0
    for it in c["items"]:
        n = c["art_k"][it].shape[0] if it >= 0 else -it
        for t in range(n):
            if it >= 0:
                seq_k.append(c["art_k"][it][t]); seq_v.append(c["art_v"][it][t])
            else:
                online_pos.append(len(seq_k)); seq_k.append(c["online_k"][row]); seq_v.append(c["online_v"][row])
                row += 1
    while row < S_kv:
        online_pos.append(len(seq_k)); seq_k.append(c["online_k"][row]); seq_v.append(c["online_v"][row])
        row += 1
    K, V = np.stack(seq_k), np.stack(seq_v)
    pos_q = np.asarray(online_pos[S_kv - S:])
    d = K.shape[-1]
    q_raw = O.lora_q_projection(c["x"], c["w_q"], c["a"], c["b"], c["s"]).reshape(S, c["n_q_heads"], d)
    q = O.rope_rotate_half(O.rms_norm_heads(q_raw, c["q_norm_w"], c["eps"]), pos_q, c["theta"])
    G = c["n_q_heads"] // K.shape[1]
    mask = torch.as_tensor(np.arange(K.shape[0])[None, :] <= pos_q[:, None])
    qt = torch.as_tensor(q).permute(1, 0, 2)
    kt = torch.as_tensor(K).permute(1, 0, 2).repeat_interleave(G, dim=0)
    vt = torch.as_tensor(V).permute(1, 0, 2).repeat_interleave(G, dim=0)
    ref = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask).permute(1, 0, 2).numpy()
    o, _ = O.layout_forward(**c)
    np.testing.assert_allclose(o, ref, rtol=1e-10, atol=1e-12)


def test_layout_queries_do_not_see_later_artifacts():
    # queries in the first online span come before every artifact: replacing
    # the artifacts' K/V must not change them; queries after an artifact must change
    c = _layout_case(items=(-6, 1, -2, 0), S=16, S_kv=16)
    o1, _ = O.layout_forward(**c)
    rng = np.random.default_rng(99)
    c2 = dict(c)
    c2["art_k"] = {i: rng.standard_normal(t.shape) for i, t in c["art_k"].items()}
    c2["art_v"] = {i: rng.standard_normal(t.shape) for i, t in c["art_v"].items()}
    o2, _ = O.layout_forward(**c2)
    np.testing.assert_array_equal(o1[:6], o2[:6])
    assert np.abs(o1[6:] - o2[6:]).max() > 1e-3


def test_query_positions():
    # tiny workload: 201 artifact tokens, S = S_kv = 16 -> positions 201..216
    np.testing.assert_array_equal(O.query_positions(201, 16, 16), np.arange(201, 217))
    # decode: 128 prior suffix entries + the new token; the query is the last one
    np.testing.assert_array_equal(O.query_positions(1000, 1, 129), [1128])


# --------------------------------------------------------------------------
# Assembly / index map
# --------------------------------------------------------------------------
def test_assemble_hand_example():
    g = _golden("assemble_37_64_100.json")
    for c in g["cases"]:
        r = O.assemble(g["art_lengths"], c["request"], g["block_tokens"])
        np.testing.assert_array_equal(r["block_table"], c["block_table"])
        np.testing.assert_array_equal(r["valid_len"], c["valid_len"])
        T = sum(g["art_lengths"][a] for a in c["request"])
        np.testing.assert_array_equal(r["index_map"], _runs(c["index_map_runs"], T))
        np.testing.assert_array_equal(r["token_art"], _const_runs(c["token_art_runs"], T))


def test_assemble_brute_force_against_flat_storage():
    # the index map must point at the same bytes as a flat concatenation
    rng = np.random.default_rng(15)
    lengths = rng.integers(1, 200, size=9).tolist()
    r = O.assemble(lengths, [4, 0, 8, 4, 2])
    pool = np.full(r["total_blocks"] * 64, -1, dtype=np.int64)
    for a, L in enumerate(lengths):
        for p in range(L):
            pool[(r["first_block"][a] + p // 64) * 64 + p % 64] = a * 10000 + p
    flat = np.concatenate([a * 10000 + np.arange(lengths[a]) for a in [4, 0, 8, 4, 2]])
    np.testing.assert_array_equal(pool[r["index_map"]], flat)
    assert np.sum(r["valid_len"]) == len(flat)


# --------------------------------------------------------------------------
# Attention, Eq. (routing-oracle)
# --------------------------------------------------------------------------
def test_attention_hand_example():
    g = _golden("softmax_3keys.json")
    q = np.array(g["q"]).reshape(1, 1, 2)
    k = np.array([[math.sqrt(2.0) * math.log(i), 0.0] for i in g["k_from_log"]]).reshape(3, 1, 2)
    v = np.array(g["v"]).reshape(3, 1, 2)
    for c in g["cases"]:
        o, lse = O.attention(q, k, v, [c["n_visible"]])
        np.testing.assert_allclose(o.reshape(-1), c["o"], atol=1e-13)
        np.testing.assert_allclose(lse.reshape(-1), [c["lse"]], atol=1e-13)


def _sdpa_f64(q, k, v, n_visible):
    """fp64 SDPA on CPU with GQA expanded (kv head = q head // G) and a prefix mask."""
    S, Hq, d = q.shape
    T, Hkv, _ = k.shape
    G = Hq // Hkv
    qt = torch.from_numpy(q).permute(1, 0, 2)[None]
    kt = torch.from_numpy(k).repeat_interleave(G, dim=1).permute(1, 0, 2)[None]
    vt = torch.from_numpy(v).repeat_interleave(G, dim=1).permute(1, 0, 2)[None]
    mask = torch.from_numpy(np.arange(T)[None, :] < np.asarray(n_visible)[:, None])
    o = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, attn_mask=mask)
    return o[0].permute(1, 0, 2).numpy()


def test_attention_matches_sdpa_f64_gqa():
    rng = np.random.default_rng(16)
    S, Hq, Hkv, d, T = 9, 8, 2, 32, 70
    q = rng.standard_normal((S, Hq, d))
    k = rng.standard_normal((T, Hkv, d))
    v = rng.standard_normal((T, Hkv, d))
    n_vis = T - S + np.arange(S) + 1
    o, lse = O.attention(q, k, v, n_vis)
    np.testing.assert_allclose(o, _sdpa_f64(q, k, v, n_vis), atol=1e-12)
    # lse against an independent log-sum-exp of the scaled logits
    from scipy.special import logsumexp
    for i in (0, S - 1):
        for h in (0, 5):
            lg = k[:n_vis[i], h // 4] @ q[i, h] / math.sqrt(d)
            assert abs(lse[i, h] - logsumexp(lg)) < 1e-12
    # sampled pairs agree with the full evaluation
    pairs = [(0, 0), (3, 7), (8, 2)]
    op, lp = O.attention(q, k, v, n_vis, pairs)
    for p, (i, h) in enumerate(pairs):
        np.testing.assert_array_equal(op[p], o[i, h])
        assert lp[p] == lse[i, h]


def test_softmax_rows_sum_to_one_and_convex_hull():
    rng = np.random.default_rng(17)
    q = rng.standard_normal((4, 2, 8)) * 3
    k = rng.standard_normal((30, 1, 8))
    v = np.ones((30, 1, 8))
    n_vis = [5, 12, 29, 30]
    o, _ = O.attention(q, k, v, n_vis)
    np.testing.assert_allclose(o, 1.0, atol=1e-14)
    v = rng.standard_normal((30, 1, 8))
    o, _ = O.attention(q, k, v, n_vis)
    for i, n in enumerate(n_vis):
        lo = v[:n, 0].min(axis=0)
        hi = v[:n, 0].max(axis=0)
        assert np.all(o[i] >= lo[None] - 1e-12) and np.all(o[i] <= hi[None] + 1e-12)


def test_gqa_equals_mha_with_duplicated_heads():
    rng = np.random.default_rng(18)
    q = rng.standard_normal((5, 4, 16))
    k = rng.standard_normal((20, 2, 16))
    v = rng.standard_normal((20, 2, 16))
    n_vis = [16, 17, 18, 19, 20]
    o_gqa, l_gqa = O.attention(q, k, v, n_vis)
    k_mha = k[:, [0, 0, 1, 1]]
    v_mha = v[:, [0, 0, 1, 1]]
    o_mha, l_mha = O.attention(q, k_mha, v_mha, n_vis)
    np.testing.assert_array_equal(o_gqa, o_mha)
    np.testing.assert_array_equal(l_gqa, l_mha)


# --------------------------------------------------------------------------
# Split-KV combine: attention over a key set from attention over its parts
# --------------------------------------------------------------------------
def test_merge_hand_example():
    g = _golden("merge_two_parts.json")
    num = {"ln3": math.log(3.0), "ln4": math.log(4.0), "-inf": -np.inf}
    val = lambda x: num[x] if isinstance(x, str) else x
    for c in g["cases"]:
        o, lse = O.merge_partials([np.array(p) for p in c["o_parts"]], [np.array(val(l)) for l in c["lse_parts"]])
        np.testing.assert_allclose(o, c["o"], atol=1e-15)
        assert abs(lse - val(c["lse"])) < 1e-15


def _part_attention(q, k, v, n_vis, a, b):
    """Attention of every query over keys [a, b) it can see; o = 0, lse = -inf where it sees none."""
    S, Hq, d = q.shape
    cnt = np.clip(np.asarray(n_vis) - a, 0, b - a)
    o, lse = np.zeros((S, Hq, d)), np.full((S, Hq), -np.inf)
    rows = np.nonzero(cnt > 0)[0]
    if len(rows):
        o_r, l_r = O.attention(q[rows], k[a:b], v[a:b], cnt[rows])
        o[rows], lse[rows] = o_r, l_r
    return o, lse


def test_merge_of_parts_equals_attention_over_all_keys():
    rng = np.random.default_rng(23)
    S, Hq, Hkv, d, T = 7, 4, 2, 16, 90
    q = rng.standard_normal((S, Hq, d)) * 2
    k = rng.standard_normal((T, Hkv, d))
    v = rng.standard_normal((T, Hkv, d))
    n_vis = T - S + np.arange(S) + 1                       # causal tail: later parts are ragged
    o_full, lse_full = O.attention(q, k, v, n_vis)
    for cuts in ([45], [10, 64], [1, 2, 89], [30, 60, 84, 88]):
        edges = [0] + cuts + [T]
        parts = [_part_attention(q, k, v, n_vis, a, b) for a, b in zip(edges[:-1], edges[1:])]
        o, lse = O.merge_partials([p[0] for p in parts], [p[1] for p in parts])
        np.testing.assert_allclose(o, o_full, atol=1e-12)
        np.testing.assert_allclose(lse, lse_full, atol=1e-12)
        # the order of the parts does not matter
        o_r, lse_r = O.merge_partials([p[0] for p in parts[::-1]], [p[1] for p in parts[::-1]])
        np.testing.assert_allclose(o_r, o_full, atol=1e-12)
    # one part is the identity
    o1, l1 = O.merge_partials([o_full], [lse_full])
    np.testing.assert_allclose(o1, o_full, atol=1e-15)
    np.testing.assert_allclose(l1, lse_full, atol=1e-15)


# --------------------------------------------------------------------------
# End-to-end properties of one request
# --------------------------------------------------------------------------
def _small_inputs(rng, hidden=32, hq=4, hkv=2, d=16, r=4):
    return dict(
        w_q=rng.standard_normal((hq * d, hidden)) / math.sqrt(hidden),
        a=rng.standard_normal((r, hidden)) / math.sqrt(hidden),
        b=rng.standard_normal((hq * d, r)) / math.sqrt(r),
        qn=1.0 + 0.1 * rng.standard_normal(d))


def test_single_artifact_equals_full_causal():
    # Eq. (full-vs-pic) with m = 1 and an empty prefix: the cached artifact is
    # the full prefill of its own tokens, so the suffix rows equal causal
    # attention over the whole L + S sequence.
    rng = np.random.default_rng(19)
    hidden, hq, hkv, d, theta, eps, s = 32, 4, 2, 16, 1.0e4, 1e-6, 2.0
    L, S = 50, 7
    w = _small_inputs(rng, hidden, hq, hkv, d)
    k_raw = rng.standard_normal((L + S, hkv, d))
    v = rng.standard_normal((L + S, hkv, d))
    k_rot = O.rope_rotate_half(k_raw, np.arange(L + S), theta)   # global positions 0..L+S-1
    x = rng.standard_normal((S, hidden))
    o, lse = O.request_forward(x, w["w_q"], w["a"], w["b"], s, w["qn"], eps, theta,
                               [k_rot[:L]], [v[:L]], k_rot[L:], v[L:], hq)
    # Full side: queries built step by step at positions L..L+S-1, random
    # queries for the artifact tokens, plain causal SDPA over L + S tokens.
    q_raw = O.lora_q_projection(x, w["w_q"], w["a"], w["b"], s).reshape(S, hq, d)
    q_suf = O.rope_rotate_half(O.rms_norm_heads(q_raw, w["qn"], eps), np.arange(L, L + S), theta)
    q_full = np.concatenate([rng.standard_normal((L, hq, d)), q_suf], axis=0)
    qt = torch.from_numpy(q_full).permute(1, 0, 2)[None]
    kt = torch.from_numpy(k_rot).repeat_interleave(hq // hkv, dim=1).permute(1, 0, 2)[None]
    vt = torch.from_numpy(v).repeat_interleave(hq // hkv, dim=1).permute(1, 0, 2)[None]
    full = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)[0].permute(1, 0, 2).numpy()
    np.testing.assert_allclose(o, full[L:], atol=1e-12)


def test_artifact_order_invariance():
    # keys are pre-rotated at local positions and every artifact token is
    # visible to every suffix query, so the output is a softmax over a set.
    rng = np.random.default_rng(20)
    hidden, hq, hkv, d = 32, 4, 2, 16
    w = _small_inputs(rng, hidden, hq, hkv, d)
    lens = [13, 64, 40]
    ak = [rng.standard_normal((L, hkv, d)) for L in lens]
    av = [rng.standard_normal((L, hkv, d)) for L in lens]
    x = rng.standard_normal((6, hidden))
    sk = rng.standard_normal((9, hkv, d))
    sv = rng.standard_normal((9, hkv, d))
    args = (x, w["w_q"], w["a"], w["b"], 2.0, w["qn"], 1e-6, 1e6)
    o0, l0 = O.request_forward(*args, ak, av, sk, sv, hq)
    for perm in ([2, 0, 1], [1, 2, 0], [2, 1, 0]):
        o1, l1 = O.request_forward(*args, [ak[i] for i in perm], [av[i] for i in perm], sk, sv, hq)
        np.testing.assert_allclose(o1, o0, atol=1e-12)
        np.testing.assert_allclose(l1, l0, atol=1e-12)


def test_tiny_workload_against_sdpa():
    # the tiny parity workload, end to end, against fp64 SDPA
    from gen import make_workload
    wl = make_workload("tiny")
    o, lse = O.workload_reference(wl, 0)
    q = O.workload_reference(wl, 0, q_only=True)
    f = O.bf16_to_f64
    k = np.concatenate([f(t) for t in wl.art_k] + [f(wl.suffix_k[0])])
    v = np.concatenate([f(t) for t in wl.art_v] + [f(wl.suffix_v[0])])
    n_vis = 201 + np.arange(16) + 1
    np.testing.assert_allclose(o, _sdpa_f64(q, k, v, n_vis), atol=1e-12)
    assert o.shape == (16, 4, 64) and np.all(np.isfinite(lse))


# --------------------------------------------------------------------------
# App. C.2, EPIC paragraph: keys stored before RoPE, rotated to their
# assembled positions at assembly
# --------------------------------------------------------------------------
def _variant_case(rng, lens=(13, 64, 40), S=6, S_kv=9, hidden=32, hq=4, hkv=2, d=16, theta=1.0e4):
    w = _small_inputs(rng, hidden, hq, hkv, d)
    return dict(
        x=rng.standard_normal((S, hidden)), w_q=w["w_q"], a=w["a"], b=w["b"], s=2.0, q_norm_w=w["qn"], eps=1e-6,
        theta=theta, art_k=[rng.standard_normal((L, hkv, d)) for L in lens],
        art_v=[rng.standard_normal((L, hkv, d)) for L in lens], suffix_k=rng.standard_normal((S_kv, hkv, d)),
        suffix_v=rng.standard_normal((S_kv, hkv, d)), n_q_heads=hq)


def _queries(c):
    # the queries of request_forward, step by step through the pinned functions
    S, S_kv, d = c["x"].shape[0], c["suffix_k"].shape[0], c["suffix_k"].shape[2]
    t_art = sum(k.shape[0] for k in c["art_k"])
    q_raw = O.lora_q_projection(c["x"], c["w_q"], c["a"], c["b"], c["s"]).reshape(S, c["n_q_heads"], d)
    pos = t_art + (S_kv - S) + np.arange(S)
    return O.rope_rotate_half(O.rms_norm_heads(q_raw, c["q_norm_w"], c["eps"]), pos, c["theta"]), pos


def _epic(c, **kw):
    return O.epic_request_forward(c["x"], c["w_q"], c["a"], c["b"], c["s"], c["q_norm_w"], c["eps"], c["theta"],
                                  c["art_k"], c["art_v"], c["suffix_k"], c["suffix_v"], c["n_q_heads"], **kw)


def test_epic_equals_full_causal_over_the_assembled_sequence():
    # With the artifacts' raw keys rotated at their assembled positions, the
    # suffix rows read exactly the keys a full prefill of the concatenation
    # would hold: fp64 causal SDPA over the whole sequence, keys rotated at
    # 0..T-1, in two runtime orders
    rng = np.random.default_rng(31)
    c = _variant_case(rng)
    for order in ([0, 1, 2], [2, 0, 1]):
        cc = dict(c, art_k=[c["art_k"][i] for i in order], art_v=[c["art_v"][i] for i in order])
        S = cc["x"].shape[0]
        q, _ = _queries(cc)
        k_raw = np.concatenate(cc["art_k"])
        T_art = k_raw.shape[0]
        K = np.concatenate([O.rope_rotate_half(k_raw, np.arange(T_art), cc["theta"]), cc["suffix_k"]])
        V = np.concatenate(cc["art_v"] + [cc["suffix_v"]])
        T = K.shape[0]
        q_full = np.concatenate([rng.standard_normal((T - S, cc["n_q_heads"], q.shape[2])), q])
        G = cc["n_q_heads"] // K.shape[1]
        qt = torch.from_numpy(q_full).permute(1, 0, 2)[None]
        kt = torch.from_numpy(K).repeat_interleave(G, dim=1).permute(1, 0, 2)[None]
        vt = torch.from_numpy(V).repeat_interleave(G, dim=1).permute(1, 0, 2)[None]
        full = torch.nn.functional.scaled_dot_product_attention(qt, kt, vt, is_causal=True)[0].permute(1, 0, 2)
        o, _ = _epic(cc)
        np.testing.assert_allclose(o, full.numpy()[T - S:], atol=1e-12)


def test_epic_relative_position_identity():
    # <R(p) q, R(t + off_a) k> = <R(p - off_a) q, R(t) k>: the keys rotated at
    # their assembled positions give the same logits as the PIC cache (keys
    # at local positions t) read by queries rotated back by each artifact's
    # offset.  Direct sums over that second form, query by query.
    rng = np.random.default_rng(32)
    c = _variant_case(rng, lens=(5, 11, 3), S=3, S_kv=4, hq=2, hkv=1, d=8)
    o, lse = _epic(c)
    S, S_kv, d = c["x"].shape[0], c["suffix_k"].shape[0], 8
    t_art = sum(k.shape[0] for k in c["art_k"])
    q_raw = O.lora_q_projection(c["x"], c["w_q"], c["a"], c["b"], c["s"]).reshape(S, 2, d)
    qn = O.rms_norm_heads(q_raw, c["q_norm_w"], c["eps"])
    for i in range(S):
        p = t_art + (S_kv - S) + i
        for h in range(2):
            logits, vals = [], []
            off = 0
            for ka, va in zip(c["art_k"], c["art_v"]):
                q_back = O.rope_rotate_half(qn[i:i + 1, h:h + 1], np.array([p - off]), c["theta"])[0, 0]
                k_loc = O.rope_rotate_half(ka[:, 0:1], np.arange(ka.shape[0]), c["theta"])[:, 0]
                for t in range(ka.shape[0]):
                    logits.append(float(q_back @ k_loc[t]) / math.sqrt(d))
                    vals.append(va[t, 0])
                off += ka.shape[0]
            q_here = O.rope_rotate_half(qn[i:i + 1, h:h + 1], np.array([p]), c["theta"])[0, 0]
            for j in range(S_kv - S + i + 1):
                logits.append(float(q_here @ c["suffix_k"][j, 0]) / math.sqrt(d))
                vals.append(c["suffix_v"][j, 0])
            e = [math.exp(z) for z in logits]
            z = sum(e)
            ref = sum(w * v for w, v in zip(e, vals)) / z
            np.testing.assert_allclose(o[i, h], ref, atol=1e-12)
            assert abs(lse[i, h] - math.log(z)) < 1e-12


def test_epic_single_artifact_is_the_pic_read():
    # the first artifact starts at position 0: rotating its raw keys at
    # assembly equals caching them rotated at their local positions
    rng = np.random.default_rng(33)
    c = _variant_case(rng, lens=(70,))
    o, lse = _epic(c)
    k_loc = O.rope_rotate_half(c["art_k"][0], np.arange(70), c["theta"])
    o2, lse2 = O.request_forward(c["x"], c["w_q"], c["a"], c["b"], c["s"], c["q_norm_w"], c["eps"], c["theta"],
                                 [k_loc], c["art_v"], c["suffix_k"], c["suffix_v"], c["n_q_heads"])
    np.testing.assert_allclose(o, o2, atol=1e-13)
    np.testing.assert_allclose(lse, lse2, atol=1e-13)


def test_epic_without_artifacts_is_causal_attention_over_the_suffix():
    # nothing to rotate: the suffix rows of plain causal attention, against
    # fp64 SDPA with the queries at positions (S_kv - S) + i
    rng = np.random.default_rng(37)
    c = _variant_case(rng, lens=())
    o, _ = _epic(c)
    q, _ = _queries(c)
    S, S_kv = c["x"].shape[0], c["suffix_k"].shape[0]
    np.testing.assert_allclose(o, _sdpa_f64(q, c["suffix_k"], c["suffix_v"], (S_kv - S) + np.arange(S) + 1),
                               atol=1e-12)


def test_rotate_at_assembly_positions():
    # token t of the concatenation is rotated at t: a unit vector in pair 0
    # turns by t * theta^0 = t radians
    k = [np.zeros((2, 1, 4)), np.zeros((3, 1, 4))]
    for a in k:
        a[:, 0, 0] = 1.0
    out = O.rotate_at_assembly(k, 1.0e4)
    for t in range(5):
        np.testing.assert_allclose(out[t, 0, [0, 2]], [math.cos(t), math.sin(t)], atol=1e-15)


# --------------------------------------------------------------------------
# App. C.2, APE paragraph: context (temperature T) and online attention
# combined through calibrated log-sum-exp terms
# --------------------------------------------------------------------------
def _ape(c, T, scale, **kw):
    return O.ape_request_forward(c["x"], c["w_q"], c["a"], c["b"], c["s"], c["q_norm_w"], c["eps"], c["theta"],
                                 c["art_k"], c["art_v"], c["suffix_k"], c["suffix_v"], c["n_q_heads"], T, scale, **kw)


def test_ape_combine_hand_example():
    g = _golden("ape_combine.json")
    num = {"ln3": math.log(3.0), "ln4": math.log(4.0), "ln5": math.log(5.0), "ln8": math.log(8.0),
           "ln16": math.log(16.0), "-inf": -np.inf}
    val = lambda x: num[x] if isinstance(x, str) else x
    for cs in g["cases"]:
        o, lse = O.ape_combine(np.array(cs["o_ctx"]), np.array(val(cs["lse_ctx"])), np.array(cs["o_on"]),
                               np.array(val(cs["lse_on"])), cs["scale"])
        np.testing.assert_allclose(o, cs["o"], atol=1e-14)
        assert abs(lse - val(cs["lse"])) < 1e-14


def test_ape_with_unit_temperature_and_scale_is_the_pic_read():
    rng = np.random.default_rng(34)
    c = _variant_case(rng)
    o, lse = _ape(c, 1.0, 1.0)
    o2, lse2 = O.request_forward(c["x"], c["w_q"], c["a"], c["b"], c["s"], c["q_norm_w"], c["eps"], c["theta"],
                                 c["art_k"], c["art_v"], c["suffix_k"], c["suffix_v"], c["n_q_heads"])
    np.testing.assert_allclose(o, o2, atol=1e-12)
    np.testing.assert_allclose(lse, lse2, atol=1e-12)


@pytest.mark.parametrize("T,scale", [(0.9, 0.9), (0.5, 1.3)])
def test_ape_against_direct_sums(T, scale):
    # no max subtraction and no log-sum-exp machinery: Z_c = sum over context
    # keys of exp(l / T), Z_o = sum over visible online keys of exp(l), and
    # o = (Z_c^(scale - 1) N_c + N_o) / (Z_c^scale + Z_o) with N the
    # exp-weighted value sums; lse = log(Z_c^scale + Z_o)
    rng = np.random.default_rng(35)
    c = _variant_case(rng, lens=(7, 4), S=3, S_kv=5, hq=2, hkv=1, d=8)
    o, lse = _ape(c, T, scale)
    q, _ = _queries(c)
    S, S_kv, d = 3, 5, 8
    k_art, v_art = np.concatenate(c["art_k"]), np.concatenate(c["art_v"])
    for i in range(S):
        for h in range(2):
            zc, nc = 0.0, np.zeros(d)
            for t in range(k_art.shape[0]):
                e = math.exp(float(q[i, h] @ k_art[t, 0]) / math.sqrt(d) / T)
                zc += e
                nc += e * v_art[t, 0]
            zo, no = 0.0, np.zeros(d)
            for j in range(S_kv - S + i + 1):
                e = math.exp(float(q[i, h] @ c["suffix_k"][j, 0]) / math.sqrt(d))
                zo += e
                no += e * c["suffix_v"][j, 0]
            ref = (zc ** (scale - 1.0) * nc + no) / (zc ** scale + zo)
            np.testing.assert_allclose(o[i, h], ref, rtol=1e-11, atol=1e-13)
            assert abs(lse[i, h] - math.log(zc ** scale + zo)) < 1e-11


def test_ape_without_artifacts_is_online_attention():
    rng = np.random.default_rng(36)
    c = _variant_case(rng, lens=())
    o, lse = _ape(c, 0.9, 0.9)
    q, _ = _queries(c)
    S, S_kv = c["x"].shape[0], c["suffix_k"].shape[0]
    o2, lse2 = O.attention(q, c["suffix_k"], c["suffix_v"], (S_kv - S) + np.arange(S) + 1)
    np.testing.assert_allclose(o, o2, atol=1e-14)
    np.testing.assert_allclose(lse, lse2, atol=1e-14)
