"""The seeded input generator against the recipe it states.

Both sides of every parity check draw from gen/, so its layouts and value
distributions are pinned here: each named workload has the shapes and lengths
its configuration gives, a seed reproduces every tensor bit for bit, and the
drawn values follow the stated distributions (K, V, x ~ N(0, 1); W_q, A ~
N(0, 1/hidden); B ~ N(0, 1/r); q_norm weight 1 + 0.1 N(0, 1)).
"""
from __future__ import annotations

import numpy as np
import pytest
import torch

from gen import WORKLOADS, Geometry, layout, make_custom, make_kv_weights, make_workload


def test_layouts_of_the_named_workloads():
    g, seed, lengths, reqs, S, S_kv = layout("tiny")
    assert (g.hidden, g.n_q_heads, g.n_kv_heads, g.head_dim, g.rank) == (256, 4, 2, 64, 8)
    assert (seed, lengths, reqs, S, S_kv) == (0, [37, 64, 100], [[0, 1, 2]], 16, 16)

    g, seed, lengths, reqs, S, S_kv = layout("qwen3_4b_prefill")
    assert (g.hidden, g.n_q_heads, g.n_kv_heads, g.head_dim, g.rank) == (2560, 32, 8, 128, 16)
    assert len(lengths) == 8 and all(512 <= L <= 2048 for L in lengths)
    assert reqs == [list(range(8))] and S == S_kv == 256

    g, seed, lengths, reqs, S, S_kv = layout("qwen3_8b_prefill_4req")
    assert (g.hidden, g.n_q_heads, g.n_kv_heads, g.head_dim, g.rank) == (4096, 32, 8, 128, 16)
    assert len(lengths) == 64 and all(1024 <= L <= 4096 for L in lengths)
    assert len(reqs) == 4 and all(len(r) == 16 and len(set(r)) == 16 for r in reqs) and S == S_kv == 512

    g, seed, lengths, reqs, S, S_kv = layout("qwen3_8b_decode_64req")
    assert len(lengths) == 256 and all(256 <= L <= 2048 for L in lengths)
    assert len(reqs) == 64 and all(4 <= len(r) <= 12 and len(set(r)) == len(r) for r in reqs)
    assert (S, S_kv) == (1, 129)

    g, seed, lengths, reqs, S, S_kv = layout("qwen3_8b_long_131k")
    assert lengths == [2048] * 64 and reqs == [list(range(64))] and S == S_kv == 2048
    assert sum(lengths) == 131072

    assert [layout(n)[1] for n in WORKLOADS] == [0, 1, 2, 3, 4]      # one seed per workload


def test_a_seed_reproduces_every_tensor():
    a, b = make_workload("tiny"), make_workload("tiny")
    for name in ("x", "w_q", "lora_a", "lora_b", "q_norm_w", "suffix_k", "suffix_v"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name
    assert all(torch.equal(p, q) for p, q in zip(a.art_k + a.art_v, b.art_k + b.art_v))
    g = Geometry(hidden=128, n_q_heads=4, n_kv_heads=2, head_dim=64, rank=8)
    c = make_custom("c", g, 5, [10, 20], [[1, 0]], 3, 4)
    d = make_custom("c", g, 6, [10, 20], [[1, 0]], 3, 4)
    assert not torch.equal(c.x, d.x)                                   # another seed, other values


def test_values_follow_the_stated_distributions():
    g = Geometry(hidden=1024, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)
    wl = make_custom("stats", g, 9, [700, 900], [[0, 1]], 64, 64)
    f = lambda t: t.double().numpy().ravel()

    def check(t, std, what):
        v = f(t)
        assert abs(v.mean()) < 4 * std / np.sqrt(v.size) + 1e-3 * std, what
        assert abs(v.std() / std - 1.0) < 0.02, (what, v.std(), std)

    check(torch.cat([k.reshape(-1) for k in wl.art_k]), 1.0, "artifact K")
    check(torch.cat([v.reshape(-1) for v in wl.art_v]), 1.0, "artifact V")
    check(wl.x, 1.0, "x")
    check(wl.suffix_k, 1.0, "suffix K")
    check(wl.w_q, 1024 ** -0.5, "W_q")
    check(wl.lora_a, 1024 ** -0.5, "A")
    check(wl.lora_b, 16 ** -0.5, "B")
    qn = f(wl.q_norm_w)
    assert abs(qn.mean() - 1.0) < 0.05 and 0.06 < qn.std() < 0.14
    w_k, w_v, kn = make_kv_weights(g, 0)
    check(w_k, 1024 ** -0.5, "W_k")
    check(w_v, 1024 ** -0.5, "W_v")
    assert w_k.shape == (4 * 128, 1024) and kn.shape == (128,)


def test_shapes_of_a_custom_workload():
    g = Geometry(hidden=128, n_q_heads=8, n_kv_heads=2, head_dim=64, rank=8)
    wl = make_custom("shapes", g, 1, [5, 70, 64], [[2, 0], [], [1]], 3, 7)
    assert [tuple(t.shape) for t in wl.art_k] == [(5, 2, 64), (70, 2, 64), (64, 2, 64)]
    assert tuple(wl.x.shape) == (3, 3, 128) and tuple(wl.suffix_k.shape) == (3, 7, 2, 64)
    assert tuple(wl.w_q.shape) == (512, 128) and tuple(wl.lora_a.shape) == (8, 128)
    assert tuple(wl.lora_b.shape) == (512, 8)
    assert [wl.t_art(r) for r in range(3)] == [69, 0, 70]
    assert all(t.dtype == torch.bfloat16 for t in [wl.x, wl.w_q, wl.q_norm_w, wl.suffix_v] + wl.art_v)
    merged = make_custom("merged", g, 1, [5], [[0]], 2, 2, with_lora=False)
    assert merged.lora_a is None and merged.lora_b is None
    with pytest.raises(AssertionError):
        make_custom("bad", g, 1, [5], [[0]], 4, 3)                     # S_kv < S
