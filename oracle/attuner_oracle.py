"""Plain float64 definitions of the artifact-KV read path (test infrastructure).

Only tests, the smoke check and the benchmark's CPU-baseline leg use this
module.  It is deliberately slow and literal: no blocking, no fusion, no
reordering beyond what each definition states.

Notation follows the paper: h (here x) is the projection input, W^Q the base
query projection, A in R^{r x d_model}, B in R^{d_q x r}, s = alpha / r.
"""

from __future__ import annotations

import math
from typing import Iterable, List, Optional, Sequence, Tuple

import numpy as np


def bf16_to_f64(t) -> np.ndarray:
    """Exact widening of a bf16 tensor (torch, any device) to float64 numpy."""
    import torch  # local: the oracle itself is numpy-only
    if isinstance(t, np.ndarray):
        return t.astype(np.float64)
    return t.detach().to("cpu").to(torch.float64).numpy()


# ---------------------------------------------------------------------------
# Sec. 3, Eq. (query-adaptation): q~ = W^Q h + (alpha/r) B A h
# ---------------------------------------------------------------------------
def lora_q_projection(x: np.ndarray, w_q: np.ndarray, a: Optional[np.ndarray],
                      b: Optional[np.ndarray], s: float) -> np.ndarray:
    """Unmerged adapted query projection, one row per token.

    x [M, d_model], w_q [d_q, d_model] (output x input), a [r, d_model],
    b [d_q, r].  Returns q_raw [M, d_q] = x W^T + s * (x A^T) B^T.
    a = b = None (or r = 0) is the merged / base path.
    """
    base = x @ w_q.T
    if a is None or b is None or a.shape[0] == 0:
        return base
    down = x @ a.T            # A h        [M, r]
    up = down @ b.T           # B (A h)    [M, d_q]
    return base + s * up


def merged_q_weight(w_q: np.ndarray, a: np.ndarray, b: np.ndarray, s: float) -> np.ndarray:
    """App. A.5 (Deployment): W^Q <- W^Q + (alpha/r) B A."""
    return w_q + s * (b @ a)


# ---------------------------------------------------------------------------
# Sec. 3 (after Eq. query-adaptation): the model's original query
# normalisation (Qwen3 per-head RMSNorm over head_dim), then RoPE.
# ---------------------------------------------------------------------------
def rms_norm_heads(q: np.ndarray, w: np.ndarray, eps: float) -> np.ndarray:
    """q [M, H, d] -> q / sqrt(mean_j q_j^2 + eps) * w, per (token, head)."""
    ms = np.mean(q * q, axis=-1, keepdims=True)
    return q / np.sqrt(ms + eps) * w


def rope_rotate_half(q: np.ndarray, pos: np.ndarray, theta: float) -> np.ndarray:
    """Rotary embedding, rotate-half pairing.

    Element j < d/2 is paired with j + d/2 and the pair is rotated by the angle
    pos * theta^(-2j/d).  q [M, H, d], pos [M] (integer positions).
    """
    d = q.shape[-1]
    half = d // 2
    j = np.arange(half, dtype=np.float64)
    inv_freq = theta ** (-2.0 * j / d)                     # [d/2]
    ang = np.asarray(pos, dtype=np.float64)[:, None] * inv_freq[None, :]   # [M, d/2]
    c = np.cos(ang)[:, None, :]
    sn = np.sin(ang)[:, None, :]
    x1 = q[..., :half]
    x2 = q[..., half:]
    out = np.empty_like(q)
    out[..., :half] = x1 * c - x2 * sn
    out[..., half:] = x2 * c + x1 * sn
    return out


def query_positions(t_art: int, S: int, S_kv: int) -> np.ndarray:
    """App. A.5: position ids of the assembled context.

    Artifacts occupy assembled positions 0..T_art-1; the suffix KV occupies
    T_art..T_art+S_kv-1 and the S query tokens are its last S entries.
    """
    return t_art + (S_kv - S) + np.arange(S, dtype=np.int64)


# ---------------------------------------------------------------------------
# Online K/V of the suffix tokens.  The adaptation changes W^Q only (Sec. 3:
# the keys and values keep the base model's projections, which is what keeps
# the cached artifact KV valid); the base model normalises each key head
# (Qwen3 k_norm) and rotates it at the token's assembled position (App. A.5).
# ---------------------------------------------------------------------------
def kv_projection(x: np.ndarray, w_k: np.ndarray, w_v: np.ndarray, k_norm_w: np.ndarray, eps: float,
                  theta: float, positions: np.ndarray, n_kv_heads: int) -> Tuple[np.ndarray, np.ndarray]:
    """x [S_new, d_model]; w_k, w_v [Hkv*d, d_model]; k_norm_w [d]; positions [S_new].

    K [S_new, Hkv, d] = RoPE(RMSNorm(x W_k^T per head) * w, pos);  V = x W_v^T.
    """
    d = w_k.shape[0] // n_kv_heads
    k = rms_norm_heads((x @ w_k.T).reshape(-1, n_kv_heads, d), k_norm_w, eps)
    k = rope_rotate_half(k, positions, theta)
    v = (x @ w_v.T).reshape(-1, n_kv_heads, d)
    return k, v


# ---------------------------------------------------------------------------
# Sec. 2 (PIC box, Eq. full-vs-pic) and App. A.3 "Cache construction and
# reuse": cached blocks are assembled in prompt order without re-encoding.
# Paging in 64-token blocks is this library's storage, not the paper's.
# ---------------------------------------------------------------------------
def assemble(art_lengths: Sequence[int], request: Sequence[int], block_tokens: int = 64) -> dict:
    """Block table and index map of one request.

    Storage rule (bump allocation in registration order): artifact j owns the
    consecutive block ids starting at sum_{i<j} ceil(L_i / block_tokens);
    local token p of artifact j lives in block first_j + p // block_tokens,
    slot p % block_tokens.

    Returns block_table, valid_len (per block of the request, runtime order),
    index_map[t] = block * block_tokens + slot for assembled token t,
    token_art[t], token_off[t] (artifact id and local offset of token t).
    """
    first = []
    nxt = 0
    for L in art_lengths:
        first.append(nxt)
        nxt += -(-int(L) // block_tokens)
    block_table: List[int] = []
    valid_len: List[int] = []
    index_map: List[int] = []
    token_art: List[int] = []
    token_off: List[int] = []
    for a in request:
        L = int(art_lengths[a])
        nb = -(-L // block_tokens)
        for bi in range(nb):
            block_table.append(first[a] + bi)
            valid_len.append(min(block_tokens, L - bi * block_tokens))
        for p in range(L):
            index_map.append((first[a] + p // block_tokens) * block_tokens + p % block_tokens)
            token_art.append(a)
            token_off.append(p)
    i32 = lambda v: np.asarray(v, dtype=np.int32)
    return dict(block_table=i32(block_table), valid_len=i32(valid_len), index_map=i32(index_map),
                token_art=i32(token_art), token_off=i32(token_off), first_block=i32(first),
                total_blocks=nxt)


# ---------------------------------------------------------------------------
# Sec. 2.2, Eq. (routing-oracle): softmax(q K^T / sqrt(d_k) + M_t) V
# ---------------------------------------------------------------------------
def attention(q: np.ndarray, k: np.ndarray, v: np.ndarray, n_visible: Sequence[int],
              pairs: Optional[Iterable[Tuple[int, int]]] = None):
    """Grouped-query attention with a prefix-visibility mask.

    q [S, Hq, d]; k, v [T, Hkv, d]; query head h reads KV head h // (Hq/Hkv).
    Query i sees keys 0..n_visible[i]-1 (M_t = 0 there, -inf elsewhere).
    Returns (o [S, Hq, d], lse [S, Hq]) or, with pairs = [(i, h), ...],
    (o [P, d], lse [P]).  lse is the natural log of the softmax denominator
    of the scaled logits.
    """
    S, Hq, d = q.shape
    Hkv = k.shape[1]
    G = Hq // Hkv
    scale = 1.0 / math.sqrt(d)

    # one contiguous [T, d] copy per KV head, so each query row reads a prefix
    k_heads = [np.ascontiguousarray(k[:, j, :]) for j in range(Hkv)]
    v_heads = [np.ascontiguousarray(v[:, j, :]) for j in range(Hkv)]

    def one(i, h):
        n = int(n_visible[i])
        kh = k_heads[h // G][:n]
        vh = v_heads[h // G][:n]
        logits = (kh @ q[i, h, :]) * scale
        m = np.max(logits)
        e = np.exp(logits - m)
        z = np.sum(e)
        return (e / z) @ vh, m + math.log(z)

    if pairs is None:
        o = np.zeros((S, Hq, d))
        lse = np.zeros((S, Hq))
        for i in range(S):
            for h in range(Hq):
                o[i, h], lse[i, h] = one(i, h)
        return o, lse
    pairs = list(pairs)
    o = np.zeros((len(pairs), d))
    lse = np.zeros(len(pairs))
    for p, (i, h) in enumerate(pairs):
        o[p], lse[p] = one(i, h)
    return o, lse


# ---------------------------------------------------------------------------
# Split-KV combine (an implementation step, not the paper's): attention over a
# key set is the softmax-weighted combination of attention over its parts.
# With o_i, lse_i the output and log-denominator of part i,
#   lse = log sum_i exp(lse_i),   o = sum_i exp(lse_i - lse) o_i.
# A part with no visible key has lse_i = -inf and weight 0.
# ---------------------------------------------------------------------------
def merge_partials(o_parts: Sequence[np.ndarray], lse_parts: Sequence[np.ndarray]):
    """o_parts: P arrays [..., d]; lse_parts: P arrays [...] (-inf for an empty
    part).  Returns (o [..., d], lse [...])."""
    lse_stack = np.stack([np.asarray(l, dtype=np.float64) for l in lse_parts])      # [P, ...]
    m = np.max(lse_stack, axis=0)
    w = np.exp(lse_stack - m)                                                       # [P, ...]
    z = np.sum(w, axis=0)
    o = sum(w[i][..., None] * np.asarray(o_parts[i], dtype=np.float64) for i in range(len(o_parts))) / z[..., None]
    return o, m + np.log(z)


# ---------------------------------------------------------------------------
# One request end to end: adapted Q -> q_norm -> RoPE -> attention over the
# assembled artifact KV followed by the suffix's own KV.
# ---------------------------------------------------------------------------
def request_forward(x, w_q, a, b, s, q_norm_w, eps, theta, art_k: List[np.ndarray],
                    art_v: List[np.ndarray], suffix_k, suffix_v, n_q_heads: int,
                    pairs=None, q_only: bool = False):
    """x [S, d_model]; art_k/art_v: per-artifact [L, Hkv, d] in runtime order;
    suffix_k/suffix_v [S_kv, Hkv, d].  All float64.

    Suffix query i sits at position T_art + (S_kv - S) + i and sees every
    artifact token plus suffix keys j <= (S_kv - S) + i.
    """
    S = x.shape[0]
    S_kv = suffix_k.shape[0]
    d = suffix_k.shape[2]
    t_art = int(sum(t.shape[0] for t in art_k))
    q_raw = lora_q_projection(x, w_q, a, b, s).reshape(S, n_q_heads, d)
    q_n = rms_norm_heads(q_raw, q_norm_w, eps)
    q = rope_rotate_half(q_n, query_positions(t_art, S, S_kv), theta)
    if q_only:
        return q
    k_all = np.concatenate(list(art_k) + [suffix_k], axis=0)
    v_all = np.concatenate(list(art_v) + [suffix_v], axis=0)
    n_visible = t_art + (S_kv - S) + np.arange(S) + 1
    return attention(q, k_all, v_all, n_visible, pairs)


# ---------------------------------------------------------------------------
# App. C.2 "Training-Free Baselines", EPIC paragraph: the cached keys are
# stored before RoPE and rotated to their target positions when the request
# is assembled.  Here the target of artifact token t is its index in the
# assembled sequence (artifacts in runtime order from position 0, App. A.5),
# and the read that follows is the PIC read of Eq. (routing-oracle) over the
# rotated keys: every artifact token visible, the suffix causal.
# ---------------------------------------------------------------------------
def rotate_at_assembly(art_k_raw: Sequence[np.ndarray], theta: float) -> np.ndarray:
    """art_k_raw: per-artifact keys before RoPE [L_a, Hkv, d], runtime order.
    Returns the assembled keys [T_art, Hkv, d], token t rotated at position t."""
    k = np.concatenate(list(art_k_raw), axis=0)
    return rope_rotate_half(k, np.arange(k.shape[0], dtype=np.int64), theta)


def epic_request_forward(x, w_q, a, b, s, q_norm_w, eps, theta, art_k_raw: List[np.ndarray],
                         art_v: List[np.ndarray], suffix_k, suffix_v, n_q_heads: int, pairs=None):
    """request_forward with the artifact keys stored before RoPE and rotated
    at their assembled positions; queries and suffix keys as there.  An empty
    artifact list leaves nothing to rotate: the plain read of the suffix."""
    if len(art_k_raw) == 0:
        return request_forward(x, w_q, a, b, s, q_norm_w, eps, theta, [], [], suffix_k, suffix_v, n_q_heads,
                               pairs=pairs)
    k_art = rotate_at_assembly(art_k_raw, theta)
    v_art = np.concatenate(list(art_v), axis=0)
    return request_forward(x, w_q, a, b, s, q_norm_w, eps, theta, [k_art], [v_art], suffix_k, suffix_v,
                           n_q_heads, pairs=pairs)


# ---------------------------------------------------------------------------
# App. C.2, APE paragraph: attention over the cached context and over the
# online tokens is computed separately, the context's logits divided by a
# temperature T, and the two results are combined through calibrated
# log-sum-exp terms.  The paper fixes T = 0.9 and a scale of 0.9 but not how
# the scale enters; the reading taken here multiplies the context's
# log-sum-exp by it (its softmax denominator Z_c counts as Z_c^scale).
# With no prefix of online text before the artifacts (a prompt that begins
# with cached artifacts), the online part is the suffix, causal.
# ---------------------------------------------------------------------------
def ape_combine(o_ctx: np.ndarray, lse_ctx: np.ndarray, o_on: np.ndarray, lse_on: np.ndarray, scale: float):
    """o = w_c o_ctx + w_o o_on with (w_c, w_o) proportional to
    (exp(scale * lse_ctx), exp(lse_on)); lse = log of their sum.  An empty
    context (lse_ctx = -inf) has weight 0.  Shapes: o [..., d], lse [...]."""
    lc = np.where(np.isneginf(lse_ctx), -np.inf, scale * np.asarray(lse_ctx, dtype=np.float64))
    lo = np.asarray(lse_on, dtype=np.float64)
    m = np.maximum(lc, lo)
    wc = np.exp(lc - m)
    wo = np.exp(lo - m)
    z = wc + wo
    oc = np.where(np.isneginf(lc)[..., None], 0.0, o_ctx)
    o = (wc[..., None] * oc + wo[..., None] * o_on) / z[..., None]
    return o, m + np.log(z)


def ape_request_forward(x, w_q, a, b, s, q_norm_w, eps, theta, art_k: List[np.ndarray], art_v: List[np.ndarray],
                        suffix_k, suffix_v, n_q_heads: int, temperature: float, scale: float, pairs=None):
    """Queries as in request_forward (positions of the assembled context);
    context part = attention over every artifact token with logits divided by
    `temperature`; online part = causal attention over the suffix keys;
    combined by ape_combine."""
    S = x.shape[0]
    S_kv = suffix_k.shape[0]
    d = suffix_k.shape[2]
    t_art = int(sum(t.shape[0] for t in art_k))
    q_raw = lora_q_projection(x, w_q, a, b, s).reshape(S, n_q_heads, d)
    q = rope_rotate_half(rms_norm_heads(q_raw, q_norm_w, eps), query_positions(t_art, S, S_kv), theta)
    o_on, lse_on = attention(q, suffix_k, suffix_v, (S_kv - S) + np.arange(S) + 1, pairs)
    if t_art == 0:
        o_ctx, lse_ctx = np.zeros_like(o_on), np.full(lse_on.shape, -np.inf)
    else:
        k_art = np.concatenate(list(art_k), axis=0)
        v_art = np.concatenate(list(art_v), axis=0)
        # logits q.k / (T sqrt(d)) = (q / T).k / sqrt(d)
        o_ctx, lse_ctx = attention(q / temperature, k_art, v_art, np.full(S, t_art), pairs)
    return ape_combine(o_ctx, lse_ctx, o_on, lse_on, scale)


# ---------------------------------------------------------------------------
# App. "Prompt Construction and Artifact Boundaries" (Tab. prompt layouts):
# text outside the cached artifact spans -- instructions, separators, the
# question -- is processed online, so online spans interleave with the cached
# artifacts in prompt order.  Online tokens are laid out in assembled order in
# one online buffer; item >= 0 is an artifact id, item < 0 an online span of
# -item tokens, and online rows left after the items form the final span.
# Every token sits at its index in the assembled sequence (App. A.5 position
# ids); a query sees the assembled prefix up to its own position.
# ---------------------------------------------------------------------------
def layout_online_positions(items: Sequence[int], art_lengths: Sequence[int], S_kv: int) -> np.ndarray:
    """Assembled position of each of the S_kv online rows."""
    pos = []
    at = 0
    for it in items:
        if it >= 0:
            at += int(art_lengths[it])
        else:
            pos.extend(range(at, at - it))
            at += -it
    pos.extend(range(at, at + S_kv - len(pos)))
    return np.asarray(pos, dtype=np.int64)


def layout_forward(x, w_q, a, b, s, q_norm_w, eps, theta, items: Sequence[int], art_k: dict, art_v: dict,
                   online_k, online_v, n_q_heads: int, pairs=None):
    """x [S, d_model]: the last S online rows; art_k/art_v: artifact id ->
    [L, Hkv, d]; online_k/online_v [S_kv, Hkv, d] in assembled order."""
    S = x.shape[0]
    S_kv = online_k.shape[0]
    d = online_k.shape[2]
    ks, vs = [], []
    row = 0
    for it in items:
        if it >= 0:
            ks.append(art_k[it])
            vs.append(art_v[it])
        else:
            ks.append(online_k[row:row - it])
            vs.append(online_v[row:row - it])
            row += -it
    ks.append(online_k[row:])
    vs.append(online_v[row:])
    lengths = {i: art_k[i].shape[0] for i in art_k}
    pos_all = layout_online_positions(items, [lengths.get(i, 0) for i in range(max(lengths) + 1)] if lengths else [],
                                      S_kv)
    pos_q = pos_all[S_kv - S:]
    q_raw = lora_q_projection(x, w_q, a, b, s).reshape(S, n_q_heads, d)
    q = rope_rotate_half(rms_norm_heads(q_raw, q_norm_w, eps), pos_q, theta)
    return attention(q, np.concatenate(ks, axis=0), np.concatenate(vs, axis=0), pos_q + 1, pairs)


def workload_reference(wl, req: int, pairs=None, q_only: bool = False):
    """Run request_forward on request `req` of a seeded workload object."""
    g = wl.geom
    f = bf16_to_f64
    a = None if wl.lora_a is None else f(wl.lora_a)
    b = None if wl.lora_b is None else f(wl.lora_b)
    ids = wl.requests[req]
    return request_forward(
        f(wl.x[req]), f(wl.w_q), a, b, g.scale, f(wl.q_norm_w), g.rms_eps, g.rope_theta,
        [f(wl.art_k[i]) for i in ids], [f(wl.art_v[i]) for i in ids],
        f(wl.suffix_k[req]), f(wl.suffix_v[req]), g.n_q_heads, pairs=pairs, q_only=q_only)
