"""Planted mistakes in the oracle, on the CPU.

Each mutant replaces one oracle function with a plausible error -- a dropped
term, a wrong sign, a wrong index or axis, an off-by-one position or mask, a
transposed operand, a swapped output -- and the pins of test_oracle_pins.py
are run against it: at least one must fail.  A mutant that no pin catches
means a mistake of that kind could hide in the oracle, so the pins (not the
mutant) would have to grow.  Nothing here touches the CUDA path.
"""
from __future__ import annotations

import math

import numpy as np
import pytest

from oracle import attuner_oracle as O
import test_oracle_pins as pins

ORIG = {n: getattr(O, n) for n in ("lora_q_projection", "merged_q_weight", "rms_norm_heads", "rope_rotate_half",
                                  "query_positions", "kv_projection", "assemble", "attention", "request_forward",
                                  "layout_online_positions", "layout_forward", "merge_partials",
                                  "rotate_at_assembly", "epic_request_forward", "ape_combine",
                                  "ape_request_forward")}
PINS = {n: f for n, f in vars(pins).items() if n.startswith("test_") and callable(f)}


# --- Eq. query-adaptation and the merged form -------------------------------
def lora_without_update(x, w_q, a, b, s):
    return x @ w_q.T


def lora_without_scale(x, w_q, a, b, s):
    return ORIG["lora_q_projection"](x, w_q, a, b, 1.0)


def lora_scale_on_base(x, w_q, a, b, s):
    base = ORIG["lora_q_projection"](x, w_q, None, None, s)
    return s * base + (ORIG["lora_q_projection"](x, w_q, a, b, s) - base)


def merged_without_scale(w_q, a, b, s):
    return w_q + b @ a


def merged_transposed_update(w_q, a, b, s):
    return w_q + s * (a.T @ b.T)                                     # (B A)^T


# --- RMSNorm -----------------------------------------------------------------
def rms_without_eps(q, w, eps):
    return q / np.sqrt(np.mean(q * q, axis=-1, keepdims=True)) * w


def rms_sum_not_mean(q, w, eps):
    return q / np.sqrt(np.sum(q * q, axis=-1, keepdims=True) + eps) * w


def rms_over_heads(q, w, eps):
    return q / np.sqrt(np.mean(q * q, axis=-2, keepdims=True) + eps) * w


def rms_without_weight(q, w, eps):
    return ORIG["rms_norm_heads"](q, np.ones_like(w), eps)


# --- RoPE --------------------------------------------------------------------
def rope_wrong_sign(q, pos, theta):
    return ORIG["rope_rotate_half"](q, -np.asarray(pos), theta)


def rope_interleaved_pairs(q, pos, theta):
    d = q.shape[-1]
    perm = np.concatenate([np.arange(0, d, 2), np.arange(1, d, 2)])   # (2j, 2j+1) paired
    inv = np.argsort(perm)
    return ORIG["rope_rotate_half"](q[..., perm], pos, theta)[..., inv]


def rope_half_frequency_exponent(q, pos, theta):
    return ORIG["rope_rotate_half"](q, pos, theta ** 0.5)             # theta^(-j/d)


def rope_position_plus_one(q, pos, theta):
    return ORIG["rope_rotate_half"](q, np.asarray(pos) + 1, theta)


# --- positions -----------------------------------------------------------------
def qpos_off_by_one(t_art, S, S_kv):
    return ORIG["query_positions"](t_art, S, S_kv) + 1


def qpos_without_prior_suffix(t_art, S, S_kv):
    return t_art + np.arange(S, dtype=np.int64)


def layout_pos_ignoring_artifacts(items, art_lengths, S_kv):
    return ORIG["layout_online_positions"](items, [0] * len(art_lengths), S_kv)


def layout_pos_final_span_shifted(items, art_lengths, S_kv):
    p = ORIG["layout_online_positions"](items, art_lengths, S_kv).copy()
    p[sum(-it for it in items if it < 0):] += 1
    return p


# --- assembly ------------------------------------------------------------------
def assemble_first_block_plus_one(art_lengths, request, block_tokens=64):
    r = ORIG["assemble"](art_lengths, request, block_tokens)
    r["block_table"] = r["block_table"] + 1
    r["index_map"] = r["index_map"] + block_tokens
    return r


def assemble_block_and_slot_swapped(art_lengths, request, block_tokens=64):
    r = ORIG["assemble"](art_lengths, request, block_tokens)
    first = r["first_block"]
    r["index_map"] = np.asarray([(first[a] + p % block_tokens) * block_tokens + p // block_tokens
                                 for a in request for p in range(int(art_lengths[a]))], dtype=np.int32)
    return r


def assemble_valid_len_full_blocks(art_lengths, request, block_tokens=64):
    r = ORIG["assemble"](art_lengths, request, block_tokens)
    r["valid_len"] = np.full_like(r["valid_len"], block_tokens)
    return r


# --- attention -----------------------------------------------------------------
def attention_without_scale(q, k, v, n_visible, pairs=None):
    return ORIG["attention"](q * math.sqrt(q.shape[-1]), k, v, n_visible, pairs)


def attention_mask_off_by_one(q, k, v, n_visible, pairs=None):
    return ORIG["attention"](q, k, v, np.maximum(np.asarray(n_visible) - 1, 1), pairs)


def attention_heads_modulo(q, k, v, n_visible, pairs=None):
    Hq, Hkv = q.shape[1], k.shape[1]
    idx = [h % Hkv for h in range(Hq)]                               # h % Hkv instead of h // G
    return ORIG["attention"](q, k[:, idx], v[:, idx], n_visible, pairs)


def attention_lse_base_two(q, k, v, n_visible, pairs=None):
    o, lse = ORIG["attention"](q, k, v, n_visible, pairs)
    return o, lse / math.log(2.0)


def attention_swapped_kv(q, k, v, n_visible, pairs=None):
    return ORIG["attention"](q, v, k, n_visible, pairs)


# --- split-KV combine ----------------------------------------------------------
def merge_unnormalised(o_parts, lse_parts):
    o, lse = ORIG["merge_partials"](o_parts, lse_parts)
    return o * np.exp(lse)[..., None], lse


def merge_plain_mean(o_parts, lse_parts):
    _, lse = ORIG["merge_partials"](o_parts, lse_parts)
    return sum(np.asarray(o) for o in o_parts) / len(o_parts), lse


def merge_lse_of_the_largest_part(o_parts, lse_parts):
    o, _ = ORIG["merge_partials"](o_parts, lse_parts)
    return o, np.max(np.stack([np.asarray(l) for l in lse_parts]), axis=0)


# --- suffix K/V ----------------------------------------------------------------
def kv_without_rope(x, w_k, w_v, k_norm_w, eps, theta, positions, n_kv_heads):
    return ORIG["kv_projection"](x, w_k, w_v, k_norm_w, eps, theta, np.zeros_like(positions), n_kv_heads)


def kv_value_normalised(x, w_k, w_v, k_norm_w, eps, theta, positions, n_kv_heads):
    k, v = ORIG["kv_projection"](x, w_k, w_v, k_norm_w, eps, theta, positions, n_kv_heads)
    return k, ORIG["rms_norm_heads"](v, np.ones(v.shape[-1]), eps)


def kv_outputs_swapped(x, w_k, w_v, k_norm_w, eps, theta, positions, n_kv_heads):
    k, v = ORIG["kv_projection"](x, w_k, w_v, k_norm_w, eps, theta, positions, n_kv_heads)
    return v, k


# --- one request -------------------------------------------------------------------
def _request(x, w_q, a, b, s, q_norm_w, eps, theta, art_k, art_v, suffix_k, suffix_v, n_q_heads,
             pairs=None, q_only=False, *, self_visible=1, causal=True, t_art_in_pos=True):
    S, S_kv, d = x.shape[0], suffix_k.shape[0], suffix_k.shape[2]
    t_art = int(sum(t.shape[0] for t in art_k))
    q_raw = ORIG["lora_q_projection"](x, w_q, a, b, s).reshape(S, n_q_heads, d)
    pos = ORIG["query_positions"](t_art if t_art_in_pos else 0, S, S_kv)
    q = ORIG["rope_rotate_half"](ORIG["rms_norm_heads"](q_raw, q_norm_w, eps), pos, theta)
    if q_only:
        return q
    k_all = np.concatenate(list(art_k) + [suffix_k], axis=0)
    v_all = np.concatenate(list(art_v) + [suffix_v], axis=0)
    n_vis = (t_art + (S_kv - S) + np.arange(S) + self_visible) if causal else np.full(S, t_art + S_kv)
    return ORIG["attention"](q, k_all, v_all, np.maximum(n_vis, 1), pairs)


def request_query_not_self_visible(*a, **kw):
    return _request(*a, self_visible=0, **kw)


def request_suffix_not_causal(*a, **kw):
    return _request(*a, causal=False, **kw)


def request_positions_without_artifacts(*a, **kw):
    return _request(*a, t_art_in_pos=False, **kw)


def layout_query_not_self_visible(x, w_q, a, b, s, q_norm_w, eps, theta, items, art_k, art_v, online_k, online_v,
                                  n_q_heads, pairs=None):
    # the layout forward with every query's mask one key short (its own key hidden)
    real_attention = O.attention
    try:
        O.attention = lambda q, k, v, n_vis, p=None: ORIG["attention"](q, k, v, np.asarray(n_vis) - 1, p)
        return ORIG["layout_forward"](x, w_q, a, b, s, q_norm_w, eps, theta, items, art_k, art_v, online_k,
                                      online_v, n_q_heads, pairs)
    finally:
        O.attention = real_attention


# --- App. C.2 variants: EPIC (rotate at assembly) and APE (calibrated combine)
def rotate_at_local_positions(art_k_raw, theta):
    # each artifact rotated at its own positions 0..L-1 (the PIC cache)
    return np.concatenate([ORIG["rope_rotate_half"](k, np.arange(k.shape[0]), theta) for k in art_k_raw], axis=0)


def rotate_positions_plus_one(art_k_raw, theta):
    k = np.concatenate(list(art_k_raw), axis=0)
    return ORIG["rope_rotate_half"](k, np.arange(k.shape[0]) + 1, theta)


def epic_values_unordered(x, w_q, a, b, s, q_norm_w, eps, theta, art_k_raw, art_v, suffix_k, suffix_v, n_q_heads,
                          pairs=None):
    # values taken in reverse artifact order against keys in runtime order
    return ORIG["epic_request_forward"](x, w_q, a, b, s, q_norm_w, eps, theta, art_k_raw, list(art_v)[::-1],
                                        suffix_k, suffix_v, n_q_heads, pairs)


def epic_queries_at_local_positions(x, w_q, a, b, s, q_norm_w, eps, theta, art_k_raw, art_v, suffix_k, suffix_v,
                                    n_q_heads, pairs=None):
    # queries rotated as if the artifacts were not there
    k_art = O.rotate_at_assembly(art_k_raw, theta)
    v_art = np.concatenate(list(art_v), axis=0)
    S, S_kv, d = x.shape[0], suffix_k.shape[0], suffix_k.shape[2]
    q_raw = O.lora_q_projection(x, w_q, a, b, s).reshape(S, n_q_heads, d)
    q = O.rope_rotate_half(O.rms_norm_heads(q_raw, q_norm_w, eps), (S_kv - S) + np.arange(S), theta)
    return O.attention(q, np.concatenate([k_art, suffix_k]), np.concatenate([v_art, suffix_v]),
                       k_art.shape[0] + (S_kv - S) + np.arange(S) + 1, pairs)


def ape_scale_additive(o_ctx, lse_ctx, o_on, lse_on, scale):
    # the scale as a factor on Z_c (log scale added) instead of a power
    return ORIG["ape_combine"](o_ctx, np.asarray(lse_ctx) + math.log(scale) / scale, o_on, lse_on, scale)


def ape_scale_on_online(o_ctx, lse_ctx, o_on, lse_on, scale):
    return ORIG["ape_combine"](o_on, lse_on, o_ctx, lse_ctx, scale)


def ape_combine_without_normalising(o_ctx, lse_ctx, o_on, lse_on, scale):
    lc = scale * np.asarray(lse_ctx, dtype=np.float64)
    m = np.maximum(lc, lse_on)
    o = np.exp(lc - m)[..., None] * o_ctx + np.exp(np.asarray(lse_on) - m)[..., None] * o_on
    return o, m + np.log(np.exp(lc - m) + np.exp(np.asarray(lse_on) - m))


def ape_temperature_multiplied(x, w_q, a, b, s, q_norm_w, eps, theta, art_k, art_v, suffix_k, suffix_v, n_q_heads,
                               temperature, scale, pairs=None):
    return ORIG["ape_request_forward"](x, w_q, a, b, s, q_norm_w, eps, theta, art_k, art_v, suffix_k, suffix_v,
                                       n_q_heads, 1.0 / temperature, scale, pairs)


def ape_online_not_causal(x, w_q, a, b, s, q_norm_w, eps, theta, art_k, art_v, suffix_k, suffix_v, n_q_heads,
                          temperature, scale, pairs=None):
    real_attention = O.attention
    S_kv = suffix_k.shape[0]
    try:
        O.attention = lambda q, k, v, n_vis, p=None: ORIG["attention"](
            q, k, v, np.full(len(n_vis), S_kv) if k.shape[0] == S_kv else n_vis, p)
        return ORIG["ape_request_forward"](x, w_q, a, b, s, q_norm_w, eps, theta, art_k, art_v, suffix_k, suffix_v,
                                           n_q_heads, temperature, scale, pairs)
    finally:
        O.attention = real_attention


MUTANTS = [
    ("lora_q_projection", lora_without_update), ("lora_q_projection", lora_without_scale),
    ("lora_q_projection", lora_scale_on_base),
    ("merged_q_weight", merged_without_scale), ("merged_q_weight", merged_transposed_update),
    ("rms_norm_heads", rms_without_eps), ("rms_norm_heads", rms_sum_not_mean),
    ("rms_norm_heads", rms_over_heads), ("rms_norm_heads", rms_without_weight),
    ("rope_rotate_half", rope_wrong_sign), ("rope_rotate_half", rope_interleaved_pairs),
    ("rope_rotate_half", rope_half_frequency_exponent), ("rope_rotate_half", rope_position_plus_one),
    ("query_positions", qpos_off_by_one), ("query_positions", qpos_without_prior_suffix),
    ("layout_online_positions", layout_pos_ignoring_artifacts),
    ("layout_online_positions", layout_pos_final_span_shifted),
    ("assemble", assemble_first_block_plus_one), ("assemble", assemble_block_and_slot_swapped),
    ("assemble", assemble_valid_len_full_blocks),
    ("attention", attention_without_scale), ("attention", attention_mask_off_by_one),
    ("attention", attention_heads_modulo), ("attention", attention_lse_base_two),
    ("attention", attention_swapped_kv),
    ("merge_partials", merge_unnormalised), ("merge_partials", merge_plain_mean),
    ("merge_partials", merge_lse_of_the_largest_part),
    ("kv_projection", kv_without_rope), ("kv_projection", kv_value_normalised),
    ("kv_projection", kv_outputs_swapped),
    ("request_forward", request_query_not_self_visible), ("request_forward", request_suffix_not_causal),
    ("request_forward", request_positions_without_artifacts),
    ("layout_forward", layout_query_not_self_visible),
    ("rotate_at_assembly", rotate_at_local_positions), ("rotate_at_assembly", rotate_positions_plus_one),
    ("epic_request_forward", epic_values_unordered), ("epic_request_forward", epic_queries_at_local_positions),
    ("ape_combine", ape_scale_additive), ("ape_combine", ape_scale_on_online),
    ("ape_combine", ape_combine_without_normalising),
    ("ape_request_forward", ape_temperature_multiplied), ("ape_request_forward", ape_online_not_causal),
]


def _pin_order(name):
    # the pins that exercise the mutated function first (stop at the first failure)
    key = {"lora_q_projection": "lora", "merged_q_weight": "merged", "rms_norm_heads": "rmsnorm",
           "rope_rotate_half": "rope", "query_positions": "query_positions", "kv_projection": "kv_projection",
           "assemble": "assemble", "attention": "attention", "request_forward": "artifact",
           "layout_online_positions": "layout", "layout_forward": "layout", "merge_partials": "merge",
           "rotate_at_assembly": "epic", "epic_request_forward": "epic", "ape_combine": "ape",
           "ape_request_forward": "ape"}[name]
    names = sorted(PINS)
    return [n for n in names if key in n] + [n for n in names if key not in n]


@pytest.mark.parametrize("target,mutant", MUTANTS, ids=[m.__name__ for _, m in MUTANTS])
def test_some_pin_catches_the_mutant(target, mutant, monkeypatch):
    monkeypatch.setattr(O, target, mutant)
    for name in _pin_order(target):
        try:
            PINS[name]()
        except Exception:           # an assertion or a shape error: the pin caught it
            return
    pytest.fail(f"no pin fails when {target} is replaced by {mutant.__name__}")


def test_every_oracle_function_has_a_mutant():
    assert {t for t, _ in MUTANTS} == set(ORIG)
