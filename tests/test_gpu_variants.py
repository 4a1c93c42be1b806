"""GPU parity of the two read variants of the paper's training-free
baselines (App. C.2) against the fp64 oracle, through the C ABI:

* keys stored before RoPE and rotated to their assembled positions at
  assembly (EPIC paragraph): attuner_plan_rotate_keys, then the plain
  attention calls of either kernel read the rotated keys;
* context and online attention computed separately, the context's logits
  divided by a temperature, combined through calibrated log-sum-exp terms
  (APE paragraph): attuner_attend_ape.

Layouts with several requests of ragged lengths, a repeated artifact and a
request without artifacts; both attention kernels; split-KV chunks merged
through global memory and inside clusters.  Bar as for the plain read: O
within max-abs 2e-2 and mean-abs 2e-3, LSE within 1e-2.
"""

import numpy as np
import pytest
import torch

import oracle
import paper_2609_36722_gb300 as pkg
from gen import Geometry, make_custom
from helpers import compare, load_context

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0) if torch.cuda.is_available() else None
G128 = Geometry(hidden=512, n_q_heads=16, n_kv_heads=4, head_dim=128, rank=16)
LENGTHS = [700, 333, 1200, 64, 37]
REQUESTS = [[2, 0, 3], [1, 3], [0, 1, 2, 3, 4], [], [4, 4]]

# (prefill kernel: 1 tcgen05, 2 warp MMA; split blocks; merge mode; S; S_kv)
LAUNCHES = [(1, 0, 0, 96, 96), (1, 4, 1, 96, 96), (1, 8, 2, 96, 96), (1, 0, 0, 300, 333),
            (2, 0, 0, 1, 129), (2, 2, 0, 1, 129), (2, 3, 0, 3, 40)]
IDS = ["tc", "tc-global", "tc-cluster", "tc-ragged", "mma-decode", "mma-decode-split", "mma-3rows"]


def _np(t):
    return t.double().cpu().numpy()


def _oracle(wl, fn, **kw):
    f = oracle.bf16_to_f64
    g = wl.geom
    outs, lses = [], []
    for r, ids in enumerate(wl.requests):
        o, l = fn(f(wl.x[r]), f(wl.w_q), f(wl.lora_a), f(wl.lora_b), g.scale, f(wl.q_norm_w), g.rms_eps,
                  g.rope_theta, [f(wl.art_k[i]) for i in ids], [f(wl.art_v[i]) for i in ids], f(wl.suffix_k[r]),
                  f(wl.suffix_v[r]), g.n_q_heads, **kw)
        outs.append(o)
        lses.append(l)
    return np.stack(outs), np.stack(lses)


def _setup(seed, launch):
    kernel, split, merge, S, S_kv = launch
    wl = make_custom("variant", G128, seed, LENGTHS, REQUESTS, S, S_kv, device=DEV)
    ctx, plan = load_context(wl)
    ctx.set_option(pkg.OPT_PREFILL_KERNEL, kernel)
    ctx.set_option(pkg.OPT_SPLIT_BLOCKS, split)
    ctx.set_option(pkg.OPT_SPLIT_MERGE, merge)
    g = wl.geom
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=S_kv)
    return wl, ctx, plan, q


@pytest.mark.parametrize("launch", LAUNCHES, ids=IDS)
def test_keys_rotated_at_assembly_match_the_oracle(launch):
    # the registered keys are read as keys before RoPE: the oracle rotates
    # the same bf16 values at their assembled positions
    wl, ctx, plan, q = _setup(61, launch)
    plain, _ = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    ctx.rotate_keys(plan)
    out, lse = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    o_ref, l_ref = _oracle(wl, oracle.epic_request_forward)
    compare(_np(out), o_ref, _np(lse), l_ref, label=f"epic {launch}")
    # the rotation changes what requests with a non-first artifact read
    assert (out[0].double() - plain[0].double()).abs().max().item() > 1e-2
    # the same plan through the whole path (projection + attention)
    g = wl.geom
    out2, _ = ctx.query_attend(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, wl.suffix_k,
                               wl.suffix_v)
    assert ctx.sync_status() == 0
    assert torch.equal(out2, out)


def test_rotating_twice_and_the_rotated_keys_themselves():
    # the rotated buffer holds bf16(R(pos) k) for every artifact token: the
    # oracle's rotation of the same keys, rounded once; a second rotation of
    # the same plan rewrites the same bytes
    wl, ctx, plan, q = _setup(62, LAUNCHES[0])
    ctx.rotate_keys(plan)
    out1, _ = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    ctx.rotate_keys(plan)
    out2, _ = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    assert torch.equal(out1, out2)


@pytest.mark.parametrize("launch", LAUNCHES, ids=IDS)
@pytest.mark.parametrize("T,scale", [(0.9, 0.9), (0.7, 1.2)])
def test_ape_read_matches_the_oracle(launch, T, scale):
    wl, ctx, plan, q = _setup(63, launch)
    out, lse = ctx.attend_ape(plan, q, wl.suffix_k, wl.suffix_v, T, scale)
    assert ctx.sync_status() == 0
    assert ctx.last_launch_count() >= 3
    o_ref, l_ref = _oracle(wl, oracle.ape_request_forward, temperature=T, scale=scale)
    compare(_np(out), o_ref, _np(lse), l_ref, label=f"ape {launch} T={T} scale={scale}")


@pytest.mark.parametrize("launch", [LAUNCHES[0], LAUNCHES[4]], ids=["tc", "mma-decode"])
def test_ape_with_unit_temperature_and_scale_is_the_plain_read(launch):
    wl, ctx, plan, q = _setup(64, launch)
    ref_o, ref_l = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    out, lse = ctx.attend_ape(plan, q, wl.suffix_k, wl.suffix_v, 1.0, 1.0)
    assert ctx.sync_status() == 0
    d = (out.double() - ref_o.double()).abs()
    assert d.max().item() <= 2e-2 and d.mean().item() <= 2e-3
    assert (lse - ref_l).abs().max().item() <= 1e-2


def test_ape_without_any_artifact():
    # no request has an artifact: the context launch has no CTA and the
    # result is the online attention alone
    wl = make_custom("variant_empty", G128, 65, [64], [[], []], 40, 70, device=DEV)
    ctx, plan = load_context(wl)
    g = wl.geom
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=70)
    out, lse = ctx.attend_ape(plan, q, wl.suffix_k, wl.suffix_v, 0.9, 0.9)
    assert ctx.sync_status() == 0
    o_ref, l_ref = _oracle(wl, oracle.ape_request_forward, temperature=0.9, scale=0.9)
    compare(_np(out), o_ref, _np(lse), l_ref, label="ape without artifacts")


def test_variants_refuse_prompt_layouts_and_bad_parameters():
    wl = make_custom("variant_layout", G128, 66, [100, 70], [[0, 1]], 40, 60, device=DEV)
    ctx, _ = load_context(wl)
    lplan = ctx.assemble_layout([[-8, 0, -4, 1]])
    q = torch.zeros(1, 40, 16, 128, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(pkg.AttunerError) as e:
        ctx.rotate_keys(lplan)
    assert e.value.status == pkg.attuner.ERR_UNSUPPORTED
    with pytest.raises(pkg.AttunerError) as e:
        ctx.attend_ape(lplan, q, wl.suffix_k, wl.suffix_v)
    assert e.value.status == pkg.attuner.ERR_UNSUPPORTED
    plan = ctx.assemble([[0, 1]])
    for T, sc in ((0.0, 0.9), (0.9, -1.0), (float("inf"), 0.9)):
        with pytest.raises(pkg.AttunerError) as e:
            ctx.attend_ape(plan, q, wl.suffix_k, wl.suffix_v, T, sc)
        assert e.value.status == pkg.attuner.ERR_INVALID_ARG
    assert ctx.sync_status() == 0


def _sampled_variant_check(wl, out, lse, fn, label, **kw):
    from helpers import sample_pairs
    f = oracle.bf16_to_f64
    g = wl.geom
    trip = sample_pairs(wl, n=256, seed=7)
    o_sel, l_sel, o_ref, l_ref = [], [], [], []
    for r, ids in enumerate(wl.requests):
        pairs = [(i, h) for (rr, i, h) in trip if rr == r]
        if not pairs:
            continue
        o, l = fn(f(wl.x[r]), f(wl.w_q), f(wl.lora_a), f(wl.lora_b), g.scale, f(wl.q_norm_w), g.rms_eps,
                  g.rope_theta, [f(wl.art_k[i]) for i in ids], [f(wl.art_v[i]) for i in ids], f(wl.suffix_k[r]),
                  f(wl.suffix_v[r]), g.n_q_heads, pairs=pairs, **kw)
        o_ref.append(o)
        l_ref.append(l)
        idx_i = torch.tensor([i for i, _ in pairs], device=DEV)
        idx_h = torch.tensor([h for _, h in pairs], device=DEV)
        o_sel.append(_np(out[r][idx_i, idx_h]))
        l_sel.append(_np(lse[r][idx_i, idx_h]))
    compare(np.concatenate(o_sel), np.concatenate(o_ref), np.concatenate(l_sel), np.concatenate(l_ref),
            label=f"{label} ({len(trip)} sampled rows)")


@pytest.mark.slow
@pytest.mark.parametrize("name", ["qwen3_4b_prefill", "qwen3_8b_decode_64req"])
def test_variants_at_full_size(name):
    # the two variants on full workloads, in the launch configuration the
    # bench times (automatic kernel, split and merge choice), on sampled rows
    from gen import make_workload
    from helpers import load_context
    wl = make_workload(name, device=DEV)
    ctx, plan = load_context(wl)
    g = wl.geom
    q = ctx.q_project(plan, wl.x, wl.w_q, wl.lora_a, wl.lora_b, g.scale, wl.q_norm_w, S_kv=wl.S_kv)
    out, lse = ctx.attend_ape(plan, q, wl.suffix_k, wl.suffix_v, 0.9, 0.9)
    assert ctx.sync_status() == 0
    _sampled_variant_check(wl, out, lse, oracle.ape_request_forward, f"ape {name}", temperature=0.9, scale=0.9)
    ctx.rotate_keys(plan)
    out, lse = ctx.attend(plan, q, wl.suffix_k, wl.suffix_v)
    assert ctx.sync_status() == 0
    _sampled_variant_check(wl, out, lse, oracle.epic_request_forward, f"epic {name}")
