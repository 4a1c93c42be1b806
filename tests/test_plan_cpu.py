"""Host planning logic of the library on the CPU: request assembly (block tables,
index maps, prompt layouts with online spans) and the split-KV decomposition of
an attention launch.

The library's own planning source (csrc/plan.cpp) is compiled here with the host
compiler alone, behind a small C shim (tests/plan_shim.cpp), so the code that
runs inside `attuner_assemble`, `attuner_assemble_layout`, `attuner_plan_export`
and every attention launch is checked without a GPU: block tables and index maps
bit-exact against the oracle's storage rule (Sec. 2.1: independently stored
artifact caches concatenated in runtime order), online positions against the
oracle's prompt-layout positions, and the work table against the CTA mapping the
kernels decode (every virtual block of every (request, KV head, row tile) in
exactly one split, every CTA index used once).
"""
from __future__ import annotations

import ctypes
import os
import shutil
import subprocess

import numpy as np
import pytest

from oracle import attuner_oracle as orc

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CSRC = os.path.join(ROOT, "paper_2609_36722_gb300", "csrc")
BUILD = os.path.join(ROOT, "tests", "_build")

OK, ERR_ARG, ERR_UNKNOWN = 0, -1, -3
K_MAX_SPLITS, K_MAX_CHUNK, K_MAX_REQ = 32, 4096, 512
I32P = ctypes.POINTER(ctypes.c_int32)
I64P = ctypes.POINTER(ctypes.c_int64)


@pytest.fixture(scope="module")
def shim():
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    os.makedirs(BUILD, exist_ok=True)
    lib = os.path.join(BUILD, "libplan_shim.so")
    cmd = [cxx, "-std=c++17", "-O1", "-shared", "-fPIC", "-Wall", "-Werror",
           "-I", CSRC, os.path.join(ROOT, "tests", "plan_shim.cpp"), os.path.join(CSRC, "plan.cpp"), "-o", lib]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    h = ctypes.CDLL(lib)
    h.shim_last_error.restype = ctypes.c_char_p
    return h


def _i32(a):
    a = np.ascontiguousarray(np.asarray(a, dtype=np.int32))
    return a, a.ctypes.data_as(I32P)


def bump_firsts(lengths):
    """Bump allocation in registration order (the pool writer's rule)."""
    first, nxt = [], 0
    for L in lengths:
        first.append(nxt)
        nxt += -(-L // 64)
    return first


def assemble(shim, lengths, requests, layout=False, firsts=None):
    """Tables of a plan over `requests` (lists of items); returns (status, dict)."""
    firsts = bump_firsts(lengths) if firsts is None else firsts
    n_req = len(requests)
    items = [it for r in requests for it in r]
    offs = np.cumsum([0] + [len(r) for r in requests])
    fa, fp = _i32(firsts)
    la, lp = _i32(lengths)
    ia, ip = _i32(items if items else [0])
    oa, op = _i32(offs)
    cap = 1 << 20
    out = np.zeros(cap, dtype=np.int32)
    lens = np.zeros(4, dtype=np.int64)
    st = shim.shim_assemble(fp, lp, len(lengths), ip, op, n_req, int(layout), out.ctypes.data_as(I32P),
                            ctypes.c_int64(cap), lens.ctypes.data_as(I64P))
    if st != OK:
        return st, None
    nb, ns, na = int(lens[0]), int(lens[1]), int(lens[2])
    sizes = [n_req + 1, nb, n_req, n_req, n_req + 1, ns, n_req + 1, na]
    names = ["blk_off", "blocks", "t_art", "o_rows", "span_off", "spans", "req_art_off", "art_ids"]
    t, at = {}, 0
    for nm, sz in zip(names, sizes):
        t[nm] = out[at:at + sz].copy()
        at += sz
    t["max_o_rows"] = int(lens[3])
    return st, t


def export(shim, lengths, requests, layout=False, caps=None):
    firsts = bump_firsts(lengths)
    n_req = len(requests)
    items = [it for r in requests for it in r]
    offs = np.cumsum([0] + [len(r) for r in requests])
    fa, fp = _i32(firsts)
    la, lp = _i32(lengths)
    ia, ip = _i32(items if items else [0])
    oa, op = _i32(offs)
    n = 1 << 18
    bufs = [np.full(n, -7, dtype=np.int32) for _ in range(5)]
    sizes = np.array(caps if caps is not None else [n] * 5 + [0], dtype=np.int64)
    st = shim.shim_export(fp, lp, len(lengths), ip, op, n_req, int(layout),
                          *[b.ctypes.data_as(I32P) for b in bufs], sizes.ctypes.data_as(I64P))
    return st, bufs, sizes


# ---------------------------------------------------------------------------
# assembly
# ---------------------------------------------------------------------------
def _random_registry(rng, n):
    # lengths across block boundaries: 1, 63, 64, 65, 128 ... and random
    special = [1, 63, 64, 65, 127, 128, 129]
    return [int(special[i]) if i < len(special) and rng.random() < 0.5 else int(rng.integers(1, 400))
            for i in range(n)]


def test_export_matches_oracle_storage_rule(shim):
    rng = np.random.default_rng(11)
    for trial in range(40):
        lengths = _random_registry(rng, int(rng.integers(1, 9)))
        n_req = int(rng.integers(1, 6))
        # runtime order, repeats allowed, empty requests allowed
        requests = [[int(a) for a in rng.integers(0, len(lengths), size=int(rng.integers(0, 6)))]
                    for _ in range(n_req)]
        st, bufs, sizes = export(shim, lengths, requests)
        assert st == OK, shim.shim_last_error()
        bt, vl, im, ta, to = bufs
        nb, nt = int(sizes[0]), int(sizes[2])
        want = {k: [] for k in ("block_table", "valid_len", "index_map", "token_art", "token_off")}
        for req in requests:
            ref = orc.assemble(lengths, req)
            for k in want:
                want[k].append(ref[k])
        cat = {k: np.concatenate(v) if v else np.zeros(0, np.int32) for k, v in want.items()}
        assert nb == len(cat["block_table"]) and nt == len(cat["index_map"])
        assert sizes[5] == n_req
        np.testing.assert_array_equal(bt[:nb], cat["block_table"])
        np.testing.assert_array_equal(vl[:nb], cat["valid_len"])
        np.testing.assert_array_equal(im[:nt], cat["index_map"])
        np.testing.assert_array_equal(ta[:nt], cat["token_art"])
        np.testing.assert_array_equal(to[:nt], cat["token_off"])
        # nothing written past the counts
        assert (bt[nb:nb + 4] == -7).all() and (im[nt:nt + 4] == -7).all()


def test_plan_tables_of_artifact_lists(shim):
    rng = np.random.default_rng(12)
    for trial in range(30):
        lengths = _random_registry(rng, int(rng.integers(1, 7)))
        firsts = bump_firsts(lengths)
        requests = [[int(a) for a in rng.integers(0, len(lengths), size=int(rng.integers(0, 5)))]
                    for _ in range(int(rng.integers(1, 5)))]
        st, t = assemble(shim, lengths, requests)
        assert st == OK
        assert t["max_o_rows"] == 0 and (t["o_rows"] == 0).all() and len(t["spans"]) == 0
        for r, req in enumerate(requests):
            ents = t["blocks"][t["blk_off"][r]:t["blk_off"][r + 1]]
            want = [((firsts[a] + b) << 7) | min(64, lengths[a] - 64 * b)
                    for a in req for b in range(-(-lengths[a] // 64))]
            np.testing.assert_array_equal(ents, np.asarray(want, np.int32))
            assert (ents > 0).all()
            assert t["t_art"][r] == sum(lengths[a] for a in req)
            ids = t["art_ids"][t["req_art_off"][r]:t["req_art_off"][r + 1]]
            assert ids.tolist() == req


def test_plan_tables_of_prompt_layouts(shim):
    """Online spans between artifacts: slot entries (artifact blocks only: the
    online rows are read after them, packed), span records and the assembled
    position of every online row against the oracle's layout positions."""
    rng = np.random.default_rng(13)
    for trial in range(40):
        lengths = _random_registry(rng, int(rng.integers(1, 6)))
        firsts = bump_firsts(lengths)
        requests = []
        for _ in range(int(rng.integers(1, 4))):
            items = []
            for _ in range(int(rng.integers(1, 7))):
                if rng.random() < 0.4:
                    items.append(-int(rng.choice([1, 5, 63, 64, 65, 130, int(rng.integers(1, 300))])))
                else:
                    items.append(int(rng.integers(0, len(lengths))))
            requests.append(items)
        st, t = assemble(shim, lengths, requests, layout=True)
        assert st == OK, shim.shim_last_error()
        for r, items in enumerate(requests):
            ents = t["blocks"][t["blk_off"][r]:t["blk_off"][r + 1]].tolist()
            spans = t["spans"][4 * t["span_off"][r]:4 * t["span_off"][r + 1]].reshape(-1, 4)
            online = [-it for it in items if it < 0]
            assert t["o_rows"][r] == sum(online)
            assert len(spans) == len(online)
            # walk the items in prompt order: slot entries and span records
            slot, orow, tok, si = 0, 0, 0, 0
            for it in items:
                if it >= 0:
                    L = lengths[it]
                    for b in range(-(-L // 64)):
                        assert ents[slot] == ((firsts[it] + b) << 7) | min(64, L - 64 * b)
                        slot += 1
                    tok += L
                else:
                    # a span takes no slot; it records the artifact slots before it
                    n = -it
                    assert spans[si].tolist() == [orow, n, slot, tok]
                    orow += n
                    si += 1
            assert slot == len(ents) and tok == t["t_art"][r]
            # assembled positions: an online row sits after every artifact token and
            # online row before it in the prompt (the oracle's layout rule)
            S_kv = orow + 3
            pos = orc.layout_online_positions(items, lengths, S_kv)
            for row0, n, _, before in spans.tolist():
                np.testing.assert_array_equal(pos[row0:row0 + n], before + row0 + np.arange(n))
            # the rows after the explicit spans follow the whole prompt
            assert pos[orow] == tok + orow
        assert t["max_o_rows"] == max(t["o_rows"].tolist())


def test_assembly_errors(shim):
    lengths = [10, 70]
    assert assemble(shim, lengths, [[0, 2]])[0] == ERR_UNKNOWN
    assert assemble(shim, lengths, [[0, -5]])[0] == ERR_UNKNOWN          # online span outside a layout
    assert assemble(shim, lengths, [[0, -5]], layout=True)[0] == OK
    assert assemble(shim, lengths, [])[0] == ERR_ARG                      # n_req = 0
    assert assemble(shim, lengths, [[0]] * (K_MAX_REQ + 1))[0] == ERR_ARG
    assert assemble(shim, lengths, [[0]] * K_MAX_REQ)[0] == OK
    assert assemble(shim, lengths, [[-(1 << 22)]], layout=True)[0] == ERR_ARG
    assert assemble(shim, lengths, [[-((1 << 22) - 1)]], layout=True)[0] == OK

    def raw(offs, n_req, items=(0,)):
        fa, fp = _i32(bump_firsts(lengths))
        la, lp = _i32(lengths)
        ia, ip = _i32(list(items))
        oa, op = _i32(offs)
        out = np.zeros(1024, np.int32)
        lens = np.zeros(4, np.int64)
        return shim.shim_assemble(fp, lp, 2, ip, op, n_req, 0, out.ctypes.data_as(I32P), ctypes.c_int64(1024),
                                  lens.ctypes.data_as(I64P))
    assert raw([1, 1], 1) == ERR_ARG                                       # offs[0] != 0
    assert raw([0, 1, 0], 2) == ERR_ARG                                    # decreasing offsets
    assert raw([0, 1], 1) == OK


def test_export_capacity_checks(shim):
    lengths = [100, 30]
    st, _, sizes = export(shim, lengths, [[0, 1]])
    assert st == OK and sizes[:5].tolist() == [3, 3, 130, 130, 130]
    for i, small in enumerate([2, 2, 129, 129, 129]):
        caps = [1 << 18] * 5 + [0]
        caps[i] = small
        assert export(shim, lengths, [[0, 1]], caps=caps)[0] == ERR_ARG


# ---------------------------------------------------------------------------
# split-KV decomposition
# ---------------------------------------------------------------------------
def split(shim, n_q, n_kv, nv_art, o_rows, S, S_kv, tc, num_sms=152, opt_split=0, opt_merge=0,
          clusters=(0, 0, 37, 0, 18, 0, 0, 0, 0), kv_part=0):
    n_req = len(nv_art)
    pol = _i32([n_q, n_kv, num_sms, opt_split, opt_merge] + list(clusters))
    blk = _i32(np.cumsum([0] + list(nv_art)))
    orow = _i32(o_rows)
    out = np.zeros(5 + 2 * n_req, np.int32)
    st = shim.shim_split_part(pol[1], blk[1], orow[1], n_req, S, S_kv, int(tc), kv_part, out.ctypes.data_as(I32P))
    assert st == OK
    w = dict(n_req=int(out[0]), row_tiles=int(out[1]), chunk=int(out[2]), n_cta=int(out[3]), cluster=int(out[4]),
             base=out[5:5 + n_req].tolist(), nsplit=out[5 + n_req:].tolist())
    # the slots the launch reads: the plan's artifact slots, the 64-row chunks
    # of all online rows, or both
    nsuf = [-(-S_kv // 64) for r in range(n_req)]
    nv = [(nv_art[r] if kv_part != 2 else 0) + (nsuf[r] if kv_part != 1 else 0) for r in range(n_req)]
    return w, nv


def check_work(w, nv, n_kv, S, G, tc):
    """The decomposition the kernels decode (CTA -> request, KV head, row tile,
    split; split -> a range of virtual blocks) covers every block once."""
    rows = 256 if tc else 16
    assert w["row_tiles"] == -(-S * G // rows)
    rt = w["row_tiles"]
    if w["cluster"]:
        ns = w["cluster"]
        assert tc and ns in (2, 4)
        assert w["n_cta"] == len(nv) * n_kv * rt * ns
        for r, n in enumerate(nv):
            chunk = ((-(-n // ns)) + 1) & ~1      # per request, whole 128-key tiles
            assert chunk <= K_MAX_CHUNK and ns * chunk >= n
            assert w["nsplit"][r] == ns and w["base"][r] == r * n_kv * rt * ns
        return
    chunk = w["chunk"]
    assert chunk >= 1
    if tc:
        assert chunk % 2 == 0
    seen = np.zeros(w["n_cta"], np.int32)
    at = 0
    for r, n in enumerate(nv):
        ns = w["nsplit"][r]
        assert w["base"][r] == at
        assert ns == -(-n // chunk)                       # no empty split, nothing left over
        if tc:
            assert ns <= K_MAX_SPLITS
        covered = np.zeros(n, np.int32)
        for s in range(ns):
            covered[s * chunk:min(n, (s + 1) * chunk)] += 1
            for h in range(n_kv):
                for t in range(rt):
                    seen[w["base"][r] + (s * n_kv + h) * rt + t] += 1
        assert (covered == 1).all()
        at += ns * n_kv * rt
    assert w["n_cta"] == at and (seen == 1).all()


def test_split_work_covers_every_block_once(shim):
    rng = np.random.default_rng(21)
    for trial in range(300):
        n_kv = int(rng.choice([1, 2, 4, 8]))
        G = int(rng.choice([1, 2, 4, 8]))
        n_req = int(rng.integers(1, 7))
        tc = bool(rng.random() < 0.6)
        S = int(rng.integers(1, 300)) if tc else int(rng.integers(1, 3))
        nv_art = [int(rng.integers(0, 400)) for _ in range(n_req)]
        o_rows = [int(rng.integers(0, 100)) if rng.random() < 0.3 else 0 for _ in range(n_req)]
        S_kv = max(o_rows) + S + int(rng.integers(0, 64))
        opt_merge = int(rng.integers(0, 3))
        opt_split = int(rng.choice([0, 0, 2, 6, 64]))
        clusters = (0, 0, int(rng.choice([0, 37, 76])), 0, int(rng.choice([0, 18, 38])), 0, 0, 0, 0)
        w, nv = split(shim, G * n_kv, n_kv, nv_art, o_rows, S, S_kv, tc, num_sms=int(rng.choice([20, 148, 152])),
                      opt_split=opt_split, opt_merge=opt_merge, clusters=clusters)
        check_work(w, nv, n_kv, S, G, tc)
        if opt_merge == 1 or not tc or not any(clusters):
            assert w["cluster"] == 0
        if not tc:
            assert w["chunk"] >= (opt_split if opt_split else 16)


def test_split_work_of_one_part_covers_its_slots_once(shim):
    # a launch over the artifact slots only (kv_part 1: requests without
    # artifacts get no CTA) or the suffix chunks only (kv_part 2), as the APE
    # read makes them; plans without online spans
    rng = np.random.default_rng(22)
    for trial in range(200):
        n_kv = int(rng.choice([1, 2, 4, 8]))
        G = int(rng.choice([1, 2, 4, 8]))
        n_req = int(rng.integers(1, 7))
        tc = bool(rng.random() < 0.6)
        S = int(rng.integers(1, 300)) if tc else int(rng.integers(1, 3))
        nv_art = [int(rng.integers(0, 400)) if rng.random() < 0.8 else 0 for _ in range(n_req)]
        S_kv = S + int(rng.integers(0, 64))
        kv_part = int(rng.integers(1, 3))
        clusters = (0, 0, int(rng.choice([0, 37, 76])), 0, int(rng.choice([0, 18, 38])), 0, 0, 0, 0)
        w, nv = split(shim, G * n_kv, n_kv, nv_art, [0] * n_req, S, S_kv, tc, opt_split=int(rng.choice([0, 2, 6])),
                      opt_merge=int(rng.integers(0, 3)), clusters=clusters, kv_part=kv_part)
        assert nv == (nv_art if kv_part == 1 else [-(-S_kv // 64)] * n_req)
        check_work(w, nv, n_kv, S, G, tc)


def test_split_work_choices(shim):
    # one long request on 152 SMs with 32 (KV head, row tile) units: split
    w, nv = split(shim, 32, 8, [400], [0], 256, 256, True, opt_merge=1)
    check_work(w, nv, 8, 256, 4, True)
    assert w["nsplit"][0] > 1 and w["n_cta"] >= 152 // 2
    # a short request is not split
    w, nv = split(shim, 32, 8, [2], [0], 256, 256, True, opt_merge=1)
    assert w["nsplit"][0] == 1
    # merge option 2 with co-resident clusters: cluster mode
    w, nv = split(shim, 32, 8, [400], [0], 256, 256, True, opt_merge=2)
    check_work(w, nv, 8, 256, 4, True)
    assert w["cluster"] in (2, 4)
    # a fixed chunk: that many blocks per split (tcgen05: rounded to whole tiles)
    w, nv = split(shim, 32, 8, [100, 37], [0, 0], 256, 256, True, opt_split=20, opt_merge=1)
    assert w["chunk"] == 20 and w["nsplit"] == [-(-nv[0] // 20), -(-nv[1] // 20)]
    # more blocks than 32 chunks of the fixed size hold: the chunk grows to 32 splits
    w, nv = split(shim, 32, 8, [2000], [0], 256, 256, True, opt_split=4, opt_merge=1)
    check_work(w, nv, 8, 256, 4, True)
    assert w["nsplit"][0] == K_MAX_SPLITS
    # decode: CTAs of at least 16 blocks, about 8 per SM
    w, nv = split(shim, 32, 8, [700] * 64, [0] * 64, 1, 1, False)
    check_work(w, nv, 8, 1, 4, False)
    assert w["chunk"] >= 16 and w["n_cta"] >= 4 * 152
    # the same inputs give the same table
    a, _ = split(shim, 32, 8, [333, 12, 90], [0, 5, 0], 128, 200, True)
    b, _ = split(shim, 32, 8, [333, 12, 90], [0, 5, 0], 128, 200, True)
    assert a == b


def test_split_work_rejects_a_launch_of_2_31_ctas(shim):
    n_req = 512
    pol = _i32([64, 8, 152, 1, 1] + [0] * 9)                 # one block per split (forced)
    blk = _i32(np.arange(n_req + 1) * 20000)
    orow = _i32([0] * n_req)
    out = np.zeros(5 + 2 * n_req, np.int32)
    # warp-MMA kernel: 32 row tiles x 8 KV heads x 512 requests x 20001 splits > 2^31
    st = shim.shim_split(pol[1], blk[1], orow[1], n_req, 64, 64, 0, out.ctypes.data_as(I32P))
    assert st == ERR_ARG and b"2^31" in shim.shim_last_error()
    # the automatic chunk keeps the same plan well inside the limit
    pol_auto = _i32([64, 8, 152, 0, 1] + [0] * 9)
    st = shim.shim_split(pol_auto[1], blk[1], orow[1], n_req, 64, 64, 0, out.ctypes.data_as(I32P))
    assert st == OK and 0 < out[3] < 1 << 31


# ---------------------------------------------------------------------------
# Q projection launch shape (rows per CTA, K slices per tile)
# ---------------------------------------------------------------------------
def qp_shape(shim, head_dim, hidden, heads, M, n_lora, num_sms=152, rows=0, split=0):
    pol, pp = _i32([head_dim, hidden, num_sms, rows, split])
    out = np.zeros(2, np.int32)
    shim.shim_qproj_shape(pp, heads, M, n_lora, out.ctypes.data_as(I32P))
    return int(out[0]), int(out[1])


def test_qproj_supported_shapes(shim):
    """The K-split epilogue needs at least 8 rotary pairs per thread (ks/mr
    threads per row) and the exchanged fp32 rows must fit the stage ring."""
    sup = lambda D, mr, ks, nl: bool(shim.shim_qproj_supported(D, mr, ks, nl))
    for D in (64, 128):
        for mr in (1, 2):
            assert sup(D, mr, 1, 0) and sup(D, mr, 1, 64)           # no split: every rank
    assert sup(128, 1, 8, 16) and sup(128, 2, 8, 16) and sup(64, 2, 8, 16)
    assert not sup(64, 1, 8, 16)                                     # 32/8 = 4 pairs per thread
    assert sup(128, 2, 2, 32) and not sup(128, 2, 2, 64)            # 256 rows x 196 floats > ring
    assert sup(128, 1, 2, 64)
    assert not sup(96, 1, 1, 0) and not sup(128, 3, 1, 0) and not sup(128, 1, 3, 0)


def test_qproj_shape_of_the_measured_layers(shim):
    """The cost model's picks on 152 SMs, measured best on GB300: Qwen3-4B
    prefill (M = 256) 128 rows and 2 slices, decode (M = 64) 128 rows and 4
    slices, the 2048-token layers 256 rows and no split; the K/V mode's 16
    grid heads of a decode step 8 slices."""
    assert qp_shape(shim, 128, 2560, 32, 256, 16) == (1, 2)
    assert qp_shape(shim, 128, 4096, 32, 64, 16) == (1, 4)
    assert qp_shape(shim, 128, 4096, 32, 2048, 16) == (2, 1)
    assert qp_shape(shim, 128, 4096, 16, 64, 0) == (1, 8)
    assert qp_shape(shim, 64, 256, 4, 16, 16) == (1, 1)


def test_qproj_shape_options_and_limits(shim):
    rng = np.random.default_rng(29)
    for _ in range(300):
        D = int(rng.choice([64, 128]))
        hidden = 64 * int(rng.integers(1, 80))
        heads = int(rng.integers(1, 70))
        M = int(rng.integers(1, 5000))
        nl = int(rng.choice([0, 16, 32, 64]))
        sms = int(rng.choice([20, 148, 152]))
        rows = int(rng.choice([0, 128, 256]))
        split = int(rng.choice([0, 1, 2, 4, 8]))
        mr, ks = qp_shape(shim, D, hidden, heads, M, nl, sms, rows, split)
        if mr == 0:
            # only pinned options can leave no shape
            assert rows or split
            assert ks == 0
            continue
        assert bool(shim.shim_qproj_supported(D, mr, ks, nl))
        assert ks <= hidden // 64                       # every CTA has a K block
        if rows:
            assert mr * 128 == rows
        if split:
            assert ks == split
    # one K block (hidden 64): no split
    for D in (64, 128):
        assert qp_shape(shim, D, 64, 8, 100, 16)[1] == 1
    assert qp_shape(shim, 64, 512, 4, 300, 8, rows=128, split=8) == (0, 0)


# ---------------------------------------------------------------------------
# shared reads of the decode kernel
# ---------------------------------------------------------------------------
def share_plan(shim, lengths, requests, S, S_kv, n_q=32, n_kv=8, num_sms=152, opt_split=0, opt_share=0,
               k_by_slot=0, kv_part=0, layout=0):
    firsts = bump_firsts(lengths)
    n_req = len(requests)
    items = [it for r in requests for it in r]
    offs = np.cumsum([0] + [len(r) for r in requests])
    fa, fp = _i32(firsts)
    la, lp = _i32(lengths)
    ia, ip = _i32(items if items else [0])
    oa, op = _i32(offs)
    pol = _i32([n_q, n_kv, num_sms, opt_split, opt_share, k_by_slot, kv_part, layout])
    cap = 1 << 20
    out = np.zeros(cap, np.int32)
    lens = np.zeros(2, np.int64)
    st = shim.shim_share(pol[1], fp, lp, len(lengths), ip, op, n_req, S, S_kv, out.ctypes.data_as(I32P),
                         ctypes.c_int64(cap), lens.ctypes.data_as(I64P))
    assert st == OK, shim.shim_last_error()
    n_refs, n_dist = int(lens[0]), int(lens[1])
    keys = ["n_cta", "chunk", "share", "members", "n_dist", "art_units", "suf_chunks", "n_part", "whole_refs"]
    w = {k: int(out[i]) for i, k in enumerate(keys)}
    at = len(keys)
    w["base"] = out[at:at + n_req].tolist()
    at += n_req
    if w["share"]:
        w["nsplit"] = out[at:at + n_dist + 1].tolist()
        at += n_dist + 1
    t = {}
    for nm, sz in (("ref_req", n_refs), ("ref_slot", n_refs), ("ref_nblk", n_refs), ("dist_off", n_dist + 1 if n_refs else 0),
                   ("dist_refs", n_refs), ("dist_src", n_dist), ("dist_nb", n_dist), ("dref_req", n_refs),
                   ("dref_j", n_refs), ("dref_nref", n_refs)):
        t[nm] = out[at:at + sz].tolist()
        at += sz
    return w, t


def check_share_tables(t, lengths, requests):
    """References in plan order (request, first slot, blocks) and their grouping
    by artifact id (ascending id, plan order within an id)."""
    refs = [(r, a) for r, req in enumerate(requests) for a in req]
    nb = [-(-lengths[a] // 64) for _, a in refs]
    assert t["ref_req"] == [r for r, _ in refs]
    assert t["ref_nblk"] == nb
    slot, want = {}, []
    for (r, a), n in zip(refs, nb):
        want.append(slot.get(r, 0))
        slot[r] = slot.get(r, 0) + n
    assert t["ref_slot"] == want
    ids = sorted(set(a for _, a in refs))
    groups = [[i for i, (_, a) in enumerate(refs) if a == x] for x in ids]
    assert t["dist_refs"] == [i for g in groups for i in g]
    assert t["dist_off"] == (list(np.cumsum([0] + [len(g) for g in groups])) if refs else [])
    # the flattened forms the kernel reads
    blk_off = list(np.cumsum([0] + [sum(-(-lengths[a] // 64) for a in req) for req in requests]))
    first = [g[0] for g in groups]
    assert t["dist_src"] == [blk_off[refs[i][0]] + want[i] for i in first]
    assert t["dist_nb"] == [nb[i] for i in first]
    order = t["dist_refs"]
    assert t["dref_req"] == [refs[i][0] for i in order]
    assert t["dref_j"] == [i - sum(len(requests[q]) for q in range(refs[i][0])) for i in order]
    assert t["dref_nref"] == [len(requests[refs[i][0]]) for i in order]


def check_share_work(w, t, lengths, requests, S, S_kv, n_q, n_kv):
    """The CTA -> work mapping the shared-read kernel decodes, restated: every
    (KV head, reference, block) and every (KV head, request, online chunk) is
    read by exactly one CTA, a CTA's members are references of the artifact it
    reads, and every request's partial records 0 .. P_r - 1 are written once
    per KV head, P_r agreeing between all CTAs that write them."""
    G = n_q // n_kv
    R = 16 // (S * G)
    C = w["chunk"]
    assert w["share"] == 1 and w["members"] == R >= 2 and 1 <= C <= 1024
    assert w["whole_refs"] == int(all(nb <= C for nb in t["ref_nblk"]))
    n_req = len(requests)
    nsuf = -(-S_kv // 64)
    assert w["suf_chunks"] == -(-nsuf // C)
    per_head = w["art_units"] + n_req * w["suf_chunks"]
    assert w["n_cta"] == per_head * n_kv
    nd = w["n_dist"]
    assert w["nsplit"][0] == 0 and w["nsplit"][nd] == w["art_units"]
    req_refs = [[i for i, r in enumerate(t["ref_req"]) if r == q] for q in range(n_req)]
    P = [sum(-(-t["ref_nblk"][i] // C) for i in req_refs[r]) + w["suf_chunks"] for r in range(n_req)]
    assert w["base"] == list(np.cumsum([0] + P[:-1])) and w["n_part"] == sum(P)
    refs = [(r, a) for r, req in enumerate(requests) for a in req]
    # CTA -> (KV head, unit): every head's artifact units, then every head's suffix units
    units = {h: [] for h in range(n_kv)}
    n_suf = n_req * w["suf_chunks"]
    for cta in range(w["n_cta"]):
        if cta < w["art_units"] * n_kv:
            units[cta // w["art_units"]].append(cta % w["art_units"])
        else:
            v = cta - w["art_units"] * n_kv
            units[v // n_suf].append(w["art_units"] + v % n_suf)
    for h in range(n_kv):
        read = {}
        parts = {}
        assert sorted(units[h]) == list(range(per_head))
        for u in units[h]:
            if u < w["art_units"]:
                # as the kernel decodes it: from dist_off / dist_nb / dist_src
                # and the dref_* tables of the members
                d = max(x for x in range(nd) if w["nsplit"][x] <= u)
                rb, re_ = t["dist_off"][d], t["dist_off"][d + 1]
                nb = t["dist_nb"][d]
                nch = -(-nb // C)
                local = u - w["nsplit"][d]
                chunk, m_beg = local % nch, rb + (local // nch) * R
                n_mem = min(R, re_ - m_beg)
                assert n_mem >= 1
                blocks = range(chunk * C, min(nb, (chunk + 1) * C))
                assert len(blocks) >= 1
                for m in range(n_mem):
                    r, jj, nref = t["dref_req"][m_beg + m], t["dref_j"][m_beg + m], t["dref_nref"][m_beg + m]
                    i = req_refs[r][jj]                                   # the member's reference
                    assert refs[i][1] == refs[t["dist_refs"][rb]][1]      # the same artifact
                    assert nref == len(req_refs[r])
                    for b in blocks:
                        read[("art", i, b)] = read.get(("art", i, b), 0) + 1
                    if w["whole_refs"]:
                        k = jj + chunk
                    else:
                        k = sum(-(-t["ref_nblk"][req_refs[r][q]] // C) for q in range(jj)) + chunk
                    assert k == sum(-(-t["ref_nblk"][j] // C) for j in req_refs[r] if j < i) + chunk
                    parts[(r, k)] = parts.get((r, k), 0) + 1
            else:
                v = u - w["art_units"]
                r, chunk = v // w["suf_chunks"], v % w["suf_chunks"]
                for b in range(chunk * C, min(nsuf, (chunk + 1) * C)):
                    read[("suf", r, b)] = read.get(("suf", r, b), 0) + 1
                k = sum(-(-t["ref_nblk"][j] // C) for j in req_refs[r]) + chunk
                parts[(r, k)] = parts.get((r, k), 0) + 1
        want = {("art", i, b) for i in range(len(refs)) for b in range(t["ref_nblk"][i])}
        want |= {("suf", r, b) for r in range(n_req) for b in range(nsuf)}
        assert set(read) == want and all(c == 1 for c in read.values())
        assert set(parts) == {(r, k) for r in range(n_req) for k in range(P[r])}
        assert all(c == 1 for c in parts.values())


def test_share_tables_and_work_cover_every_read_once(shim):
    rng = np.random.default_rng(5)
    for trial in range(60):
        lengths = _random_registry(rng, int(rng.integers(1, 12)))
        n_req = int(rng.integers(1, 9))
        requests = []
        for r in range(n_req):
            k = int(rng.integers(0, 6))
            # repeats across requests and now and then within one request
            requests.append([int(a) for a in rng.integers(0, len(lengths), k)])
        S = int(rng.choice([1, 1, 2]))
        n_kv = int(rng.choice([1, 2, 8]))
        G = int(rng.choice([1, 2, 4])) if S == 2 else int(rng.choice([1, 2, 4, 8]))
        S_kv = S + int(rng.integers(0, 200))
        opt_split = int(rng.choice([0, 1, 2, 5, 16]))
        w, t = share_plan(shim, lengths, requests, S, S_kv, n_q=G * n_kv, n_kv=n_kv, opt_split=opt_split, opt_share=2)
        check_share_tables(t, lengths, requests)
        if not any(requests):
            assert w["share"] == 0      # no artifact: nothing to share
            continue
        check_share_work(w, t, lengths, requests, S, S_kv, G * n_kv, n_kv)


def test_share_choice(shim):
    lengths = [640, 1280, 320, 2048, 700]
    shared = [[0, 1, 3], [1, 3, 4], [0, 3], [2, 3, 1]]
    distinct = [[0], [1], [2, 3], [4]]
    plan = lambda req, S=1, **kw: share_plan(shim, lengths, req, S, 129, **kw)[0]
    assert plan(shared)["share"] == 1                    # 25 % fewer block reads and more
    assert plan(distinct)["share"] == 0                  # nothing shared
    assert plan(distinct, opt_share=2)["share"] == 1     # forced
    assert plan(shared, opt_share=1)["share"] == 0       # off
    assert plan(shared, k_by_slot=1)["share"] == 0       # keys rotated per slot
    assert plan(shared, kv_part=1)["share"] == 0         # one part only
    assert plan(shared, S=3)["share"] == 0               # 12 rows per request: one request per CTA
    assert plan(shared, S=2)["share"] == 1 and plan(shared, S=2)["members"] == 2
    # the 64-request decode step: whole artifacts (4 to 32 blocks) per chunk
    rng = np.random.default_rng(0)
    pool = [int(x) for x in rng.integers(256, 2049, 256)]
    reqs = [[int(a) for a in rng.choice(256, int(rng.integers(4, 13)), replace=False)] for _ in range(64)]
    w, t = share_plan(shim, pool, reqs, 1, 129)
    assert w["share"] == 1 and w["members"] == 4 and w["chunk"] == 32
    check_share_work(w, t, pool, reqs, 1, 129, 32, 8)


def test_share_falls_back_beyond_the_distinct_artifact_table(shim):
    # the work table holds 511 distinct artifacts' unit offsets: a plan with
    # more reads per request even when shared reads are forced on
    lengths = [64] * 600
    reqs = [[i, (i + 1) % 600] for i in range(0, 600, 2)] + [[i] for i in range(1, 600, 2)]
    w, _ = share_plan(shim, lengths, reqs[:512], 1, 9, opt_share=2)
    assert w["share"] == 0
    w, t = share_plan(shim, lengths[:511], [[i, (i + 7) % 511] for i in range(511)], 1, 9, opt_share=2)
    assert w["share"] == 1 and w["n_dist"] == 511
    check_share_work(w, t, lengths[:511], [[i, (i + 7) % 511] for i in range(511)], 1, 9, 32, 8)


def test_share_reads_of_prompt_layouts(shim):
    # online spans before and between artifacts: a decode token (in the final
    # span) sees every artifact, so the reads can be shared; queries that sit
    # in an earlier span see only some artifacts, so they cannot
    lengths = [640, 1280, 320, 2048]
    layouts = [[-12, 1, -5, 0, -5, 3], [-7, 1, -5, 3, 0], [0, -9, 1, 3], [3, 1]]
    w, t = share_plan(shim, lengths, layouts, 1, 129, layout=1)
    assert w["share"] == 1
    arts = [[a for a in lay if a >= 0] for lay in layouts]
    check_share_work(w, t, lengths, arts, 1, 129, 32, 8)
    # every query row in the final span: 2 rows of 129 - 22 (the largest explicit span total)
    assert share_plan(shim, lengths, layouts, 2, 129, layout=1)[0]["share"] == 1
    # G = 1, S = 8 (two requests per CTA): with 25 online rows, request 0's 22
    # explicit rows leave 3 in its final span, so 8 queries reach into the
    # spans and cannot share; 3 queries can
    assert share_plan(shim, lengths, layouts, 8, 25, n_q=8, n_kv=8, opt_share=2, layout=1)[0]["share"] == 0
    w3, t3 = share_plan(shim, lengths, layouts, 3, 25, n_q=8, n_kv=8, opt_share=2, layout=1)
    assert w3["share"] == 1
    check_share_work(w3, t3, lengths, arts, 3, 25, 8, 8)
