"""Seeded synthetic workloads for the artifact-KV read path.

Each workload mirrors one of the five layer geometries the path is measured
on (a tiny parity case, a Qwen3-4B layer, a Qwen3-8B layer with four
requests, a 64-request decode step, and a 131k-token long context).  The
paper's own datasets (SRA-Bench skills, MuSiQue, PersonaMem-v2, ...) are not
available; these tensors stand in for them with the shapes, lengths and
value distributions listed below.

Value recipe (all tensors stored as bf16):
  artifact K, V, suffix K, V, hidden states x  ~ N(0, 1)
  W_q, A                                       ~ N(0, 1/hidden)   (variance)
  B                                            ~ N(0, 1/r)
  q_norm weight                                = 1 + 0.1 * N(0, 1)

Keys are stored "already rotated" (artifact K at local positions 0..L-1,
suffix K at its assembled positions).  A rotation of an i.i.d. N(0, 1) pair
is again an i.i.d. N(0, 1) pair, so drawing the rotated keys directly gives
exactly the distribution of draw-then-rotate, without putting any rotary
arithmetic in this shared module.

Lengths, artifact choices and runtime orders come from
numpy.random.default_rng(seed); tensor values come from a torch.Generator
seeded with the same seed on the requested device, drawn in a fixed order.
"""

from __future__ import annotations

import dataclasses
from typing import List, Optional

import numpy as np
import torch


@dataclasses.dataclass(frozen=True)
class Geometry:
    hidden: int
    n_q_heads: int
    n_kv_heads: int
    head_dim: int
    rank: int
    scale: float = 2.0          # s = alpha / r (alpha = 16, r = 8 in the paper's training table)
    rope_theta: float = 1.0e6
    rms_eps: float = 1.0e-6
    block_tokens: int = 64

    @property
    def group(self) -> int:
        return self.n_q_heads // self.n_kv_heads

    @property
    def d_q(self) -> int:
        return self.n_q_heads * self.head_dim


@dataclasses.dataclass
class Workload:
    name: str
    geom: Geometry
    seed: int
    art_lengths: List[int]            # pool, in registration order
    requests: List[List[int]]         # artifact ids per request, runtime order
    S: int                            # query tokens per request
    S_kv: int                         # suffix KV entries per request (S_kv >= S)
    # tensors (bf16)
    art_k: List[torch.Tensor]         # each [L, Hkv, d]
    art_v: List[torch.Tensor]
    x: torch.Tensor                   # [n_req, S, hidden]
    w_q: torch.Tensor                 # [Hq*d, hidden]
    lora_a: Optional[torch.Tensor]    # [r, hidden]
    lora_b: Optional[torch.Tensor]    # [Hq*d, r]
    q_norm_w: torch.Tensor            # [d]
    suffix_k: torch.Tensor            # [n_req, S_kv, Hkv, d]
    suffix_v: torch.Tensor

    @property
    def n_req(self) -> int:
        return len(self.requests)

    def t_art(self, req: int) -> int:
        return int(sum(self.art_lengths[a] for a in self.requests[req]))

    def to(self, device) -> "Workload":
        mv = lambda t: None if t is None else t.to(device)
        return dataclasses.replace(
            self,
            art_k=[mv(t) for t in self.art_k],
            art_v=[mv(t) for t in self.art_v],
            x=mv(self.x), w_q=mv(self.w_q), lora_a=mv(self.lora_a),
            lora_b=mv(self.lora_b), q_norm_w=mv(self.q_norm_w),
            suffix_k=mv(self.suffix_k), suffix_v=mv(self.suffix_v))


def _normal(shape, std, gen, device):
    t = torch.randn(*shape, generator=gen, device=device, dtype=torch.float32)
    if std != 1.0:
        t.mul_(std)
    return t.to(torch.bfloat16)


def make_custom(name: str, geom: Geometry, seed: int, art_lengths, requests, S: int,
                S_kv: Optional[int] = None, device="cpu", with_lora: bool = True) -> Workload:
    """Draw tensors for an explicit layout (lengths, requests, S, S_kv)."""
    S_kv = S if S_kv is None else S_kv
    assert S_kv >= S >= 1
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed))
    hkv, d = geom.n_kv_heads, geom.head_dim
    art_k, art_v = [], []
    for L in art_lengths:
        art_k.append(_normal((L, hkv, d), 1.0, gen, device))
        art_v.append(_normal((L, hkv, d), 1.0, gen, device))
    n_req = len(requests)
    x = _normal((n_req, S, geom.hidden), 1.0, gen, device)
    w_q = _normal((geom.d_q, geom.hidden), geom.hidden ** -0.5, gen, device)
    if with_lora and geom.rank > 0:
        lora_a = _normal((geom.rank, geom.hidden), geom.hidden ** -0.5, gen, device)
        lora_b = _normal((geom.d_q, geom.rank), geom.rank ** -0.5, gen, device)
    else:
        lora_a = lora_b = None
    qn = torch.randn(d, generator=gen, device=device, dtype=torch.float32)
    q_norm_w = (1.0 + 0.1 * qn).to(torch.bfloat16)
    suffix_k = _normal((n_req, S_kv, hkv, d), 1.0, gen, device)
    suffix_v = _normal((n_req, S_kv, hkv, d), 1.0, gen, device)
    return Workload(name=name, geom=geom, seed=seed, art_lengths=list(map(int, art_lengths)),
                    requests=[list(map(int, r)) for r in requests], S=S, S_kv=S_kv,
                    art_k=art_k, art_v=art_v, x=x, w_q=w_q, lora_a=lora_a, lora_b=lora_b,
                    q_norm_w=q_norm_w, suffix_k=suffix_k, suffix_v=suffix_v)


QWEN3_4B = Geometry(hidden=2560, n_q_heads=32, n_kv_heads=8, head_dim=128, rank=16)
QWEN3_8B = Geometry(hidden=4096, n_q_heads=32, n_kv_heads=8, head_dim=128, rank=16)
TINY = Geometry(hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=64, rank=8)


def make_kv_weights(geom: Geometry, seed: int, device="cpu"):
    """Base k_proj / v_proj weights [Hkv*d, hidden] ~ N(0, 1/hidden) and a key
    norm weight 1 + 0.1 N(0, 1), bf16, from a generator of their own seed."""
    device = torch.device(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(seed) + 1000)
    n_out = geom.n_kv_heads * geom.head_dim
    w_k = _normal((n_out, geom.hidden), geom.hidden ** -0.5, gen, device).to(torch.bfloat16)
    w_v = _normal((n_out, geom.hidden), geom.hidden ** -0.5, gen, device).to(torch.bfloat16)
    k_norm_w = (1.0 + 0.1 * _normal((geom.head_dim,), 1.0, gen, device)).to(torch.bfloat16)
    return w_k, w_v, k_norm_w


def _layout(name: str):
    """Lengths / requests / S / S_kv of the named workload (numpy-seeded)."""
    if name == "tiny":
        # 3 artifacts of 37, 64, 100 tokens; a 16-token suffix at positions 201..216
        return TINY, 0, [37, 64, 100], [[0, 1, 2]], 16, 16
    if name == "qwen3_4b_prefill":
        rng = np.random.default_rng(1)
        lengths = rng.integers(512, 2048, size=8, endpoint=True).tolist()
        return QWEN3_4B, 1, lengths, [list(range(8))], 256, 256
    if name == "qwen3_8b_prefill_4req":
        rng = np.random.default_rng(2)
        lengths = rng.integers(1024, 4096, size=64, endpoint=True).tolist()
        reqs = [rng.choice(64, size=16, replace=False).tolist() for _ in range(4)]
        return QWEN3_8B, 2, lengths, reqs, 512, 512
    if name == "qwen3_8b_decode_64req":
        rng = np.random.default_rng(3)
        lengths = rng.integers(256, 2048, size=256, endpoint=True).tolist()
        reqs = []
        for _ in range(64):
            k = int(rng.integers(4, 12, endpoint=True))
            reqs.append(rng.choice(256, size=k, replace=False).tolist())
        # 128 prior suffix entries + the new token's own K/V; one query token
        return QWEN3_8B, 3, lengths, reqs, 1, 129
    if name == "qwen3_8b_long_131k":
        return QWEN3_8B, 4, [2048] * 64, [list(range(64))], 2048, 2048
    raise KeyError(name)


WORKLOADS = ["tiny", "qwen3_4b_prefill", "qwen3_8b_prefill_4req",
             "qwen3_8b_decode_64req", "qwen3_8b_long_131k"]


def layout(name: str):
    """(geometry, seed, art_lengths, requests, S, S_kv) without drawing tensors."""
    return _layout(name)


def make_workload(name: str, device="cpu") -> Workload:
    geom, seed, lengths, reqs, S, S_kv = _layout(name)
    return make_custom(name, geom, seed, lengths, reqs, S, S_kv, device=device)
