"""ctypes binding of libattuner (include/attuner.h).

Argument marshalling only: every step of the path runs in the library's CUDA
kernels.  PyTorch supplies device memory (``tensor.data_ptr()``) and streams
(``torch.cuda.current_stream().cuda_stream``).  There is no fallback: if the
shared library is missing, importing this module raises.
"""

from __future__ import annotations

import array
import ctypes
import itertools
import os
from typing import List, Optional, Sequence

import torch

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libattuner.so")

OK = 0
ERR_INVALID_ARG = -1
ERR_OOM = -2
ERR_UNKNOWN_ARTIFACT = -3
ERR_CUDA = -4
ERR_TIMEOUT = -5
ERR_UNSUPPORTED = -6
ERR_DEVICE_CHECK = -7

OPT_PREFILL_KERNEL = 1
OPT_SPLIT_BLOCKS = 2
OPT_WAIT_LIMIT = 3
OPT_QPROJ_SPLIT_K = 4
OPT_SPLIT_MERGE = 5
OPT_SYNC_CHECK = 6
OPT_QPROJ_ROWS = 7
OPT_SHARE_READS = 8
OPT_TEST_STUCK_WAIT = 1000

BLOCK_TOKENS = 64

# every symbol include/attuner.h declares
EXPORTS = [
    "attuner_create", "attuner_destroy", "attuner_register_artifact", "attuner_assemble",
    "attuner_plan_export", "attuner_plan_t_art", "attuner_plan_free", "attuner_q_project",
    "attuner_attend", "attuner_query_attend", "attuner_pool_info", "attuner_sync_status",
    "attuner_set_option", "attuner_last_launch_count", "attuner_last_error",
    "attuner_attend_static_scratch", "attuner_register_artifacts_host", "attuner_pool_reset",
    "attuner_kv_project", "attuner_assemble_layout", "attuner_plan_rotate_keys", "attuner_attend_ape",
    "attuner_query_attend_host",
]


class AttunerError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"attuner status {status}: {msg}")
        self.status = status


class Config(ctypes.Structure):
    _fields_ = [
        ("hidden", ctypes.c_int32), ("n_q_heads", ctypes.c_int32), ("n_kv_heads", ctypes.c_int32),
        ("head_dim", ctypes.c_int32), ("block_tokens", ctypes.c_int32), ("pool_blocks", ctypes.c_int32),
        ("rope_theta", ctypes.c_float), ("rms_eps", ctypes.c_float), ("device", ctypes.c_int32),
    ]


_vp = ctypes.c_void_p
_i32 = ctypes.c_int32
_p_i32 = ctypes.POINTER(ctypes.c_int32)
_p_i64 = ctypes.POINTER(ctypes.c_int64)


# argument and return types of every entry point, in the order include/attuner.h gives
SIGNATURES = {
    "attuner_create": ([ctypes.POINTER(Config), ctypes.POINTER(_vp)], _i32),
    "attuner_destroy": ([_vp], _i32),
    "attuner_register_artifact": ([_vp, _vp, _vp, _i32, _vp, _p_i32], _i32),
    "attuner_assemble": ([_vp, _p_i32, _p_i32, _i32, ctypes.POINTER(_vp)], _i32),
    "attuner_plan_export": ([_vp, _p_i32, _p_i32, _p_i32, _p_i32, _p_i32, _p_i64], _i32),
    "attuner_plan_t_art": ([_vp, _p_i32, _i32], _i32),
    "attuner_plan_free": ([_vp], _i32),
    "attuner_q_project": ([_vp, _vp, _vp, _vp, _vp, _vp, _i32, ctypes.c_float, _vp, _i32, _i32, _vp, _vp], _i32),
    "attuner_attend": ([_vp, _vp, _vp, _vp, _vp, _i32, _i32, _vp, _vp, _vp], _i32),
    "attuner_attend_static_scratch": ([_vp, _vp, _vp, _vp, _vp, _i32, _i32, _vp, _vp, _vp], _i32),
    "attuner_query_attend": ([_vp, _vp, _vp, _vp, _vp, _vp, _i32, ctypes.c_float, _vp, _vp, _vp, _i32, _i32,
                              _vp, _vp, _vp], _i32),
    "attuner_query_attend_host": ([_vp, _vp, _vp, _vp, _vp, _vp, _i32, ctypes.c_float, _vp, _vp, _vp, _vp, _vp,
                                   _i32, _i32, _vp, _vp, _vp], _i32),
    "attuner_pool_info": ([_vp, ctypes.POINTER(_vp), ctypes.POINTER(_vp), _p_i32, _p_i32], _i32),
    "attuner_sync_status": ([_vp, _vp], _i32),
    "attuner_set_option": ([_vp, _i32, ctypes.c_int64], _i32),
    "attuner_last_launch_count": ([_vp], _i32),
    "attuner_last_error": ([], ctypes.c_char_p),
    "attuner_register_artifacts_host": ([_vp, _i32, ctypes.POINTER(_vp), ctypes.POINTER(_vp), _p_i32, _vp,
                                         _p_i32], _i32),
    "attuner_pool_reset": ([_vp], _i32),
    "attuner_kv_project": ([_vp, _vp, _vp, _vp, _vp, _vp, _i32, _i32, _vp, _vp, _vp], _i32),
    "attuner_assemble_layout": ([_vp, _p_i32, _p_i32, _i32, ctypes.POINTER(_vp)], _i32),
    "attuner_plan_rotate_keys": ([_vp, _vp, _vp], _i32),
    "attuner_attend_ape": ([_vp, _vp, _vp, _vp, _vp, _i32, _i32, ctypes.c_float, ctypes.c_float, _vp, _vp, _vp],
                           _i32),
}


def load_library(path: str = LIB_PATH) -> ctypes.CDLL:
    if not os.path.exists(path):
        raise ImportError(f"libattuner.so is not built ({path}); run __graft_entry__.build() "
                          "or python -m paper_2609_36722_gb300.build")
    lib = ctypes.CDLL(path)
    for name, (args, ret) in SIGNATURES.items():
        f = getattr(lib, name)
        f.argtypes = args
        f.restype = ret
    return lib


_LIB: Optional[ctypes.CDLL] = None


def lib() -> ctypes.CDLL:
    global _LIB
    if _LIB is None:
        _LIB = load_library()
    return _LIB


def _check(status: int):
    if status != OK:
        raise AttunerError(status, lib().attuner_last_error().decode())


def _ptr(t: Optional[torch.Tensor], name: str, dtype=torch.bfloat16, device=None) -> Optional[int]:
    if t is None:
        return None
    # the usual case in one test; which rule a tensor breaks is worked out
    # only when it breaks one
    if (t.dtype is dtype and t.is_cuda and (device is None or t.get_device() == device.index)
            and t.is_contiguous()):
        return t.data_ptr()
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, the context on {device}")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


def _host_ptr(t: Optional[torch.Tensor], name: str, dtype=torch.bfloat16) -> Optional[int]:
    # a host (CPU) tensor's address; pinned memory keeps the library's copies asynchronous
    if t is None:
        return None
    if t.is_cuda:
        raise ValueError(f"{name} must be a CPU tensor")
    if t.dtype != dtype:
        raise ValueError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    return t.data_ptr()


# the current stream of a device as a raw handle, without building a Stream object
_RAW_STREAM = getattr(torch._C, "_cuda_getCurrentRawStream", None)


def _stream(stream, device=None) -> Optional[int]:
    # the caller's stream, else the current stream of the context's device
    if stream is None:
        if _RAW_STREAM is not None and device is not None and torch.cuda.is_initialized():
            return _RAW_STREAM(device.index)
        stream = torch.cuda.current_stream(device)
    elif device is not None and getattr(stream, "device", device) != device:
        raise ValueError(f"stream is on {stream.device}, the context on {device}")
    return stream.cuda_stream


class Plan:
    """Assembled requests: block tables and index maps on the device."""

    def __init__(self, ctx: "Context", handle: ctypes.c_void_p, requests: List[List[int]]):
        self.ctx = ctx
        self.handle = handle
        self.requests = requests
        self.n_req = len(requests)

    def t_art(self) -> List[int]:
        arr = (ctypes.c_int32 * self.n_req)()
        _check(lib().attuner_plan_t_art(self.handle, arr, self.n_req))
        return list(arr)

    def export(self):
        """Host copies of block table, valid lengths, index map, token artifact and offset."""
        import numpy as np
        sizes = (ctypes.c_int64 * 6)(0, 0, 0, 0, 0, 0)
        _check(lib().attuner_plan_export(self.handle, None, None, None, None, None, sizes))
        nb, nt = sizes[0], sizes[2]
        arrs = [np.zeros(max(n, 1), dtype=np.int32) for n in (nb, nb, nt, nt, nt)]
        ptrs = [a.ctypes.data_as(_p_i32) for a in arrs]
        _check(lib().attuner_plan_export(self.handle, *ptrs, sizes))
        bt, vl, im, ta, to = (a[:n] for a, n in zip(arrs, (nb, nb, nt, nt, nt)))
        return dict(block_table=bt, valid_len=vl, index_map=im, token_art=ta, token_off=to)

    def free(self):
        if self.handle:
            lib().attuner_plan_free(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.free()
        except Exception:
            pass


class Context:
    """One layer's artifact KV store on one GPU (attuner_create)."""

    def __init__(self, hidden: int, n_q_heads: int, n_kv_heads: int, head_dim: int, pool_blocks: int,
                 rope_theta: float = 1.0e6, rms_eps: float = 1.0e-6, device: int = 0):
        cfg = Config(hidden, n_q_heads, n_kv_heads, head_dim, BLOCK_TOKENS, pool_blocks, rope_theta, rms_eps,
                     device)
        h = ctypes.c_void_p()
        _check(lib().attuner_create(ctypes.byref(cfg), ctypes.byref(h)))
        self.handle = h
        self.cfg = cfg
        self.device = torch.device("cuda", device)

    @classmethod
    def for_geometry(cls, geom, pool_blocks: int, device: int = 0) -> "Context":
        return cls(geom.hidden, geom.n_q_heads, geom.n_kv_heads, geom.head_dim, pool_blocks,
                   geom.rope_theta, geom.rms_eps, device)

    def close(self):
        if getattr(self, "handle", None):
            lib().attuner_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    # --- artifacts and plans
    def register_artifact(self, k: torch.Tensor, v: torch.Tensor, stream=None) -> int:
        if k.shape != v.shape or k.dim() != 3:
            raise ValueError("k and v must both be [L, Hkv, d]")
        aid = ctypes.c_int32(-1)
        _check(lib().attuner_register_artifact(self.handle, self._p(k, "k"), self._p(v, "v"), k.shape[0],
                                               self._s(stream), ctypes.byref(aid)))
        return aid.value

    def register_artifacts_host(self, ks: Sequence[torch.Tensor], vs: Sequence[torch.Tensor], stream=None) -> list:
        """Warm-cache load: artifacts whose K/V are pinned CPU tensors [L, Hkv, d]
        bf16, copied into the pool by one kernel on `stream`.  Keep the tensors
        alive and unchanged until that stream has run the copy."""
        n = len(ks)
        if n != len(vs) or n == 0:
            raise ValueError("ks and vs must be non-empty lists of the same length")
        for k, v in zip(ks, vs):
            if k.is_cuda or v.is_cuda or not (k.is_pinned() and v.is_pinned()):
                raise ValueError("ks and vs must be pinned CPU tensors")
            if k.dtype != torch.bfloat16 or v.dtype != torch.bfloat16 or k.shape != v.shape or k.dim() != 3:
                raise ValueError("each k, v must be bf16 [L, Hkv, d] of the same shape")
            if not (k.is_contiguous() and v.is_contiguous()):
                raise ValueError("ks and vs must be contiguous")
        kp = (_vp * n)(*[k.data_ptr() for k in ks])
        vp = (_vp * n)(*[v.data_ptr() for v in vs])
        lens = (ctypes.c_int32 * n)(*[k.shape[0] for k in ks])
        ids = (ctypes.c_int32 * n)()
        _check(lib().attuner_register_artifacts_host(self.handle, n, kp, vp, lens, self._s(stream), ids))
        return list(ids)

    def pool_reset(self) -> None:
        _check(lib().attuner_pool_reset(self.handle))

    def _p(self, t, name, dtype=torch.bfloat16):
        return _ptr(t, name, dtype, self.device)

    def _s(self, stream):
        return _stream(stream, self.device)

    @staticmethod
    def _csr(reqs):
        # int32 arrays of the flattened items and their offsets (array.array fills
        # them in C; ctypes views their buffers without copying)
        flat = array.array("i", itertools.chain.from_iterable(reqs))
        if not flat:
            flat.append(0)
        offs = array.array("i", [0])
        offs.extend(itertools.accumulate(len(r) for r in reqs))
        c_flat = (ctypes.c_int32 * len(flat)).from_buffer(flat)
        c_offs = (ctypes.c_int32 * len(offs)).from_buffer(offs)
        return (flat, offs), c_flat, c_offs

    def assemble(self, requests: Sequence[Sequence[int]]) -> Plan:
        reqs = [list(map(int, r)) for r in requests]
        keep, ids, off_arr = self._csr(reqs)
        h = ctypes.c_void_p()
        _check(lib().attuner_assemble(self.handle, ids, off_arr, len(reqs), ctypes.byref(h)))
        return Plan(self, h, reqs)

    def assemble_layout(self, layouts: Sequence[Sequence[int]]) -> Plan:
        """Plans of prompt layouts: per request, items in prompt order, item >= 0
        an artifact id, item < 0 an online span of -item tokens (the online
        rows after the last item form the final span)."""
        reqs = [list(map(int, r)) for r in layouts]
        keep, items, off_arr = self._csr(reqs)
        h = ctypes.c_void_p()
        _check(lib().attuner_assemble_layout(self.handle, items, off_arr, len(reqs), ctypes.byref(h)))
        return Plan(self, h, [[a for a in r if a >= 0] for r in reqs])

    # --- compute
    def q_project(self, plan: Plan, x, w_q, lora_a, lora_b, s: float, q_norm_w, S_kv: Optional[int] = None,
                  out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
        n_req, S, _ = x.shape
        S_kv = S if S_kv is None else S_kv
        r = 0 if lora_a is None else lora_a.shape[0]
        if out is None:
            out = torch.empty(n_req, S, self.cfg.n_q_heads, self.cfg.head_dim, dtype=torch.bfloat16, device=x.device)
        _check(lib().attuner_q_project(self.handle, plan.handle, self._p(x, "x"), self._p(w_q, "w_q"),
                                       self._p(lora_a, "lora_a"), self._p(lora_b, "lora_b"), r, float(s),
                                       self._p(q_norm_w, "q_norm_w"), S, S_kv, self._p(out, "out"), self._s(stream)))
        return out

    def kv_project(self, plan: Plan, x, w_k, w_v, k_norm_w, suffix_k, suffix_v, stream=None) -> None:
        """Write the new suffix tokens' K and V (the last S token rows of each
        request in suffix_k / suffix_v [n_req, S_kv, Hkv, d]) from x [n_req, S, hidden]."""
        n_req, S, hidden = x.shape
        S_kv = suffix_k.shape[1]
        if suffix_k.shape != suffix_v.shape or suffix_k.shape[0] != n_req:
            raise ValueError("suffix_k and suffix_v must both be [n_req, S_kv, Hkv, d]")
        _check(lib().attuner_kv_project(self.handle, plan.handle, self._p(x, "x"), self._p(w_k, "w_k"), self._p(w_v, "w_v"),
                                        self._p(k_norm_w, "k_norm_w"), S, S_kv, self._p(suffix_k, "suffix_k"),
                                        self._p(suffix_v, "suffix_v"), self._s(stream)))

    def attend(self, plan: Plan, q, suffix_k, suffix_v, out: Optional[torch.Tensor] = None,
               lse: Optional[torch.Tensor] = None, want_lse: bool = True, stream=None):
        n_req, S, Hq, d = q.shape
        S_kv = suffix_k.shape[1]
        if out is None:
            out = torch.empty_like(q)
        if lse is None and want_lse:
            lse = torch.empty(n_req, S, Hq, dtype=torch.float32, device=q.device)
        _check(lib().attuner_attend(self.handle, plan.handle, self._p(q, "q"), self._p(suffix_k, "suffix_k"),
                                    self._p(suffix_v, "suffix_v"), S, S_kv, self._p(out, "out"),
                                    self._p(lse, "lse", torch.float32), self._s(stream)))
        return out, lse

    def attend_static_scratch(self, plan: Plan, q, suffix_k, suffix_v, out: Optional[torch.Tensor] = None,
                              lse: Optional[torch.Tensor] = None, want_lse: bool = True, stream=None):
        """attend() without any allocation inside the library (fixed device scratch)."""
        n_req, S, Hq, d = q.shape
        S_kv = suffix_k.shape[1]
        if out is None:
            out = torch.empty_like(q)
        if lse is None and want_lse:
            lse = torch.empty(n_req, S, Hq, dtype=torch.float32, device=q.device)
        _check(lib().attuner_attend_static_scratch(self.handle, plan.handle, self._p(q, "q"),
                                                   self._p(suffix_k, "suffix_k"), self._p(suffix_v, "suffix_v"), S,
                                                   S_kv, self._p(out, "out"), self._p(lse, "lse", torch.float32),
                                                   self._s(stream)))
        return out, lse

    def rotate_keys(self, plan: Plan, stream=None) -> None:
        """Rotate the plan's artifact keys (registered before RoPE) to their
        assembled positions; later attention calls with the plan read them."""
        _check(lib().attuner_plan_rotate_keys(self.handle, plan.handle, self._s(stream)))

    def attend_ape(self, plan: Plan, q, suffix_k, suffix_v, temperature: float = 0.9, scale: float = 0.9,
                   out: Optional[torch.Tensor] = None, lse: Optional[torch.Tensor] = None, want_lse: bool = True,
                   stream=None):
        """Context (logits / temperature) and online attention combined by
        calibrated log-sum-exp terms (scale on the context's)."""
        n_req, S, Hq, d = q.shape
        S_kv = suffix_k.shape[1]
        if out is None:
            out = torch.empty_like(q)
        if lse is None and want_lse:
            lse = torch.empty(n_req, S, Hq, dtype=torch.float32, device=q.device)
        _check(lib().attuner_attend_ape(self.handle, plan.handle, self._p(q, "q"), self._p(suffix_k, "suffix_k"),
                                        self._p(suffix_v, "suffix_v"), S, S_kv, float(temperature), float(scale),
                                        self._p(out, "out"), self._p(lse, "lse", torch.float32), self._s(stream)))
        return out, lse

    def query_attend(self, plan: Plan, x, w_q, lora_a, lora_b, s: float, q_norm_w, suffix_k, suffix_v,
                     out: Optional[torch.Tensor] = None, lse: Optional[torch.Tensor] = None,
                     want_lse: bool = True, stream=None):
        n_req, S, _ = x.shape
        S_kv = suffix_k.shape[1]
        r = 0 if lora_a is None else lora_a.shape[0]
        if out is None:
            out = torch.empty(n_req, S, self.cfg.n_q_heads, self.cfg.head_dim, dtype=torch.bfloat16, device=x.device)
        if lse is None and want_lse:
            lse = torch.empty(n_req, S, self.cfg.n_q_heads, dtype=torch.float32, device=x.device)
        _check(lib().attuner_query_attend(self.handle, plan.handle, self._p(x, "x"), self._p(w_q, "w_q"),
                                          self._p(lora_a, "lora_a"), self._p(lora_b, "lora_b"), r, float(s),
                                          self._p(q_norm_w, "q_norm_w"), self._p(suffix_k, "suffix_k"),
                                          self._p(suffix_v, "suffix_v"), S, S_kv, self._p(out, "out"),
                                          self._p(lse, "lse", torch.float32), self._s(stream)))
        return out, lse

    def query_attend_host(self, plan: Plan, x_host, w_q, lora_a, lora_b, s: float, q_norm_w, suffix_k, suffix_v,
                          k_new_host=None, v_new_host=None, out_host: Optional[torch.Tensor] = None,
                          lse_host: Optional[torch.Tensor] = None, stream=None):
        """attuner_query_attend_host: x_host [n_req, S, hidden], k_new_host / v_new_host
        [n_req, S, Hkv, d] (or None) and out_host / lse_host are CPU tensors (pinned for
        asynchronous copies); suffix_k / suffix_v [n_req, S_kv, Hkv, d] and the weights are
        on the device.  The outputs are valid once `stream` has run the call."""
        n_req, S, _ = x_host.shape
        S_kv = suffix_k.shape[1]
        r = 0 if lora_a is None else lora_a.shape[0]
        if (k_new_host is None) != (v_new_host is None):
            raise ValueError("k_new_host and v_new_host must both be given or both be None")
        if k_new_host is not None and (k_new_host.shape != v_new_host.shape or k_new_host.shape[:2] != (n_req, S)):
            raise ValueError("k_new_host and v_new_host must be [n_req, S, Hkv, d]")
        if out_host is None:
            out_host = torch.empty(n_req, S, self.cfg.n_q_heads, self.cfg.head_dim, dtype=torch.bfloat16,
                                   pin_memory=True)
        _check(lib().attuner_query_attend_host(
            self.handle, plan.handle, _host_ptr(x_host, "x_host"), self._p(w_q, "w_q"), self._p(lora_a, "lora_a"),
            self._p(lora_b, "lora_b"), r, float(s), self._p(q_norm_w, "q_norm_w"),
            _host_ptr(k_new_host, "k_new_host"), _host_ptr(v_new_host, "v_new_host"),
            self._p(suffix_k, "suffix_k"), self._p(suffix_v, "suffix_v"), S, S_kv, _host_ptr(out_host, "out_host"),
            _host_ptr(lse_host, "lse_host", torch.float32), self._s(stream)))
        return out_host, lse_host

    # --- misc
    def pool_tensors(self):
        """(K pool, V pool) as torch views [pool_blocks, Hkv, 64, d] of the library's memory, and blocks used."""
        k = ctypes.c_void_p()
        v = ctypes.c_void_p()
        used = ctypes.c_int32()
        cap = ctypes.c_int32()
        _check(lib().attuner_pool_info(self.handle, ctypes.byref(k), ctypes.byref(v), ctypes.byref(used),
                                       ctypes.byref(cap)))
        shape = (cap.value, self.cfg.n_kv_heads, BLOCK_TOKENS, self.cfg.head_dim)
        return _wrap(k.value, shape, self.device), _wrap(v.value, shape, self.device), used.value

    def sync_status(self, stream=None) -> int:
        """Synchronise and return the device status (0 = OK) without raising."""
        return lib().attuner_sync_status(self.handle, self._s(stream))

    def set_option(self, option: int, value: int):
        _check(lib().attuner_set_option(self.handle, option, int(value)))

    def last_launch_count(self) -> int:
        return lib().attuner_last_launch_count(self.handle)


def _wrap(ptr: int, shape, device) -> torch.Tensor:
    """A non-owning torch view of library-owned bf16 device memory."""
    n = 1
    for s in shape:
        n *= s

    class _Arr:
        __cuda_array_interface__ = {
            "shape": (n,), "typestr": "<i2", "data": (ptr, False), "version": 3, "strides": None,
        }

    t = torch.as_tensor(_Arr(), device=device)
    return t.view(torch.bfloat16).view(*shape)
