"""The Python binding's argument marshalling, on the CPU with stand-ins.

The binding only turns tensors into device pointers and streams into handles.
These tests drive it with stand-in tensors and streams and a recording stand-in
for the library, so no GPU is needed: a tensor or a stream on another device
than the context's is refused before the library is called (a pointer into
another GPU's memory, or another GPU's stream, would otherwise reach a kernel),
and matching arguments reach the C entry point in the order the header gives.
"""
from __future__ import annotations

import ctypes

import pytest
import torch

from paper_2609_36722_gb300 import attuner as A


class FakeTensor:
    def __init__(self, shape, dtype=torch.bfloat16, device="cuda:0", ptr=0x1000, contiguous=True):
        self.shape = tuple(shape)
        self.dtype = dtype
        self.device = torch.device(device)
        self.is_cuda = self.device.type == "cuda"
        self._ptr = ptr
        self._contiguous = contiguous

    def is_contiguous(self):
        return self._contiguous

    def data_ptr(self):
        return self._ptr

    def dim(self):
        return len(self.shape)


class FakeStream:
    def __init__(self, device="cuda:0", handle=0x77):
        self.device = torch.device(device)
        self.cuda_stream = handle


class RecordingLib:
    def __init__(self):
        self.calls = []

    def attuner_last_error(self):
        return b"recorded"

    def __getattr__(self, name):
        if not name.startswith("attuner_"):
            raise AttributeError(name)

        def fn(*args):
            self.calls.append((name, args))
            return 0
        return fn


@pytest.fixture
def ctx(monkeypatch):
    fake = RecordingLib()
    monkeypatch.setattr(A, "_LIB", fake)
    c = object.__new__(A.Context)
    c.handle = ctypes.c_void_p(0x42)
    c.cfg = A.Config(256, 4, 2, 64, 64, 10, 1.0e6, 1.0e-6, 0)
    c.device = torch.device("cuda", 0)
    plan = object.__new__(A.Plan)
    plan.handle = ctypes.c_void_p(0x43)
    yield c, plan, fake
    c.handle = None         # stand-in handles: nothing for the real library to destroy or free
    plan.handle = None


def _attend_args(dev_q="cuda:0", dev_k="cuda:0"):
    q = FakeTensor((2, 3, 4, 64), device=dev_q, ptr=0x1000)
    sk = FakeTensor((2, 5, 2, 64), device=dev_k, ptr=0x2000)
    sv = FakeTensor((2, 5, 2, 64), device=dev_k, ptr=0x3000)
    out = FakeTensor((2, 3, 4, 64), ptr=0x4000)
    lse = FakeTensor((2, 3, 4), dtype=torch.float32, ptr=0x5000)
    return q, sk, sv, out, lse


def test_matching_arguments_reach_the_entry_point(ctx):
    c, plan, fake = ctx
    q, sk, sv, out, lse = _attend_args()
    c.attend(plan, q, sk, sv, out=out, lse=lse, stream=FakeStream())
    name, args = fake.calls[-1]
    assert name == "attuner_attend"
    # ctx, plan, q, suffix_k, suffix_v, S, S_kv, out, lse, stream
    assert args[2:] == (0x1000, 0x2000, 0x3000, 3, 5, 0x4000, 0x5000, 0x77)


@pytest.mark.parametrize("where", ["q", "suffix"])
def test_tensor_on_another_device_is_refused(ctx, where):
    c, plan, fake = ctx
    q, sk, sv, out, lse = _attend_args(dev_q="cuda:1" if where == "q" else "cuda:0",
                                       dev_k="cuda:1" if where == "suffix" else "cuda:0")
    with pytest.raises(ValueError, match="cuda:1"):
        c.attend(plan, q, sk, sv, out=out, lse=lse, stream=FakeStream())
    assert fake.calls == []


def test_stream_of_another_device_is_refused(ctx):
    c, plan, fake = ctx
    q, sk, sv, out, lse = _attend_args()
    with pytest.raises(ValueError, match="stream"):
        c.attend(plan, q, sk, sv, out=out, lse=lse, stream=FakeStream("cuda:1"))
    assert fake.calls == []


def test_wrong_dtype_layout_or_host_memory_is_refused(ctx):
    c, plan, fake = ctx
    q, sk, sv, out, lse = _attend_args()
    for bad in (FakeTensor(q.shape, dtype=torch.float16), FakeTensor(q.shape, contiguous=False),
                FakeTensor(q.shape, device="cpu")):
        with pytest.raises(ValueError):
            c.attend(plan, bad, sk, sv, out=out, lse=lse, stream=FakeStream())
    with pytest.raises(ValueError):
        c.attend(plan, q, sk, sv, out=out, lse=FakeTensor(lse.shape, dtype=torch.bfloat16), stream=FakeStream())
    assert fake.calls == []


def test_a_failing_status_raises_with_the_library_message(ctx, monkeypatch):
    c, plan, fake = ctx
    monkeypatch.setattr(fake, "attuner_set_option", lambda *a: A.ERR_INVALID_ARG, raising=False)
    with pytest.raises(A.AttunerError, match="recorded") as e:
        c.set_option(A.OPT_SPLIT_BLOCKS, 3)
    assert e.value.status == A.ERR_INVALID_ARG
