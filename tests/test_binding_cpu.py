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
    def __init__(self, shape, dtype=torch.bfloat16, device="cuda:0", ptr=0x1000, contiguous=True, pinned=False):
        self.shape = tuple(shape)
        self.dtype = dtype
        self.device = torch.device(device)
        self.is_cuda = self.device.type == "cuda"
        self._ptr = ptr
        self._contiguous = contiguous
        self._pinned = pinned

    def is_contiguous(self):
        return self._contiguous

    def is_pinned(self):
        return self._pinned

    def get_device(self):
        return self.device.index if self.is_cuda else -1

    def data_ptr(self):
        return self._ptr

    def dim(self):
        return len(self.shape)


class FakeStream:
    def __init__(self, device="cuda:0", handle=0x77):
        self.device = torch.device(device)
        self.cuda_stream = handle


class RecordingLib:
    """Records each call after converting every argument through the ctypes
    type the binding declares for it, so a wrong arity, a Python object where a
    pointer belongs or a misspelt attribute fails here as it would in ctypes."""

    def __init__(self):
        self.calls = []

    def attuner_last_error(self):
        return b"recorded"

    def __getattr__(self, name):
        if name not in A.SIGNATURES:
            raise AttributeError(name)
        argtypes, _ = A.SIGNATURES[name]

        def fn(*args):
            assert len(args) == len(argtypes), f"{name}: {len(args)} arguments, header has {len(argtypes)}"
            for i, (a, t) in enumerate(zip(args, argtypes)):
                try:
                    t.from_param(a)
                except (TypeError, ctypes.ArgumentError) as e:
                    raise AssertionError(f"{name} argument {i}: {a!r} is not a {t.__name__}: {e}")
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


def test_host_artifact_load_passes_host_pointers_lengths_and_stream(ctx):
    c, plan, fake = ctx
    ks = [FakeTensor((37, 2, 64), device="cpu", ptr=0x10000, pinned=True),
          FakeTensor((100, 2, 64), device="cpu", ptr=0x20000, pinned=True)]
    vs = [FakeTensor((37, 2, 64), device="cpu", ptr=0x30000, pinned=True),
          FakeTensor((100, 2, 64), device="cpu", ptr=0x40000, pinned=True)]
    ids = c.register_artifacts_host(ks, vs, stream=FakeStream())
    name, args = fake.calls[-1]
    assert name == "attuner_register_artifacts_host"
    assert args[1] == 2
    assert [args[2][i] for i in range(2)] == [0x10000, 0x20000]
    assert [args[3][i] for i in range(2)] == [0x30000, 0x40000]
    assert list(args[4]) == [37, 100]
    assert args[5] == 0x77
    assert ids == [0, 0]     # the stand-in library leaves the id array as allocated


@pytest.mark.parametrize("bad", ["cuda", "pageable", "dtype", "shape", "empty"])
def test_host_artifact_load_refuses_unusable_tensors(ctx, bad):
    c, plan, fake = ctx
    k = FakeTensor((37, 2, 64), device="cpu", pinned=True)
    v = FakeTensor((37, 2, 64), device="cpu", pinned=True)
    if bad == "cuda":
        k = FakeTensor((37, 2, 64))
    elif bad == "pageable":
        v = FakeTensor((37, 2, 64), device="cpu")
    elif bad == "dtype":
        v = FakeTensor((37, 2, 64), dtype=torch.float16, device="cpu", pinned=True)
    elif bad == "shape":
        v = FakeTensor((36, 2, 64), device="cpu", pinned=True)
    with pytest.raises(ValueError):
        c.register_artifacts_host([] if bad == "empty" else [k], [] if bad == "empty" else [v], stream=FakeStream())
    assert fake.calls == []


def test_every_public_method_reaches_its_entry_point(ctx, monkeypatch):
    """Each public method of Context and Plan, called once with matching
    stand-ins, reaches the library with arguments its declared ctypes types
    accept.  A public method missing from this table fails the test, so a new
    method cannot skip the check."""
    c, plan, fake = ctx
    monkeypatch.setattr(A, "_wrap", lambda ptr, shape, device: ("view", ptr, shape))
    plan.ctx = c
    plan.n_req = 2
    plan.requests = [[0], [1]]
    dev = FakeTensor((4,))
    q, sk, sv, out, lse = _attend_args()
    x = FakeTensor((2, 3, 256), ptr=0x6000)
    w = FakeTensor((256, 256), ptr=0x7000)
    la, lb = FakeTensor((8, 256), ptr=0x8000), FakeTensor((256, 8), ptr=0x9000)
    qn = FakeTensor((64,), ptr=0xA000)
    wk, wv = FakeTensor((128, 256), ptr=0xB000), FakeTensor((128, 256), ptr=0xC000)
    kn = FakeTensor((64,), ptr=0xD000)
    hk = FakeTensor((5, 2, 64), device="cpu", pinned=True, ptr=0xE000)
    hv = FakeTensor((5, 2, 64), device="cpu", pinned=True, ptr=0xF000)
    xh = FakeTensor((2, 3, 256), device="cpu", pinned=True, ptr=0x10000)
    kh = FakeTensor((2, 3, 2, 64), device="cpu", pinned=True, ptr=0x11000)
    vh = FakeTensor((2, 3, 2, 64), device="cpu", pinned=True, ptr=0x12000)
    oh = FakeTensor((2, 3, 4, 64), device="cpu", pinned=True, ptr=0x13000)
    lh = FakeTensor((2, 3, 4), dtype=torch.float32, device="cpu", pinned=True, ptr=0x14000)
    st = FakeStream()
    ctx_calls = {
        "register_artifact": (lambda: c.register_artifact(FakeTensor((5, 2, 64)), FakeTensor((5, 2, 64)), stream=st),
                              "attuner_register_artifact"),
        "register_artifacts_host": (lambda: c.register_artifacts_host([hk], [hv], stream=st),
                                    "attuner_register_artifacts_host"),
        "pool_reset": (lambda: c.pool_reset(), "attuner_pool_reset"),
        "assemble": (lambda: c.assemble([[0, 1], []]), "attuner_assemble"),
        "assemble_layout": (lambda: c.assemble_layout([[-16, 0, -5, 1], [0]]), "attuner_assemble_layout"),
        "q_project": (lambda: c.q_project(plan, x, w, la, lb, 2.0, qn, S_kv=5, out=q, stream=st),
                      "attuner_q_project"),
        "kv_project": (lambda: c.kv_project(plan, x, wk, wv, kn, sk, sv, stream=st), "attuner_kv_project"),
        "attend": (lambda: c.attend(plan, q, sk, sv, out=out, lse=lse, stream=st), "attuner_attend"),
        "attend_static_scratch": (lambda: c.attend_static_scratch(plan, q, sk, sv, out=out, lse=lse, stream=st),
                                  "attuner_attend_static_scratch"),
        "query_attend": (lambda: c.query_attend(plan, x, w, la, lb, 2.0, qn, sk, sv, out=q, lse=lse, stream=st),
                         "attuner_query_attend"),
        "query_attend_host": (lambda: c.query_attend_host(plan, xh, w, la, lb, 2.0, qn, sk, sv, kh, vh, out_host=oh,
                                                          lse_host=lh, stream=st), "attuner_query_attend_host"),
        "rotate_keys": (lambda: c.rotate_keys(plan, stream=st), "attuner_plan_rotate_keys"),
        "attend_ape": (lambda: c.attend_ape(plan, q, sk, sv, 0.9, 0.9, out=out, lse=lse, stream=st),
                       "attuner_attend_ape"),
        "pool_tensors": (lambda: c.pool_tensors(), "attuner_pool_info"),
        "sync_status": (lambda: c.sync_status(stream=st), "attuner_sync_status"),
        "set_option": (lambda: c.set_option(A.OPT_SPLIT_BLOCKS, 4), "attuner_set_option"),
        "last_launch_count": (lambda: c.last_launch_count(), "attuner_last_launch_count"),
    }
    plan_calls = {
        "t_art": (lambda: plan.t_art(), "attuner_plan_t_art"),
        "export": (lambda: plan.export(), "attuner_plan_export"),
    }
    ignore = {"for_geometry", "close", "free"}   # a constructor and the two releases (checked last)
    public = {n for n in dir(A.Context) if not n.startswith("_")} - ignore
    assert public == set(ctx_calls), sorted(public ^ set(ctx_calls))
    public_plan = {n for n in dir(A.Plan) if not n.startswith("_")} - ignore
    assert public_plan == set(plan_calls), sorted(public_plan ^ set(plan_calls))
    for method, (call, entry) in {**ctx_calls, **plan_calls}.items():
        n = len(fake.calls)
        call()
        assert [name for name, _ in fake.calls[n:]][-1] == entry, method
    plan.free()
    assert fake.calls[-1][0] == "attuner_plan_free"
    c.close()
    assert fake.calls[-1][0] == "attuner_destroy"
    assert dev.dim() == 1


def test_query_attend_host_refuses_device_or_mismatched_host_buffers(ctx):
    """The host-buffer call takes CPU tensors for the step's inputs and outputs
    and device tensors for the resident state; the wrong kind, or only one of
    the new K/V row buffers, is refused before the library is called."""
    c, plan, fake = ctx
    plan.ctx = c
    plan.n_req = 2
    q, sk, sv, out, lse = _attend_args()
    w = FakeTensor((256, 256), ptr=0x7000)
    qn = FakeTensor((64,), ptr=0xA000)
    xh = FakeTensor((2, 3, 256), device="cpu", pinned=True, ptr=0x10000)
    xd = FakeTensor((2, 3, 256), ptr=0x6000)
    kh = FakeTensor((2, 3, 2, 64), device="cpu", pinned=True, ptr=0x11000)
    oh = FakeTensor((2, 3, 4, 64), device="cpu", pinned=True, ptr=0x13000)
    st = FakeStream()
    with pytest.raises(ValueError):
        c.query_attend_host(plan, xd, w, None, None, 2.0, qn, sk, sv, out_host=oh, stream=st)
    with pytest.raises(ValueError):
        c.query_attend_host(plan, xh, w, None, None, 2.0, qn, sk, sv, kh, None, out_host=oh, stream=st)
    with pytest.raises(ValueError):
        c.query_attend_host(plan, xh, w, None, None, 2.0, qn, sk, sv, out_host=out, stream=st)
    assert fake.calls == []
    c.query_attend_host(plan, xh, w, None, None, 2.0, qn, sk, sv, out_host=oh, stream=st)
    name, args = fake.calls[-1]
    assert name == "attuner_query_attend_host"
    assert args[2] == 0x10000 and args[9] is None and args[10] is None and args[15] == 0x13000
