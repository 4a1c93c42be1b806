"""CPU checks of the C-ABI library: it builds, loads without a GPU, exports
every symbol include/attuner.h declares, and rejects bad arguments on the
host before touching the device."""

import ctypes
import os
import re

import pytest

from conftest import ROOT


def _header_symbols():
    with open(os.path.join(ROOT, "include", "attuner.h")) as f:
        text = f.read()
    return sorted(set(re.findall(r"\b(attuner_[a-z_]+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib():
    from paper_2609_36722_gb300 import build
    build.build()
    import paper_2609_36722_gb300 as pkg
    return pkg.lib()


def test_library_exports_every_declared_symbol(lib):
    import paper_2609_36722_gb300 as pkg
    syms = _header_symbols()
    assert len(syms) >= 15
    assert sorted(pkg.EXPORTS) == syms
    for s in syms:
        assert hasattr(lib, s), s


def test_create_rejects_bad_geometry_on_host(lib):
    import paper_2609_36722_gb300 as pkg
    h = ctypes.c_void_p()
    bad = [
        dict(head_dim=96), dict(head_dim=128, n_q_heads=12, n_kv_heads=8), dict(hidden=100),
        dict(block_tokens=32), dict(pool_blocks=0), dict(n_q_heads=48, n_kv_heads=3),
    ]
    for over in bad:
        f = dict(hidden=256, n_q_heads=4, n_kv_heads=2, head_dim=64, block_tokens=64, pool_blocks=16,
                 rope_theta=1e6, rms_eps=1e-6, device=0)
        f.update(over)
        cfg = pkg.attuner.Config(**f)
        assert lib.attuner_create(ctypes.byref(cfg), ctypes.byref(h)) == pkg.attuner.ERR_INVALID_ARG, over
        assert lib.attuner_last_error() != b""


def test_null_arguments_are_rejected(lib):
    import paper_2609_36722_gb300 as pkg
    E = pkg.attuner.ERR_INVALID_ARG
    assert lib.attuner_create(None, None) == E
    assert lib.attuner_register_artifact(None, None, None, 5, None, None) == E
    assert lib.attuner_assemble(None, None, None, 1, None) == E
    assert lib.attuner_attend(None, None, None, None, None, 1, 1, None, None, None) == E
    assert lib.attuner_set_option(None, 1, 0) == E
    assert lib.attuner_destroy(None) == 0
    assert lib.attuner_plan_free(None) == 0
    assert lib.attuner_last_launch_count(None) == 0


def test_binding_fails_loudly_without_library(tmp_path):
    import paper_2609_36722_gb300 as pkg
    with pytest.raises(ImportError):
        pkg.load_library(str(tmp_path / "missing.so"))


def test_product_path_does_not_import_oracle():
    # the package and its sources never reference the test oracle
    pkg_dir = os.path.join(ROOT, "paper_2609_36722_gb300")
    for dirpath, _, files in os.walk(pkg_dir):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h", ".cpp")):
                with open(os.path.join(dirpath, f)) as fh:
                    src = fh.read()
                assert not re.search(r"^\s*(import|from)\s+oracle\b", src, re.M), f
                assert "oracle/" not in src and "oracle." not in src, f


def test_every_status_entry_point_documents_its_errors():
    # the header states, above each declaration, what the call returns on error
    import re
    with open(os.path.join(ROOT, "include", "attuner.h")) as f:
        src = f.read()
    for m in re.finditer(r"attuner_status\s+(attuner_\w+)\s*\(", src):
        comment = src[:m.start()].rsplit("/*", 1)[-1]
        assert "Errors" in comment, m.group(1)


def test_binding_constants_match_the_header():
    # every status code and option the header defines has the same value in
    # the Python binding (a drift would silently pass the wrong option)
    from paper_2609_36722_gb300 import attuner as A
    with open(os.path.join(ROOT, "include", "attuner.h")) as f:
        text = f.read()
    defs = {m.group(1): int(m.group(2)) for m in
            re.finditer(r"^#define ATTUNER_((?:OK|ERR_[A-Z_]+|OPT_[A-Z_]+))\s+\(?(-?\d+)\)?", text, re.M)}
    assert len([k for k in defs if k.startswith("OPT_")]) >= 9 and len([k for k in defs if k.startswith("ERR_")]) >= 7
    for name, value in defs.items():
        assert getattr(A, name) == value, name
    assert A.BLOCK_TOKENS == int(re.search(r"#define ATTUNER_BLOCK_TOKENS\s+(\d+)", text).group(1))
