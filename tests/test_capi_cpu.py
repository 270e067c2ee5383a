"""CPU checks of the boundary: the library builds for sm_103a, loads, and
exports every entry point that include/pipo.h declares; the binding's struct
layouts match the header's field lists.  No compute calls (no GPU here)."""
import ctypes as C
import os
import re

import pytest

from paper_2605_27255_gb300 import build, capi

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "pipo.h")


def declared_functions():
    src = open(HEADER).read()
    return sorted(set(re.findall(r"PIPO_API\s+[\w\s\*]*?\b(pipo_\w+)\s*\(", src)))


def struct_fields(name):
    src = open(HEADER).read()
    m = re.search(r"typedef struct \{([^{}]*)\}\s*" + name + ";", src)
    body = re.sub(r"/\*.*?\*/", "", m.group(1), flags=re.S)
    fields = []
    for decl in body.split(";"):
        decl = decl.strip()
        if not decl:
            continue
        names = decl.split(None, 1)[1] if decl.split()[0] not in ("const",) else decl.split(None, 2)[2]
        for part in names.split(","):
            fields.append(part.replace("*", "").strip())
    return fields


@pytest.fixture(scope="module")
def lib():
    path = build.build()
    return C.CDLL(path)


def test_every_declared_entry_point_is_exported(lib):
    names = declared_functions()
    assert len(names) >= 15
    for n in names:
        assert hasattr(lib, n), f"{n} declared in pipo.h but not exported"
    assert set(names) == set(capi.SIGNATURES), "binding and header disagree"


def test_struct_layouts_match_header():
    assert [f for f, _ in capi.pipo_config._fields_] == struct_fields("pipo_config")
    assert [f for f, _ in capi.pipo_weights._fields_] == struct_fields("pipo_weights")
    assert [f for f, _ in capi.pipo_debug._fields_] == struct_fields("pipo_debug")


def test_init_error_without_gpu_is_a_status(lib):
    """With no device, pipo_init returns a status and a message; no abort."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    capi.load()
    cfg = capi.pipo_config()
    w = capi.pipo_weights()
    ctx = C.c_void_p()
    rc = capi.load().pipo_init(C.byref(cfg), C.byref(w), C.byref(ctx))
    assert rc == capi.PIPO_EINVAL and not ctx.value
    assert "invalid config" in capi.pipo_last_error(None)


def test_missing_library_fails_loudly(monkeypatch, tmp_path):
    """No fallback: without the CUDA library the binding raises."""
    monkeypatch.setattr(capi, "_lib", None)
    with pytest.raises(RuntimeError, match="not built"):
        capi.load(str(tmp_path / "libpipo.so"))


def test_failed_call_raises_status_error(lib):
    """A non-OK status becomes a PipoError carrying the status and message."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    with pytest.raises(capi.PipoError) as e:
        capi.pipo_op_gemv(1, 0, 16, 10, 12, 16, 1, 16, 0)  # K not a multiple of 8
    assert e.value.status == capi.PIPO_EINVAL
