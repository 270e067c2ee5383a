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


def test_every_context_entry_point_rejects_a_null_context(lib):
    """Status, not a crash: each entry point that takes a context returns
    EINVAL for NULL (before any CUDA call), with a message."""
    capi.load()
    L = capi.load()
    null = None
    ib = (C.c_int32 * 4)()
    fb = (C.c_float * 4)()
    calls = {
        "pipo_prefill": lambda: L.pipo_prefill(null, 1, ib, 1, ib, ib, ib),
        "pipo_regular_prefill": lambda: L.pipo_regular_prefill(null, 1, ib, 1, ib, ib, ib),
        "pipo_prefill_slot": lambda: L.pipo_prefill_slot(null, 0, ib, 1, ib, ib),
        "pipo_decode_step": lambda: L.pipo_decode_step(null, None, None),
        "pipo_decode_step_async": lambda: L.pipo_decode_step_async(null, None, None),
        "pipo_decode_steps": lambda: L.pipo_decode_steps(null, 1, None, None),
        "pipo_regular_step": lambda: L.pipo_regular_step(null, None),
        "pipo_regular_step_async": lambda: L.pipo_regular_step_async(null, None),
        "pipo_rollback": lambda: L.pipo_rollback(null, ib),
        "pipo_set_threshold": lambda: L.pipo_set_threshold(null, 0.5, 0),
        "pipo_set_sampler": lambda: L.pipo_set_sampler(null, 1.0, 20, 0.95, 1.5, fb, 1),
        "pipo_set_pending": lambda: L.pipo_set_pending(null, ib),
        "pipo_get_counters": lambda: L.pipo_get_counters(null, None, None),
        "pipo_debug_dump": lambda: L.pipo_debug_dump(null, C.byref(capi.pipo_debug())),
        "pipo_read_cache": lambda: L.pipo_read_cache(null, 0, 0, 1, fb, fb),
        "pipo_load_cache": lambda: L.pipo_load_cache(null, 0, 1, fb, fb),
        "pipo_set_stream": lambda: L.pipo_set_stream(null, None),
        "pipo_describe_step": lambda: L.pipo_describe_step(null, C.create_string_buffer(8), 8),
        "pipo_profile_step": lambda: L.pipo_profile_step(null, 0, None, None, None, ib),
    }
    for name, call in calls.items():
        assert call() == capi.PIPO_EINVAL, name
        assert capi.pipo_last_error(None), name
    assert L.pipo_step_launches(null) == 0
    L.pipo_free(null)  # a no-op


def test_residual_compressor_needs_the_mlp_variant(lib):
    """comp_residual is the residual form of the MLP compressor: with the
    Linear variant the config is invalid (checked before any CUDA call)."""
    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    from paper_2605_27255_gb300 import synth
    L = capi.load()
    w = capi.pipo_weights()
    ctx = C.c_void_p()
    cfg = capi.make_config(synth.TINY.with_(comp_residual=1), 1, 16)  # Tiny: Linear compressor
    assert L.pipo_init(C.byref(cfg), C.byref(w), C.byref(ctx)) == capi.PIPO_EINVAL
    assert "invalid config" in capi.pipo_last_error(None)
    cfg = capi.make_config(synth.TINY.with_(compressor="mlp", comp_residual=1), 1, 16)
    rc = L.pipo_init(C.byref(cfg), C.byref(w), C.byref(ctx))
    assert "invalid config" not in capi.pipo_last_error(None) and not ctx.value  # fails later: no GPU
    assert rc != capi.PIPO_OK


C_PROGRAM = os.path.join(ROOT, "tests", "c", "pipo_c_api.c")


def build_c_program(lib_path):
    """Compile the C99 user program against include/pipo.h and the library
    (the binary goes next to the library, a build output)."""
    import subprocess
    exe = os.path.join(os.path.dirname(lib_path), "pipo_c_api")
    libdir = os.path.dirname(lib_path)
    subprocess.check_call(["gcc", "-std=c99", "-Wall", "-Wextra", "-Werror", "-pedantic", "-I",
                           os.path.join(ROOT, "include"), C_PROGRAM, "-o", exe, "-L", libdir, "-lpipo",
                           "-Wl,-rpath," + libdir])
    return exe


def test_header_is_c99_and_a_c_program_links_and_fails_cleanly_without_a_device(lib):
    """The boundary is usable from C alone: the header compiles as strict C99,
    the program links against the library, and without a device pipo_init
    returns a status that the program reports (exit 2), no crash."""
    import subprocess

    import torch
    if torch.cuda.is_available():
        pytest.skip("a GPU is present")
    exe = build_c_program(build.build())
    r = subprocess.run([exe], capture_output=True, text=True, timeout=120)
    assert r.returncode == 2, (r.returncode, r.stdout, r.stderr)
    assert "pipo_init: status" in r.stdout


def test_every_kernel_unit_is_built():
    """Every .cu file of csrc is a unit of the library build, and every launch
    handle declared in kernel_tables.h is defined by some unit."""
    import glob
    import re as _re
    csrc = os.path.join(ROOT, "paper_2605_27255_gb300", "csrc")
    units = sorted(os.path.basename(p) for p in glob.glob(os.path.join(csrc, "*.cu")))
    assert units == sorted(build.SOURCES)
    decl = _re.findall(r"\b(k_\w+)\(", open(os.path.join(csrc, "kernel_tables.h")).read())
    defs = "".join(open(os.path.join(csrc, u)).read() for u in units)
    for name in set(decl):
        assert _re.search(r"\b" + name + r"\([^;{]*\)\s*\{", defs), f"{name} declared but not defined"


def test_header_compiles_as_cplusplus():
    """The header also compiles as C++ (its extern "C" block), with warnings as errors."""
    import subprocess
    subprocess.check_call(["g++", "-std=c++17", "-Wall", "-Wextra", "-Werror", "-fsyntax-only", "-x", "c++", HEADER])
