"""The C99 user program (tests/c/pipo_c_api.c, only include/pipo.h and the
library) on the GPU: a step before the prefill is ESTATE, an odd prompt's
prefill and 8 decode steps give in-range, self-consistent outputs and the
expected counters.
"""
import subprocess

import pytest

from paper_2605_27255_gb300 import build
from test_capi_cpu import build_c_program

pytestmark = pytest.mark.gpu


def test_c_program_decodes():
    exe = build_c_program(build.build())
    r = subprocess.run([exe], capture_output=True, text=True, timeout=300)
    assert r.returncode == 0, (r.returncode, r.stdout, r.stderr)
    lines = r.stdout.strip().splitlines()
    assert lines[-1] == "ok" and sum(1 for l in lines if l.startswith("position ")) == 9
