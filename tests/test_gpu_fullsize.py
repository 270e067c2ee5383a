"""Full-size parity: the 4B-class and 9B-class shapes of the benchmark, through
the same C-ABI path and kernels that bench.py times, against the fp64 oracle
(forced replay; short prompts so that the oracle finishes in seconds).

The weights are generated on the GPU (the seeded generator is bit-identical
on CPU and GPU, which test_generator_cpu_equals_gpu checks) and copied to the
host for the oracle.
"""
import numpy as np
import pytest
import torch

from paper_2605_27255_gb300 import synth
from parity_util import run_forced_replay

pytestmark = pytest.mark.gpu


def test_generator_cpu_equals_gpu():
    for name, shape, std, dt in (("blk.Wq", (3, 1000, 17), 0.02, torch.bfloat16),
                                 ("E", (4096, 33), 0.02, torch.float32),
                                 ("kv.K", (2, 777), 1.0, torch.float32)):
        a = synth.gen_tensor(5, name, shape, std, dt, "cpu")
        b = synth.gen_tensor(5, name, shape, std, dt, "cuda").cpu()
        assert torch.equal(a.view(torch.int16) if dt == torch.bfloat16 else a,
                           b.view(torch.int16) if dt == torch.bfloat16 else b)
    p0 = synth.gen_prompts(3, 50, 151936, seed=1, device="cpu")
    p1 = synth.gen_prompts(3, 50, 151936, seed=1, device="cuda").cpu()
    assert torch.equal(p0, p1)


def _weights(shape):
    w = synth.gen_weights(shape, seed=0, device="cuda")
    host = {k: v.cpu() for k, v in w.items()}
    return w, host


@pytest.fixture(scope="module")
def w4b():
    w, host = _weights(synth.B4)
    yield w, host
    del w
    torch.cuda.empty_cache()


def test_4b_b1_forced_replay(w4b):
    """4b-b1 launch configuration (B=1, bf16, 36 layers, V=151936)."""
    w, host = w4b
    prompts = synth.gen_prompts(1, 64, synth.B4.V, seed=1).numpy()
    st = run_forced_replay(synth.B4, w, prompts, 6, oracle_weights=host)
    assert st.tok_checked >= 0.8 * st.tok_total
    assert st.max_logit_err < 2e-2


def test_4b_b4_forced_replay(w4b):
    """4b-b4: four sequences in one step (4-sequence GEMV tile)."""
    w, host = w4b
    prompts = synth.gen_prompts(4, 20, synth.B4.V, seed=3).numpy()
    st = run_forced_replay(synth.B4, w, prompts, 3, oracle_weights=host, force=1)
    assert st.tok_checked >= 0.8 * st.tok_total


def test_4b_b16_forced_replay(w4b):
    """4b-b16: sixteen sequences, tcgen05 projections and tensor-core attention."""
    w, host = w4b
    prompts = synth.gen_prompts(16, 8, synth.B4.V, seed=5).numpy()
    st = run_forced_replay(synth.B4, w, prompts, 2, oracle_weights=host, force=1)
    assert st.tok_checked >= 0.8 * st.tok_total
    assert st.max_logit_err < 2e-2


def test_9b_b1_forced_replay():
    """9B-class shapes (H=4096, F=12288)."""
    w, host = _weights(synth.B9)
    prompts = synth.gen_prompts(1, 16, synth.B9.V, seed=2).numpy()
    st = run_forced_replay(synth.B9, w, prompts, 3, oracle_weights=host, tau=0.3)
    assert st.tok_checked >= 0.8 * st.tok_total
    del w
    torch.cuda.empty_cache()
