"""The residual MLP compressor (comp_residual = 1: z = a + b + W2 SiLU(W1
[a;b])) on the GPU against the oracle, with forced replay: the CUDA-core
(B = 1) and tensor-core (B = 4) projections, position-by-position and
chunked prefill.
"""

import pytest

from paper_2605_27255_gb300 import synth
from parity_util import run_forced_replay

pytestmark = pytest.mark.gpu

MID = synth.ModelShape("mid", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1376, V=5003,
                       compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1e6, tau=0.5, comp_residual=1)


def test_residual_compressor_tiny_fp32():
    s = synth.TINY.with_(compressor="mlp", comp_residual=1)
    w = synth.gen_weights(s, seed=1)
    prompts = synth.gen_prompts(2, 41, s.V, seed=2).numpy()  # odd: the last pair holds PAD
    st = run_forced_replay(s, w, prompts, 8)
    assert st.tok_checked >= 0.5 * st.tok_total


@pytest.mark.parametrize("B", [1, 4])
@pytest.mark.parametrize("rows", [0, 32])
def test_residual_compressor_bf16(monkeypatch, B, rows):
    if rows:
        monkeypatch.setenv("PIPO_PREFILL_ROWS", str(rows))
    w = synth.gen_weights(MID, seed=3)
    prompts = synth.gen_prompts(B, 61, MID.V, seed=4).numpy()
    st = run_forced_replay(MID, w, prompts, 6)
    assert st.tok_checked >= 0.5 * st.tok_total
