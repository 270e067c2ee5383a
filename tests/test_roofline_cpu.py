"""The algorithmic byte count behind every reported roofline fraction, checked
against an independent count: the element counts of the model's tensors (the
list the generator, the oracle and the library all consume), E twice (the
draft head's LM-head pass needs the backbone token first, Eq. 3-5), and the
KV entries read and written.  CPU only."""
import math

import pytest

from paper_2605_27255_gb300 import roofline, synth


@pytest.mark.parametrize("shape", [synth.TINY, synth.B4, synth.B9])
def test_weight_bytes_equal_the_tensor_list(shape):
    shapes = synth.tensor_shapes(shape)
    streamed = sum(math.prod(d) for n, d in shapes.items() if n not in ("E", "x_pad"))
    # x_pad is read only for a PAD slot (a gather of H values), E twice per step
    assert roofline.weight_params(shape) == streamed
    e = roofline.esize(shape)
    step0 = roofline.step_bytes(shape, 1, 0)
    kv0 = 2 * roofline.kv_entry_bytes(shape)  # one entry read (the new one), one written
    assert step0 == (streamed + 2 * shape.V * shape.H) * e + kv0


def test_kv_entry_bytes_closed_form():
    # 4B: (36 backbone + 1 MTP) layers x K,V x 8 heads x 128 dims x 2 bytes
    assert roofline.kv_entry_bytes(synth.B4) == 37 * 2 * 8 * 128 * 2 == 151552
    # Tiny (fp32): (2 + 1) x 2 x 2 x 64 x 4
    assert roofline.kv_entry_bytes(synth.TINY) == 3 * 2 * 2 * 64 * 4


def test_step_bytes_scale_with_batch_and_context():
    s = synth.B4
    w = (roofline.weight_params(s) + 2 * s.V * s.H) * 2
    kv = roofline.kv_entry_bytes(s)
    # weights once per step whatever the batch; B x (ctx + 1) entries read, B written
    assert roofline.step_bytes(s, 16, 530.0) == w + 16 * 531.0 * kv + 16 * kv
    assert roofline.step_bytes(s, 4, 15872.0) - roofline.step_bytes(s, 4, 15871.0) == 4 * kv
    # the 4B weights with E twice: about 9.12 GB
    assert 9.10e9 < w < 9.13e9


@pytest.mark.parametrize("shape", [synth.TINY, synth.B4, synth.B9])
def test_regular_step_bytes_are_the_backbone_part_of_the_pair_step(shape):
    """Regular decoding moves the backbone blocks, the final norm and E once;
    the pair step adds the compressor, the MTP input projection and block, the
    confidence head, E a second time and the MTP block's cache entries."""
    H, e = shape.H, roofline.esize(shape)
    comp = H * 2 * H + (H * H if shape.compressor == "mlp" else H)
    mtp = 2 * H + H * 2 * H + (roofline.block_params(shape) if shape.mtp_block else 0) + H
    conf = 2 * H + H * 2 * H + H
    mtp_entry = (2 * shape.n_kv * shape.d_h * e) if shape.mtp_block else 0
    for B, ctx in ((1, 0.0), (4, 100.0), (16, 530.5)):
        extra = (comp + mtp + conf + shape.V * H) * e + B * (ctx + 2) * mtp_entry
        assert roofline.step_bytes(shape, B, ctx) - roofline.regular_step_bytes(shape, B, ctx) == pytest.approx(extra)
    # 4B, written out: a block holds 2*2560 norm + (4096 + 2*1024)*2560 QKV +
    # 2560*4096 O + 3*9728*2560 SwiGLU = 100,930,560 parameters; 36 of them,
    # the final norm and E (151936 x 2560) in bf16, plus one entry read and one
    # written of 36 x K,V x 8 heads x 128 dims x 2 bytes
    if shape is synth.B4:
        w = (36 * 100_930_560 + 2560 + 151_936 * 2560) * 2
        assert w == 8_044_917_760
        assert roofline.regular_step_bytes(shape, 1, 0.0) == w + 2 * 36 * 2 * 8 * 128 * 2


@pytest.mark.parametrize("shape", [synth.TINY, synth.B4, synth.B9])
def test_prefill_flops_equal_the_tensor_list(shape):
    """A pair prefill multiplies every matrix of the compressor, the backbone
    blocks and the MTP head at each position, attends causally (q.k and p.v
    per earlier-or-same position, every cached block), and runs the heads
    (E twice, the confidence matrices) once."""
    shapes = synth.tensor_shapes(shape)
    per_pos = sum(math.prod(d) for n, d in shapes.items() if ".W" in n and not n.startswith("conf."))
    heads = sum(math.prod(d) for n, d in shapes.items() if n.startswith("conf.W")) + 2 * math.prod(shapes["E"])
    layers = shape.L + (1 if shape.mtp_block else 0)
    for B, N in ((1, 1), (2, 7), (1, 8192)):
        attn = sum(layers * shape.n_q * shape.d_h * 2 * (j + 1) for j in range(N))
        assert roofline.prefill_flops(shape, B, N) == pytest.approx(2 * B * (N * per_pos + attn + heads), rel=1e-12)
