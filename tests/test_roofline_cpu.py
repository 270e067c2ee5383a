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
