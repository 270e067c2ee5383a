"""Failure detection on the GPU, with failures made on the host or bounded on
the device (nothing here faults, traps or hangs a GPU):

* a bounded device wait given a short limit on an mbarrier that nothing
  completes gives up, records its site and is reported as PIPO_ECUDA; the
  same wait on a completed barrier reports nothing; the device stays usable;
* an out-of-memory on the k-th device allocation of pipo_init (injected on
  the host, PIPO_TEST_FAIL_ALLOC) returns PIPO_ENOMEM, frees everything
  allocated before it (device memory back to where it was, repeatedly), and
  the next init succeeds;
* a missing weight tensor or inconsistent shapes are EINVAL with nothing
  left allocated.
"""
import time

import numpy as np
import pytest
import torch

from oracle import oracle as O
from paper_2605_27255_gb300 import capi, synth

pytestmark = pytest.mark.gpu

MID = synth.ModelShape("mid", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1376, V=5003,
                       compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1e6, tau=0.5)


def _free_bytes():
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info()[0]


def _tiny_step_matches_oracle():
    s = synth.TINY
    w = synth.gen_weights(s, seed=0)
    prompt = synth.gen_prompts(1, 8, s.V, seed=1).numpy()
    g = capi.Pipo(s, w, max_batch=1, max_ctx=16, debug=True)
    try:
        g.prefill(prompt)
        o = O.State(O.Model(s, w, max_ctx=16), 1).prefill(prompt, tau=s.tau)
        assert np.abs(g.debug()["logits_b"][0] - o["logits_b"][0]).max() < 1e-4
    finally:
        g.close()


def test_bounded_wait_gives_up_and_reports_its_site():
    torch.cuda.init()
    t0 = time.perf_counter()
    st, msg, info = capi.pipo_selftest_wait(0, 1_000_000)  # 1 ms limit, never signalled
    assert time.perf_counter() - t0 < 5.0
    assert st == capi.PIPO_ECUDA, (st, msg)
    assert info[0] == 90 and "wait site 90" in msg
    # a completed barrier: no timeout, and the error word was cleared by the first call
    st, msg, info = capi.pipo_selftest_wait(1, 1_000_000)
    assert st == capi.PIPO_OK and info == [0, 0, 0, 0], (st, msg, info)
    # limits outside (0, 10 s] are refused before any launch
    assert capi.pipo_selftest_wait(0, 0)[0] == capi.PIPO_EINVAL
    # the context survives: a decode runs and matches the oracle
    _tiny_step_matches_oracle()


def test_injected_allocation_failure_frees_everything(monkeypatch):
    w = synth.gen_weights(MID, seed=1, device="cuda")
    kw = dict(max_batch=16, max_ctx=4096)  # about 100 MB of KV cache: a leak would show
    before = _free_bytes()
    n_ok = None
    for k in range(1, 200):
        monkeypatch.setenv("PIPO_TEST_FAIL_ALLOC", str(k))
        try:
            g = capi.Pipo(MID, w, **kw)
        except capi.PipoError as e:
            assert e.status == capi.PIPO_ENOMEM, str(e)
            assert f"injected failure of device allocation {k}" in str(e)
            continue
        n_ok = k  # k is past the last allocation: this init succeeded
        g.close()
        break
    assert n_ok is not None and n_ok > 20
    # repeated failures late in the sequence (after the caches) leak nothing
    for _ in range(3):
        for k in (n_ok - 1, n_ok // 2, 2):
            monkeypatch.setenv("PIPO_TEST_FAIL_ALLOC", str(k))
            with pytest.raises(capi.PipoError) as e:
                capi.Pipo(MID, w, **kw)
            assert e.value.status == capi.PIPO_ENOMEM
    after = _free_bytes()
    assert abs(before - after) < 32 << 20, (before, after)
    monkeypatch.delenv("PIPO_TEST_FAIL_ALLOC")
    g = capi.Pipo(MID, w, **kw)
    g.close()


def test_bad_weights_and_shapes_are_einval():
    w = synth.gen_weights(MID, seed=2, device="cuda")
    before = _free_bytes()
    for missing in ("E", "blk.Wdown", "mtp.W_fc", "conf.norm"):
        ww = {k: v for k, v in w.items() if k != missing}
        with pytest.raises(capi.PipoError) as e:
            capi.Pipo(MID, ww, max_batch=2, max_ctx=64)
        assert e.value.status == capi.PIPO_EINVAL and "missing weight tensor" in str(e.value)
    for bad in (dict(n_kv=3), dict(d_h=96), dict(H=500)):
        with pytest.raises(capi.PipoError) as e:
            capi.Pipo(MID.with_(**bad), w, max_batch=2, max_ctx=64)
        assert e.value.status == capi.PIPO_EINVAL
    assert abs(before - _free_bytes()) < 16 << 20
