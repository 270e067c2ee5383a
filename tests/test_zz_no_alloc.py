"""The LM-head argmax entry point for callers that cannot allocate device
memory (pipo_op_lm_head_argmax_noalloc) against the entry point that takes
caller scratch, through the C ABI.  Kept in the last-collected file."""
import pytest
import torch

from paper_2605_27255_gb300 import capi

pytestmark = pytest.mark.gpu


def _inputs(seed, V, H, B):
    g = torch.Generator().manual_seed(seed)
    E = (torch.randn(V, H, generator=g) * 0.05).to(torch.bfloat16).cuda()
    gam = (1.0 + 0.1 * torch.randn(H, generator=g)).to(torch.bfloat16).cuda()
    h = (torch.randn(B, H, generator=g) * 3).cuda()
    return E, gam, h


def _with_scratch(E, gam, h, V, H, B, stream):
    tok = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    logits = torch.empty(B, V, device="cuda")
    scratch = torch.empty(B, dtype=torch.int64, device="cuda")
    capi.pipo_op_lm_head_argmax(1, E.data_ptr(), V, H, h.data_ptr(), gam.data_ptr(), 1e-6, B, tok.data_ptr(),
                                logits.data_ptr(), scratch.data_ptr(), 8 * B, stream)
    return tok, logits


def _no_alloc(E, gam, h, V, H, B, stream):
    tok = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    logits = torch.empty(B, V, device="cuda")
    capi.pipo_op_lm_head_argmax_noalloc(1, E.data_ptr(), V, H, h.data_ptr(), gam.data_ptr(), 1e-6, B,
                                        tok.data_ptr(), logits.data_ptr(), stream)
    return tok, logits


def test_no_alloc_lm_head_matches_scratch_version_twice():
    V, H = 30011, 512
    stream = torch.cuda.current_stream().cuda_stream
    # two calls in a row on different inputs: the shared scratch must be
    # cleared by each call, not carry the previous call's keys
    for seed, B in ((1, 5), (2, 64)):
        E, gam, h = _inputs(seed, V, H, B)
        t_ref, l_ref = _with_scratch(E, gam, h, V, H, B, stream)
        t_na, l_na = _no_alloc(E, gam, h, V, H, B, stream)
        torch.cuda.synchronize()
        assert (l_na - l_ref).abs().max().item() <= 1e-4
        assert torch.equal(t_na, t_ref)
        assert int(t_na.min()) >= 0


def test_no_alloc_lm_head_rejects_more_than_64_sequences():
    with pytest.raises(capi.PipoError) as e:
        capi.pipo_op_lm_head_argmax_noalloc(1, 16, 8, 16, 16, 0, 1e-6, 65, 16, 0, 0)
    assert e.value.status == capi.PIPO_EINVAL
    assert "at most 64" in str(e.value)
