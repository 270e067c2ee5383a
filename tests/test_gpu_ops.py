"""Kernel-level GPU tests through the C ABI (pipo_op_*): each kernel against a
float64 evaluation of the same operation on the same inputs."""
import numpy as np
import pytest
import torch

from paper_2605_27255_gb300 import capi

pytestmark = pytest.mark.gpu


def _run_gemv(dtype, mode, N, K, B, seed=0):
    g = torch.Generator().manual_seed(seed)
    rows = 2 * N if mode else N
    W = torch.randn(rows, K, generator=g) * 0.05
    W = W.to(torch.bfloat16) if dtype == 1 else W
    x = torch.randn(B, K, generator=g)
    Wd, xd = W.cuda(), x.cuda()
    y = torch.full((B, N), float("nan"), device="cuda")
    capi.pipo_op_gemv(dtype, mode, Wd.data_ptr(), N, K, xd.data_ptr(), B, y.data_ptr(),
                      torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    ref = x.double() @ W.double().t()
    if mode:
        gate, up = ref[:, 0::2], ref[:, 1::2]
        ref = gate * torch.sigmoid(gate) * up
    return y.cpu().double(), ref


@pytest.mark.parametrize("dtype", [0, 1])
@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("N,K", [(2560, 2560), (333, 4096), (1000, 1376), (7, 520), (4096, 256)])
@pytest.mark.parametrize("B", [1, 3, 6])
def test_gemv_matches_float64(dtype, mode, N, K, B):
    y, ref = _run_gemv(dtype, mode, N, K, B)
    assert not torch.isnan(y).any()
    scale = ref.abs().max().item() + 1e-6
    err = (y - ref).abs().max().item()
    assert err <= 2e-5 * scale * max(1.0, K / 1024) + 1e-6, (err, scale)


def test_gemv_rejects_bad_shapes():
    with pytest.raises(capi.PipoError) as e:
        capi.pipo_op_gemv(1, 0, 16, 10, 12, 16, 1, 16, 0)  # K not a multiple of 8
    assert e.value.status == capi.PIPO_EINVAL


def lm_head_inputs(dtype, V, H, B, seed, with_gamma=True):
    g = torch.Generator().manual_seed(seed)
    E = torch.randn(V, H, generator=g) * 0.05
    gam = 1.0 + 0.1 * torch.randn(H, generator=g)
    if dtype == 1:
        E, gam = E.to(torch.bfloat16), gam.to(torch.bfloat16)
    h = torch.randn(B, H, generator=g) * 3
    if with_gamma:  # RMSNorm(h; gamma)
        y = h.double() / torch.sqrt((h.double() ** 2).mean(1, keepdim=True) + 1e-6) * gam.double()
    else:  # a NULL gain means no norm
        y = h.double()
    ref = y @ E.double().t()
    return E, gam if with_gamma else None, h, ref


def run_lm_head(dtype, E, gam, h, V, H, B, fn=None):
    Ed, hd = E.cuda(), h.cuda()
    gd = gam.cuda() if gam is not None else None
    tok = torch.full((B,), -7, dtype=torch.int32, device="cuda")
    logits = torch.empty(B, V, device="cuda")
    scratch = torch.empty(B, dtype=torch.int64, device="cuda")
    capi.pipo_op_lm_head_argmax(dtype, Ed.data_ptr(), V, H, hd.data_ptr(), gd.data_ptr() if gd is not None else 0,
                                1e-6, B, tok.data_ptr(), logits.data_ptr(), scratch.data_ptr(), 8 * B,
                                torch.cuda.current_stream().cuda_stream)
    torch.cuda.synchronize()
    return tok.cpu(), logits.cpu().double()


@pytest.mark.parametrize("dtype", [0, 1])
@pytest.mark.parametrize("B", [1, 3, 6])
@pytest.mark.parametrize("with_gamma", [True, False])
def test_lm_head_argmax_matches_float64(dtype, B, with_gamma):
    V, H = 30011, 512
    E, gam, h, ref = lm_head_inputs(dtype, V, H, B, seed=B + 10 * dtype, with_gamma=with_gamma)
    tok, logits = run_lm_head(dtype, E, gam, h, V, H, B)
    assert (logits - ref).abs().max().item() < 1e-4 * max(1.0, ref.abs().max().item())
    top2 = ref.topk(2, dim=1).values
    for b in range(B):
        if top2[b, 0] - top2[b, 1] > 1e-4:
            assert int(tok[b]) == int(ref[b].argmax())


def test_lm_head_argmax_ties_take_lowest_row():
    V, H, B = 5000, 256, 2
    E = torch.zeros(V, H)
    E[[17, 4000, 999], 0] = 1.0  # three equal maxima
    h = torch.zeros(B, H)
    h[:, 0] = 1.0
    tok, _ = run_lm_head(0, E, None, h, V, H, B)
    assert tok.tolist() == [17, 17]


def test_lm_head_argmax_rejects_short_scratch():
    with pytest.raises(capi.PipoError) as e:
        capi.pipo_op_lm_head_argmax(1, 16, 8, 16, 16, 0, 1e-6, 4, 16, 0, 16, 8, 0)
    assert e.value.status == capi.PIPO_EINVAL
