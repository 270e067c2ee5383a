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
