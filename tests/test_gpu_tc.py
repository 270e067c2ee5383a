"""Tensor-core (tcgen05) projections: the kernel through its C-ABI entry point
against a float64 evaluation of the fp32-activation projection, and the decode
path with batches that route the projections to it, against the fp64 oracle
(forced replay)."""
import pytest
import torch

from paper_2605_27255_gb300 import capi, synth
from parity_util import run_forced_replay

pytestmark = pytest.mark.gpu


def _run_tc(mode, N, K, B, splits, seed=0):
    g = torch.Generator().manual_seed(seed + 7 * N + K + B)
    rows = 2 * N if mode else N
    W = (torch.randn(rows, K, generator=g) * 0.05).to(torch.bfloat16)
    x = torch.randn(B, K, generator=g)
    Wd, xd = W.cuda(), x.cuda()
    y = torch.full((B, N), float("nan"), device="cuda")
    nbytes = capi.pipo_op_gemm_tc_scratch(mode, N, K, B, splits)
    assert nbytes > 0
    scratch = torch.empty(nbytes + 1024, dtype=torch.uint8, device="cuda")
    base = (scratch.data_ptr() + 1023) // 1024 * 1024
    stream = torch.cuda.current_stream().cuda_stream
    for _ in range(2):  # twice: the split-K arrival counters must come back to zero
        y.fill_(float("nan"))
        capi.pipo_op_gemm_tc(mode, Wd.data_ptr(), N, K, xd.data_ptr(), B, y.data_ptr(), splits, base, nbytes,
                             stream)
        torch.cuda.synchronize()
    # fp32 activations: the kernel carries them as bf16 hi + lo parts
    ref = x.double() @ W.double().t()
    if mode:
        gate, up = ref[:, 0::2], ref[:, 1::2]
        ref = gate * torch.sigmoid(gate) * up
    return y.cpu().double(), ref


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("N,K", [(2560, 2560), (333, 4096), (1000, 1408), (4096, 256), (128, 64)])
@pytest.mark.parametrize("B", [1, 16, 24, 37, 64, 128])
@pytest.mark.parametrize("splits", [0, 1, 3])
def test_gemm_tc_matches_float64(mode, N, K, B, splits):
    y, ref = _run_tc(mode, N, K, B, splits)
    assert not torch.isnan(y).any()
    scale = ref.abs().max().item() + 1e-6
    err = (y - ref).abs().max().item()
    assert err <= 2e-5 * scale * max(1.0, K / 1024) + 1e-6, (err, scale)


def test_gemm_tc_split_orders_agree():
    """Different K splits change only the fp32 summation order."""
    a, ref = _run_tc(0, 2560, 9728, 16, 1)
    b, _ = _run_tc(0, 2560, 9728, 16, 19)
    assert (a - b).abs().max().item() <= 2e-5 * ref.abs().max().item() * 9728 / 1024


def test_gemm_tc_rejects_bad_arguments():
    assert capi.pipo_op_gemm_tc_scratch(0, 256, 100, 4, 0) == 0  # K not a multiple of 64
    assert capi.pipo_op_gemm_tc_scratch(0, 256, 128, 129, 0) == 0  # B > 128
    assert capi.pipo_op_gemm_tc_scratch(0, 64, 128, 4, 0) == 0  # fewer than 128 rows
    W = torch.zeros(256, 128, dtype=torch.bfloat16, device="cuda")
    x = torch.zeros(4, 128, device="cuda")
    y = torch.zeros(4, 256, device="cuda")
    need = capi.pipo_op_gemm_tc_scratch(0, 256, 128, 4, 0)
    s = torch.empty(need + 2048, dtype=torch.uint8, device="cuda")
    base = (s.data_ptr() + 1023) // 1024 * 1024
    with pytest.raises(capi.PipoError) as e:  # short scratch
        capi.pipo_op_gemm_tc(0, W.data_ptr(), 256, 128, x.data_ptr(), 4, y.data_ptr(), 0, base, need - 4, 0)
    assert e.value.status == capi.PIPO_EINVAL
    with pytest.raises(capi.PipoError) as e:  # scratch not 1024-byte aligned
        capi.pipo_op_gemm_tc(0, W.data_ptr(), 256, 128, x.data_ptr(), 4, y.data_ptr(), 0, base + 256, need, 0)
    assert e.value.status == capi.PIPO_EINVAL


def _rms(v, eps=1e-6):
    return v / torch.sqrt((v * v).mean(1, keepdim=True) + eps)


def _run_tc_norm(mode, N, K0, K1, B, form, splits=0, seed=0):
    """form: "one" (one segment, gain), "joint" (two segments, one gain over
    K0 + K1), "sep" (two segments, a gain each), "half" (two segments, gain on
    the first only).  Gains around 1 with distinct values per element."""
    g = torch.Generator().manual_seed(seed + 13 * N + K0 + 3 * K1 + B)
    rows = 2 * N if mode else N
    K = K0 + (K1 if form != "one" else 0)
    W = (torch.randn(rows, K, generator=g) * 0.05).to(torch.bfloat16)
    x0 = torch.randn(B, K0, generator=g) * 2.0
    x1 = torch.randn(B, K1, generator=g) * 0.5 if form != "one" else None
    gam = lambda n: (1.0 + 0.2 * torch.randn(n, generator=g)).to(torch.bfloat16)
    g0 = gam(K if form == "joint" else K0)
    g1 = gam(K1) if form == "sep" else None
    if form == "one":
        inp = _rms(x0.double()) * g0.double()
    elif form == "joint":
        inp = _rms(torch.cat([x0, x1], 1).double()) * g0.double()
    else:
        s1 = _rms(x1.double()) * g1.double() if form == "sep" else x1.double()
        inp = torch.cat([_rms(x0.double()) * g0.double(), s1], 1)
    ref = inp @ W.double().t()
    if mode:
        gate, up = ref[:, 0::2], ref[:, 1::2]
        ref = gate * torch.sigmoid(gate) * up
    dev = [t.cuda() if t is not None else None for t in (W, x0, x1, g0, g1)]
    ptr = lambda t: t.data_ptr() if t is not None else 0
    y = torch.full((B, N), float("nan"), device="cuda")
    nbytes = capi.pipo_op_gemm_tc_scratch(mode, N, K, B, splits)
    assert nbytes > 0
    scratch = torch.empty(nbytes + 1024, dtype=torch.uint8, device="cuda")
    base = (scratch.data_ptr() + 1023) // 1024 * 1024
    stream = torch.cuda.current_stream().cuda_stream
    for _ in range(2):
        y.fill_(float("nan"))
        capi.pipo_op_gemm_tc_norm(mode, ptr(dev[0]), N, ptr(dev[1]), K0, ptr(dev[3]), ptr(dev[2]),
                                  K1 if form != "one" else 0, ptr(dev[4]), int(form == "joint"), 1e-6, B,
                                  y.data_ptr(), splits, base, nbytes, stream)
        torch.cuda.synchronize()
    return y.cpu().double(), ref


@pytest.mark.parametrize("form", ["one", "joint", "sep", "half"])
@pytest.mark.parametrize("mode,N,K0,K1", [(0, 2560, 2560, 2560), (1, 1000, 1024, 512), (0, 333, 4096, 64)])
@pytest.mark.parametrize("B", [4, 16, 32, 37, 100])
def test_gemm_tc_normalised_segments_match_float64(form, mode, N, K0, K1, B):
    """RMSNorm gains on the tensor-core path: B = 16 and 32 with one
    segment or a joint norm run the converter warps of the fused GEMM; the
    other batches and the separately normalised segments take the prepared
    bf16 operand (prep_bf16_kernel).  A gain skipped, misplaced or taken from
    the other segment fails the comparison."""
    y, ref = _run_tc_norm(mode, N, K0, K1, B, form)
    assert not torch.isnan(y).any()
    K = K0 + (K1 if form != "one" else 0)
    scale = ref.abs().max().item() + 1e-6
    err = (y - ref).abs().max().item()
    assert err <= 2e-5 * scale * max(1.0, K / 1024) + 1e-6, (err, scale)


def test_gemm_tc_norm_rejects_bad_arguments():
    W = torch.zeros(256, 256, dtype=torch.bfloat16, device="cuda")
    x = torch.zeros(4, 128, device="cuda")
    gm = torch.ones(256, dtype=torch.bfloat16, device="cuda")
    y = torch.zeros(4, 256, device="cuda")
    need = capi.pipo_op_gemm_tc_scratch(0, 256, 256, 4, 0)
    s = torch.empty(need + 2048, dtype=torch.uint8, device="cuda")
    base = (s.data_ptr() + 1023) // 1024 * 1024
    bad = [
        dict(joint=1, x1=0, K1=0),                     # joint norm needs two segments
        dict(joint=1, g1=gm.data_ptr()),               # joint norm takes one gain
        dict(K1=96),                                   # K1 not a multiple of 64
        dict(x1=0, K1=128),                            # K1 without a second segment
        dict(g0=gm.data_ptr() + 2),                    # misaligned gain
        dict(nbytes=need - 16),                        # short scratch
    ]
    for kw in bad:
        a = dict(x1=x.data_ptr(), K1=128, g0=gm.data_ptr(), g1=0, joint=0, nbytes=need)
        a.update(kw)
        with pytest.raises(capi.PipoError) as e:
            capi.pipo_op_gemm_tc_norm(0, W.data_ptr(), 256, x.data_ptr(), 128, a["g0"], a["x1"], a["K1"], a["g1"],
                                      a["joint"], 1e-6, 4, y.data_ptr(), 0, base, a["nbytes"], 0)
        assert e.value.status == capi.PIPO_EINVAL, kw


# model-level: 512-wide blocks, ragged vocabulary; the FFN down projection
# (K = 1376, not a multiple of 64) stays on the CUDA-core kernel
MID = synth.ModelShape("mid", H=512, L=3, n_q=8, n_kv=2, d_h=128, F=1376, V=5003,
                       compressor="mlp", mtp_block=1, dtype="bf16", rope_theta=1.0e4, tau=0.5)


@pytest.mark.parametrize("B", [16, 24, 37, 64])
def test_mid_bf16_tensor_core_batches(B):
    """B = 16 and 24 take the fused projections (batch widths 16 and 32),
    B = 37 and 64 the split-kernel form (width 64); tensor-core attention;
    forced replay against the oracle."""
    w = synth.gen_weights(MID, seed=21)
    prompts = synth.gen_prompts(B, 24, MID.V, seed=B).numpy()
    st = run_forced_replay(MID, w, prompts, 4, force=0, page_shuffle_seed=5)
    assert st.tok_checked >= 0.8 * st.tok_total
    assert st.max_logit_err < 2e-2


def test_mid_bf16_cuda_core_batches_over_8(monkeypatch):
    """The CUDA-core GEMV at B = 37: five 8-sequence groups, split-K residual adds."""
    monkeypatch.setenv("PIPO_TC_MIN_BATCH", "100000")
    w = synth.gen_weights(MID, seed=22)
    prompts = synth.gen_prompts(37, 24, MID.V, seed=9).numpy()
    st = run_forced_replay(MID, w, prompts, 3, force=1)
    assert st.tok_checked >= 0.8 * st.tok_total
    assert st.max_logit_err < 2e-2


def test_decode_path_uses_tensor_core_kernels():
    """At B = 16 the block projections and the attention take the tcgen05 and
    mma.sync kernels (the down projection, K = 1376, stays on CUDA cores); a
    single sequence keeps the CUDA-core GEMV (a matrix-vector product) and
    takes the tensor-core attention (its 4 query heads per kv head are the
    MMA rows) in 8-CTA clusters, one CTA per SM, on the deep stage ring."""
    w = synth.gen_weights(MID, seed=23)
    g = capi.Pipo(MID, w, max_batch=16, max_ctx=40)
    try:
        g.prefill(synth.gen_prompts(16, 8, MID.V, seed=1).numpy())
        d = g.describe()
        assert "gemm_tcf_kernel<16>" in d and "1 of 4 block projections on gemv_kernel" in d, d
        assert "attn_mma_kernel" in d, d
    finally:
        g.close()
    g = capi.Pipo(MID, w, max_batch=1, max_ctx=40)
    try:
        g.prefill(synth.gen_prompts(1, 8, MID.V, seed=1).numpy())
        d = g.describe()
        assert "projections=gemv_rows_kernel" in d and "attention=attn_mma_kernel cluster=8 stages=20" in d, d
    finally:
        g.close()
