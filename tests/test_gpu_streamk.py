"""The stream-K schedule of the tensor-core GEMM: with a caller workspace, a prefill layer
whose tiles leave SMs idle has the k range of all its tiles cut into one equal range per
SM, and the partial tiles are added through the workspace. Checked here against the
oracle on shapes that take it (one and two token tiles per CTA, heads that add one tail
and heads that add several, ragged M / N / K, every epilogue), together with the contract
of the workspace: handed back zero-filled, results deterministic, and within the same
bound as the schedule without a workspace."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
from tests.gpu_util import check_close, to_dev_bf16
from workloads import activation_bits_np, weight_np

pytestmark = pytest.mark.gpu
Q8, Q4, Q6 = emb.EMB_Q8_0, emb.EMB_Q4_0, emb.EMB_Q6_0

# (fmt, M, N, K), all taking the stream-K schedule on a 152-SM GB300: one token tile of 256
# per CTA (157 tiles); two token tiles per CTA with heads adding up to four tails; ragged
# M, N and K (19.75 raw stages of 256, Q6_0); ragged N and K (62.5 steps of 64)
CASES = [(Q8, 256, 20000, 2048), (Q4, 280, 5000, 4096), (Q6, 300, 5000, 5056), (Q8, 280, 5500, 4000)]


def _setup(fmt, M, N, K, seed):
    W = weight_np(N, K, seed)
    Xb = activation_bits_np(M, K, seed + 1)
    img = emb.quantize(fmt, torch.from_numpy(W).cuda())
    X = to_dev_bf16(Xb)
    return W, Xb, img, X


def _run(fmt, img, X, Y, M, N, K, ws, kind=emb.EMB_EPI_F32):
    emb.emb_qlayer_seq([(fmt, img, N, K, X, Y, kind)], M, ws, 0 if ws is None else ws.numel())
    torch.cuda.synchronize()
    assert emb.emb_device_status() == emb.EMB_OK


def test_workspace_wanted_only_where_tiles_leave_sms_idle(cuda_device):
    """Llama-7B gate/up at M = 280 (172 tiles of two token tiles on 152 SMs) wants the
    workspace; Gemma-2B q/k/v at M = 816 (80 tiles) and every M <= 50 shape do not."""
    M, K = 280, 4096
    img = emb.quantize(Q4, torch.randn(11008, K, device="cuda") * 0.02)
    X = torch.zeros(M, K, dtype=torch.bfloat16, device="cuda")
    Y = torch.empty(M, 11008, device="cuda")
    n = emb.emb_qlayer_seq_workspace([(Q4, img, 11008, K, X, Y), (Q4, img, 11008, K, X, Y.clone())], M)
    sms = torch.cuda.get_device_properties(0).multi_processor_count
    # 4 KB of flags, then one fp32 partial tile (2 x 144 tokens x 128 rows) per SM
    assert n == 4096 + sms * 2 * 144 * 128 * 4
    for m in (1, 4, 50):
        assert emb.emb_qlayer_seq_workspace([(Q4, img, 11008, K, X[:m], Y[:m])], m) == 0
    W, Xb, img8, X8 = _setup(Q8, 816, 2560, 2048, 3)
    assert emb.emb_qlayer_seq_workspace([(Q8, img8, 2560, 2048, X8, torch.empty(816, 2560, device="cuda"))], 816) == 0


@pytest.mark.parametrize("fmt,M,N,K", CASES)
def test_streamk_parity(cuda_device, fmt, M, N, K):
    W, Xb, img, X = _setup(fmt, M, N, K, 11 + N + K)
    Y = torch.full((M, N), float("nan"), device="cuda")
    # (the query validates the layer as a call would: Y must be a real [M][N] buffer)
    n = emb.emb_qlayer_seq_workspace([(fmt, img, N, K, X, Y)], M)
    assert n > 0, "this shape should take the stream-K schedule"
    ws = torch.zeros(n, dtype=torch.uint8, device="cuda")
    _run(fmt, img, X, Y, M, N, K, ws)
    assert int(ws[:4096].count_nonzero()) == 0, "ready flags left set"
    Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
    worst = check_close(Y.cpu().numpy(), Yref, B, f"stream-K fmt={fmt} M={M} N={N} K={K}")
    # deterministic, and a chain replay gives the same bits
    Y2 = torch.full_like(Y, float("nan"))
    _run(fmt, img, X, Y2, M, N, K, ws)
    assert torch.equal(Y.view(torch.int32), Y2.view(torch.int32))
    rec = emb.RecordedChain([(fmt, img, N, K, X, Y2)], M)
    Y2.fill_(float("nan"))
    rec.launch()
    torch.cuda.synchronize()
    rec.close()
    assert torch.equal(Y.view(torch.int32), Y2.view(torch.int32))
    # the schedule without a workspace meets the same bound
    Y3 = torch.full_like(Y, float("nan"))
    _run(fmt, img, X, Y3, M, N, K, None)
    check_close(Y3.cpu().numpy(), Yref, B, f"no workspace fmt={fmt} M={M} N={N} K={K}")
    print(f"max err/sum|wx| {worst:.2e}")


EPI_CASES = [(Q4, 280, 5000, 4096, k) for k in (emb.EMB_EPI_BF16, emb.EMB_EPI_ADD, emb.EMB_EPI_GEGLU,
                                               emb.EMB_EPI_SWIGLU)] + \
            [(Q8, 256, 20000, 2048, k) for k in (emb.EMB_EPI_ADD, emb.EMB_EPI_GEGLU)]


@pytest.mark.parametrize("fmt,M,N,K,kind", EPI_CASES)
def test_streamk_epilogues(cuda_device, fmt, M, N, K, kind):
    W, Xb, img, X = _setup(fmt, M, N, K, 7 + kind)
    R = (np.random.default_rng(kind).standard_normal((M, N)) * 3).astype(np.float32)
    if kind == emb.EMB_EPI_ADD:
        Y = torch.from_numpy(R.copy()).cuda()
    else:
        cols = N // 2 if kind >= emb.EMB_EPI_GEGLU else N
        Y = torch.full((M, cols), float("nan"), dtype=torch.bfloat16, device="cuda")
    layers = [(fmt, img, N, K, X, Y, kind)]
    ws = emb.chain_workspace(layers, M)
    assert ws is not None
    _run(fmt, img, X, Y, M, N, K, ws, kind)
    Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
    ref, bound = oracle.epilogue_reference(kind, Yref, B, R)
    out = Y.float().cpu().numpy().astype(np.float64)
    err = np.abs(out - ref)
    assert np.isfinite(out).all()
    bad = err > bound
    assert not bad.any(), (f"kind={kind}: {int(bad.sum())} outside, first {np.argwhere(bad)[:4].tolist()} "
                           f"err={err[bad][:4]} bound={bound[bad][:4]}")


def test_streamk_one_hot_rows_are_exact(cuda_device):
    """One-hot activation rows through the stream-K schedule: every output is one
    dequantised weight, bf16-rounded (K >= 1024: one bf16 operand), plus zero partials."""
    fmt, M, N, K = Q8, 280, 5000, 4096
    W = weight_np(N, K, 5)
    img = emb.quantize(fmt, torch.from_numpy(W).cuda())
    ks = np.random.default_rng(9).choice(K, M, replace=False)
    Xb = np.zeros((M, K), dtype=np.uint16)
    Xb[np.arange(M), ks] = 0x3F80
    X = to_dev_bf16(Xb)
    Y = torch.full((M, N), float("nan"), device="cuda")
    layers = [(fmt, img, N, K, X, Y)]
    ws = emb.chain_workspace(layers, M)
    assert ws is not None
    _run(fmt, img, X, Y, M, N, K, ws)
    deq = oracle.dequant_bf16(fmt, oracle.quantize(fmt, W), N, K)  # bf16 bits [N][K]
    want = (deq[:, ks].T.astype(np.uint32) << 16).view(np.float32)
    got = Y.cpu().numpy()
    assert np.array_equal(got.view(np.uint32), want.view(np.uint32))


def test_workspace_errors(cuda_device):
    fmt, M, N, K = Q4, 280, 5000, 4096
    W, Xb, img, X = _setup(fmt, M, N, K, 2)
    Y = torch.empty(M, N, device="cuda")
    layers = [(fmt, img, N, K, X, Y)]
    n = emb.emb_qlayer_seq_workspace(layers, M)
    ws = torch.zeros(n + 512, dtype=torch.uint8, device="cuda")
    with pytest.raises(emb.EmbError) as e:
        emb.emb_qlayer_seq(layers, M, ws, n - 1)
    assert e.value.status == emb.EMB_ENOSPC
    with pytest.raises(emb.EmbError) as e:
        emb.emb_qlayer_seq(layers, M, ws[16:], n)
    assert e.value.status == emb.EMB_EALIGN
