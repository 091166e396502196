"""Fused epilogues of layer chains against the oracle: bf16 output, in-place residual add,
GeGLU / SwiGLU of interleaved gate/up rows, on every kernel path (register and staged
GEMV, Q4_0 tensor-core GEMV, tcgen05 GEMM with one or two token tiles per CTA, split K
and the split operand), and a chain whose layers feed each other (gated bf16 output into
the down projection, residual add)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
from tests.gpu_util import to_dev_bf16
from workloads import activation_bits_np, weight_np

pytestmark = pytest.mark.gpu
Q8, Q4, Q6 = emb.EMB_Q8_0, emb.EMB_Q4_0, emb.EMB_Q6_0
KINDS = [emb.EMB_EPI_BF16, emb.EMB_EPI_ADD, emb.EMB_EPI_GEGLU, emb.EMB_EPI_SWIGLU]


def _out_buffer(kind, M, N, R=None):
    if kind == emb.EMB_EPI_ADD:
        return torch.from_numpy(R.copy()).cuda()
    cols = N // 2 if kind >= emb.EMB_EPI_GEGLU else N
    return torch.full((M, cols), float("nan"), dtype=torch.bfloat16, device="cuda")


def _as_f64(Y):
    return Y.float().cpu().numpy().astype(np.float64)


def _check(out, ref, bound, what):
    err = np.abs(out - ref)
    assert np.isfinite(out).all(), f"{what}: non-finite output"
    bad = err > bound
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} outside, first "
                           f"{np.argwhere(bad)[:4].tolist()} err={err[bad][:4]} bound={bound[bad][:4]}")


def run_epilogue(fmt, kind, M, N, K, seed):
    W = weight_np(N, K, seed)
    Xb = activation_bits_np(M, K, seed + 1)
    R = (np.random.default_rng(seed + 2).standard_normal((M, N)) * 3).astype(np.float32)
    img = emb.quantize(fmt, torch.from_numpy(W).cuda())
    X = to_dev_bf16(Xb)
    Y = _out_buffer(kind, M, N, R)
    emb.emb_qlayer_seq([(fmt, img, N, K, X, Y, kind)], M)
    torch.cuda.synchronize()
    Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
    ref, bound = oracle.epilogue_reference(kind, Yref, B, R)
    _check(_as_f64(Y), ref, bound, f"fmt={fmt} kind={kind} M={M} N={N} K={K}")
    return Y


# (fmt, M, N, K): register GEMV, staged GEMV (>= 12 MB), register GEMV at M = 4, Q4_0
# tensor-core GEMV (M = 2..8, >= 12 MB), GEMM split operand (K < 1024), GEMM split K,
# GEMM one token tile per CTA, GEMM two token tiles per CTA, Q6_0 GEMV and GEMM, Q8_0
# register GEMV loading whole row shares before the wait (long rows, two rows per CTA), Q4_0
# staged GEMV at M = 1 with a ragged last tile, GEMM with persistent CTAs (320 tiles), the
# ring GEMV (long rows, >= 12 MB, M = 1; the second and third with a ragged last CTA, the
# third with the Q6_0 high plane)
PATHS = [(Q8, 1, 256, 1024), (Q8, 1, 24576, 2048), (Q4, 4, 600, 2080), (Q4, 4, 32768, 1024),
         (Q8, 64, 384, 320), (Q8, 50, 1000, 1024), (Q4, 136, 640, 2048), (Q8, 280, 11008, 1024),
         (Q6, 1, 4096, 2048), (Q6, 50, 512, 2048), (Q8, 1, 1300, 7168), (Q4, 1, 16392, 2048),
         (Q8, 816, 10240, 1024), (Q8, 1, 2048, 16384), (Q4, 1, 1538, 16384), (Q6, 1, 1026, 16384)]


@pytest.mark.parametrize("kind", KINDS)
@pytest.mark.parametrize("fmt,M,N,K", PATHS)
def test_epilogue_parity(cuda_device, fmt, M, N, K, kind):
    if kind >= emb.EMB_EPI_GEGLU and fmt == Q4 and M == 4 and N == 32768:
        pytest.skip("gated layers do not take the Q4_0 tensor-core GEMV (pairs rows elsewhere)")
    run_epilogue(fmt, kind, M, N, K, seed=M * 3 + N + K + 17 * kind)


@pytest.mark.parametrize("kind", [emb.EMB_EPI_GEGLU, emb.EMB_EPI_SWIGLU])
def test_gated_q4_tensor_core_shape_still_correct(cuda_device, kind):
    """A gated Q4_0 layer at the tensor-core GEMV's shape runs on the FFMA2 kernels."""
    run_epilogue(Q4, kind, 4, 32768, 1024, seed=5 + kind)


@pytest.mark.parametrize("fmt,M", [(Q8, 1), (Q4, 1), (Q8, 50), (Q6, 280)])
def test_mlp_block_chain(cuda_device, fmt, M):
    """gate/up (interleaved rows, GeGLU, bf16 H) -> down (X = H, added into the residual R):
    one chain with a real dependency, checked layer by layer against the oracle, then
    replayed from a recording with the same bits."""
    D, F = 512, 1536
    Wgu = weight_np(2 * F, D, 100 + M)
    Wd = weight_np(D, F, 101 + M)
    Xb = activation_bits_np(M, D, 102 + M)
    R0 = (np.random.default_rng(103 + M).standard_normal((M, D)) * 2).astype(np.float32)
    img_gu = emb.quantize(fmt, torch.from_numpy(Wgu).cuda())
    img_d = emb.quantize(fmt, torch.from_numpy(Wd).cuda())
    X = to_dev_bf16(Xb)
    H = torch.empty(M, F, dtype=torch.bfloat16, device="cuda")
    Rbuf = torch.from_numpy(R0.copy()).cuda()
    specs = [(fmt, img_gu, 2 * F, D, X, H, emb.EMB_EPI_GEGLU),
             (fmt, img_d, D, F, H, Rbuf, emb.EMB_EPI_ADD)]
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    # layer 1 against the oracle
    Ygu, Bgu = oracle.qmatmul(fmt, oracle.quantize(fmt, Wgu), Xb, 2 * F, D)
    ref_h, bound_h = oracle.epilogue_reference(emb.EMB_EPI_GEGLU, Ygu, Bgu)
    _check(_as_f64(H), ref_h, bound_h, "gated gate/up")
    # layer 2 from the bf16 H the GPU produced
    Hb = H.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)
    Yd, Bd = oracle.qmatmul(fmt, oracle.quantize(fmt, Wd), Hb, D, F)
    ref_r, bound_r = oracle.epilogue_reference(emb.EMB_EPI_ADD, Yd, Bd, R0)
    _check(_as_f64(Rbuf), ref_r, bound_r, "down + residual")
    first_h, first_r = H.clone(), Rbuf.clone()
    # a recording replays the same bits (the residual is reset before each replay)
    rec = emb.RecordedChain(specs, M)
    for _ in range(2):
        Rbuf.copy_(torch.from_numpy(R0))
        H.fill_(float("nan"))
        rec.launch()
        torch.cuda.synchronize()
        assert torch.equal(H.view(torch.int16), first_h.view(torch.int16))
        assert torch.equal(Rbuf.view(torch.int32), first_r.view(torch.int32))
    rec.close()
    assert emb.emb_device_status() == emb.EMB_OK


def test_residual_adds_accumulate_in_order(cuda_device):
    """Three layers add into one fp32 buffer in turn (o, then down of two layers): the
    result is R0 + Y1 + Y2 + Y3 with each add rounded once, in chain order."""
    M, N, K = 1, 2048, 2048
    specs, ys = [], []
    R0 = (np.random.default_rng(9).standard_normal((M, N))).astype(np.float32)
    Rbuf = torch.from_numpy(R0.copy()).cuda()
    for i in range(3):
        W = weight_np(N, K, 200 + i)
        Xb = activation_bits_np(M, K, 210 + i)
        img = emb.quantize(Q8, torch.from_numpy(W).cuda())
        specs.append((Q8, img, N, K, to_dev_bf16(Xb), Rbuf, emb.EMB_EPI_ADD))
        ys.append((img, specs[-1][4]))
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    # the same three products as plain fp32 outputs, then the adds in order on the host
    expect = torch.from_numpy(R0.copy()).cuda()
    for img, X in ys:
        Y = emb.qmatmul(Q8, img, X, N)
        torch.cuda.synchronize()
        expect = expect + Y   # one fp32 rounding per add, as the epilogue does
    assert torch.equal(Rbuf, expect)


def test_epilogues_are_deterministic(cuda_device):
    for kind in KINDS:
        fmt, M, N, K = Q8, 50, 1000, 1024
        W = weight_np(N, K, 3)
        Xb = activation_bits_np(M, K, 4)
        img = emb.quantize(fmt, torch.from_numpy(W).cuda())
        X = to_dev_bf16(Xb)
        R = np.zeros((M, N), dtype=np.float32)
        outs = []
        for _ in range(2):
            Y = _out_buffer(kind, M, N, R)
            emb.emb_qlayer_seq([(fmt, img, N, K, X, Y, kind)], M)
            torch.cuda.synchronize()
            outs.append(Y)
        assert torch.equal(outs[0].view(torch.int16) if outs[0].dtype == torch.bfloat16 else outs[0],
                           outs[1].view(torch.int16) if outs[1].dtype == torch.bfloat16 else outs[1])
