"""The 6-bit configuration (Q6_0) end to end on the GPU against the oracle: GEMV
(register and staged kernels, M = 1..4) and tcgen05 GEMM (one and two token tiles per
CTA, split K, the split operand for K < 1024), ragged shapes, fused groups and chains."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
from tests.gpu_util import check_close, run_case, to_dev_bf16
from workloads import activation_bits_np, weight_np

pytestmark = pytest.mark.gpu
Q6 = emb.EMB_Q6_0

# M <= 4: one unit per row (K = 32), ragged units, long rows (register kernel), large
# layers with short rows (staged kernel: >= 12 MB), several tokens
GEMV_SHAPES = [(1, 1, 32), (1, 136, 96), (1, 2048, 2048), (1, 300, 11008), (1, 130, 16384),
               (1, 20000, 2048), (2, 200, 4608), (3, 129, 1056), (4, 1000, 2080), (4, 24000, 1024)]

# M > 4 with K % 64 == 0: split operand (K < 1024), split K, one and two token tiles per
# CTA (280 x 11008 x 1024 takes pairs), ragged N and M
GEMM_SHAPES = [(5, 128, 256), (16, 8, 64), (50, 1000, 1024), (50, 130, 4096), (64, 384, 320),
               (136, 640, 2048), (280, 11008, 1024), (300, 9000, 1152), (816, 384, 2048)]


@pytest.mark.parametrize("M,N,K", GEMV_SHAPES)
def test_q6_gemv_parity(cuda_device, M, N, K):
    Y, Yref, B, img, ref_img = run_case(Q6, M, N, K, seed=M * 7 + N + K)
    assert np.array_equal(img.cpu().numpy(), ref_img)
    check_close(Y, Yref, B, f"q6 gemv M={M} N={N} K={K}")


@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
def test_q6_gemm_parity(cuda_device, M, N, K):
    Y, Yref, B, _, _ = run_case(Q6, M, N, K, seed=M * 5 + N + K)
    check_close(Y, Yref, B, f"q6 gemm M={M} N={N} K={K}")


@pytest.mark.parametrize("K", [96, 1056])
def test_q6_gemm_needs_k_multiple_of_64(cuda_device, K):
    """The high plane's tensor map needs a 16-byte row pitch (K/4): other K are refused
    for M > 4 before anything is launched; M <= 4 runs."""
    N = 64
    img = emb.quantize(Q6, torch.from_numpy(weight_np(N, K, 3)).cuda())
    X = to_dev_bf16(activation_bits_np(8, K, 4))
    with pytest.raises(emb.EmbError) as e:
        emb.qmatmul(Q6, img, X, N)
    assert e.value.status == emb.EMB_EUNSUPPORTED
    Y = emb.qmatmul(Q6, img, X[:4].contiguous(), N)
    torch.cuda.synchronize()
    assert torch.isfinite(Y).all()


@pytest.mark.parametrize("M", [1, 50, 280])
def test_q6_chain_fused_groups_and_replay(cuda_device, M):
    """A two-layer decoder chain (fused q/k/v and gate/up) through emb_qlayer_seq and a
    recorded chain: every layer against the oracle, replay bits equal."""
    specs, host = [], []
    s = 9000 + M
    for _ in range(2):
        for group in ([(512, 512), (128, 512), (128, 512)], [(512, 512)],
                      [(1536, 512), (1536, 512)], [(512, 1536)]):
            K = group[0][1]
            Xb = activation_bits_np(M, K, s)
            X = to_dev_bf16(Xb)
            for N, _ in group:
                s += 1
                W = weight_np(N, K, s)
                img = emb.quantize(Q6, torch.from_numpy(W).cuda())
                Y = torch.full((M, N), float("nan"), device="cuda")
                specs.append((Q6, img, N, K, X, Y))
                host.append((W, Xb))
            s += 1
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    first = [sp[5].clone() for sp in specs]
    for i, (sp, (W, Xb)) in enumerate(zip(specs, host)):
        Yref, B = oracle.qmatmul(Q6, oracle.quantize(Q6, W), Xb, sp[2], sp[3])
        check_close(first[i].cpu().numpy(), Yref, B, f"q6 chain layer {i}")
    rec = emb.RecordedChain(specs, M)
    for sp in specs:
        sp[5].fill_(float("nan"))
    rec.launch()
    torch.cuda.synchronize()
    for a, sp in zip(first, specs):
        assert torch.equal(a.view(torch.int32), sp[5].view(torch.int32))
    rec.close()
    assert emb.emb_device_status() == emb.EMB_OK
