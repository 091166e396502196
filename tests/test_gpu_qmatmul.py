"""emb_qmatmul against the oracle: GEMV (M <= 4) and tcgen05 GEMM (M > 4) paths on
shapes spanning several tiles with ragged tails in every dimension."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
from tests.gpu_util import check_close, run_case, to_dev_bf16
from workloads import activation_bits_np, weight_np

pytestmark = pytest.mark.gpu

FMTS = [emb.EMB_Q8_0, emb.EMB_Q4_0]

# (1, 130, 16384), (1, 300, 11008) and (1, 1300, 7168) take the Q8_0 register kernel that
# loads a thread's whole row share before the wait (1 to 4 passes, ragged last pass);
# (1, 64, 40960) has rows longer than four passes and streams them one unit ahead.
GEMV_SHAPES = [(1, 1, 32), (1, 8, 64), (1, 136, 96), (1, 256, 2048), (1, 2048, 2048),
               (1, 130, 16384), (1, 300, 11008), (1, 1300, 7168), (1, 64, 40960),
               (1, 4096, 1152), (2, 200, 4608), (3, 129, 1024), (4, 1000, 2080)]

GEMM_SHAPES = [(5, 128, 1024), (7, 136, 96), (16, 8, 32), (49, 256, 2048), (50, 1024, 1024),
               (51, 264, 1152), (64, 384, 256), (127, 128, 1088), (129, 640, 2048),
               (255, 136, 512), (257, 256, 1024), (280, 512, 4096), (500, 300, 320),
               (768, 256, 1152), (816, 384, 2048)]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("M,N,K", GEMV_SHAPES)
def test_gemv_parity(cuda_device, fmt, M, N, K):
    Y, Yref, B, _, _ = run_case(fmt, M, N, K, seed=M * 7 + N + K)
    check_close(Y, Yref, B, f"gemv fmt={fmt} M={M} N={N} K={K}")


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("M,N,K", GEMM_SHAPES)
def test_gemm_parity(cuda_device, fmt, M, N, K):
    Y, Yref, B, _, _ = run_case(fmt, M, N, K, seed=M * 13 + N + K)
    check_close(Y, Yref, B, f"gemm fmt={fmt} M={M} N={N} K={K}")


@pytest.mark.parametrize("M,N,K", [(1, 384, 2048), (3, 384, 2048), (50, 384, 2048),
                                   (280, 384, 2048), (1, 1300, 7168)])
def test_deterministic(cuda_device, M, N, K):
    W = torch.from_numpy(weight_np(N, K, 3)).cuda()
    X = to_dev_bf16(activation_bits_np(M, K, 4))
    for fmt in FMTS:
        img = emb.quantize(fmt, W)
        Y1 = emb.qmatmul(fmt, img, X, N)
        Y2 = emb.qmatmul(fmt, img, X, N)
        torch.cuda.synchronize()
        assert torch.equal(Y1.view(torch.int32), Y2.view(torch.int32))


def test_outliers_q4_0(cuda_device):
    """1% of weights x8 (the 7B configuration's outlier pattern) at both paths."""
    N, K = 512, 4096
    rng = np.random.default_rng(77)
    W = weight_np(N, K, 78)
    W[rng.random((N, K)) < 0.01] *= 8
    for M in (1, 280):
        Xb = activation_bits_np(M, K, 79)
        img = emb.quantize(emb.EMB_Q4_0, torch.from_numpy(W).cuda())
        Y = emb.qmatmul(emb.EMB_Q4_0, img, to_dev_bf16(Xb), N).cpu().numpy()
        Yref, B = oracle.qmatmul(emb.EMB_Q4_0, oracle.quantize(emb.EMB_Q4_0, W), Xb, N, K)
        check_close(Y, Yref, B, f"outliers M={M}")


def test_extreme_activations(cuda_device):
    """bf16 activations spanning 2^-60..2^40 plus zeros of both signs, where a handful of
    terms dominate sum|w x|: the GEMV (exact products) and the split-operand GEMM
    (K < 1024, operand error 2^-16) must meet the bound for such inputs too."""
    from workloads import bf16_bits_np
    rng = np.random.default_rng(91)
    for M, N, K in ((1, 256, 1024), (64, 256, 512)):
        W = weight_np(N, K, 90)
        x = (rng.standard_normal((M, K)) * np.exp2(rng.integers(-60, 40, size=(M, K)))).astype(np.float32)
        x[:, ::17] = 0.0
        x[:, 5::23] = -0.0
        Xb = bf16_bits_np(x)
        for fmt in FMTS:
            img = emb.quantize(fmt, torch.from_numpy(W).cuda())
            Y = emb.qmatmul(fmt, img, to_dev_bf16(Xb), N).cpu().numpy()
            Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
            check_close(Y, Yref, B, f"extreme x M={M} fmt={fmt}")


def test_y_fully_overwritten(cuda_device):
    N, K = 200, 512
    W = torch.from_numpy(weight_np(N, K, 5)).cuda()
    for M in (1, 70):
        X = to_dev_bf16(activation_bits_np(M, K, 6))
        for fmt in FMTS:
            img = emb.quantize(fmt, W)
            Y0 = emb.qmatmul(fmt, img, X, N)
            Y1 = torch.full((M, N), float("nan"), device="cuda")
            emb.qmatmul(fmt, img, X, N, out=Y1)
            torch.cuda.synchronize()
            assert torch.equal(Y0, Y1)


# Layers of at least 12 MB of packed weights take the staged (bulk-copy ring) GEMV: ragged
# row counts (partial last tile and partial last run of tiles per CTA), K not a multiple of
# the warps' K slices, M = 1..4 and the largest staged activation row (K = 16384 at M = 1).
STAGED_SHAPES = [(1, 24593, 1056), (2, 6151, 4128), (3, 6151, 4096), (4, 12301, 2048),
                 (1, 1543, 16384), (1, 12289, 2048), (2, 12289, 2048), (1, 6151, 4096)]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("M,N,K", STAGED_SHAPES)
def test_staged_gemv_parity(cuda_device, fmt, M, N, K):
    Y, Yref, B, _, _ = run_case(fmt, M, N, K, seed=M * 5 + N + K)
    check_close(Y, Yref, B, f"staged gemv fmt={fmt} M={M} N={N} K={K}")


@pytest.mark.parametrize("fmt", FMTS)
def test_staged_gemv_fused_group(cuda_device, fmt):
    """Two matrices sharing X in one launch (gate/up): tiles of both in one CTA's run."""
    M, K, Ns = 1, 2048, (12289, 12291)
    Xb = activation_bits_np(M, K, 31)
    X = to_dev_bf16(Xb)
    specs, host = [], []
    for i, N in enumerate(Ns):
        W = weight_np(N, K, 40 + i)
        img = emb.quantize(fmt, torch.from_numpy(W).cuda())
        Y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        specs.append((fmt, img, N, K, X, Y))
        host.append(W)
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    first = [sp[5].clone() for sp in specs]
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    for a, sp in zip(first, specs):
        assert torch.equal(a.view(torch.int32), sp[5].view(torch.int32))   # deterministic
    for (f, img, N, _, _, Y), W in zip(specs, host):
        Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
        check_close(Y.cpu().numpy(), Yref, B, f"fused staged N={N}")


# Problems with at least 152 output tiles (128 weight rows x up to 256 tokens): several
# waves of CTAs, tiles that straddle a ragged N, M and K (partial 64-k step and partial
# 256-k raw stage), and a fused pair. Checked element by element against the oracle.
MANY_TILE_SHAPES = [(208, 19461, 1056), (417, 6531, 2080), (816, 4864, 1024), (280, 11008, 1024)]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("M,N,K", MANY_TILE_SHAPES)
def test_many_tile_gemm_parity(cuda_device, fmt, M, N, K):
    Y, Yref, B, _, _ = run_case(fmt, M, N, K, seed=M * 3 + N + K)
    check_close(Y, Yref, B, f"many-tile gemm fmt={fmt} M={M} N={N} K={K}")


@pytest.mark.parametrize("fmt", FMTS)
def test_many_tile_gemm_fused_pair_and_determinism(cuda_device, fmt):
    M, K, Ns = 280, 1024, (11008, 11001)   # two token tiles per CTA (as Llama-7B gate/up)
    Xb = activation_bits_np(M, K, 61)
    X = to_dev_bf16(Xb)
    specs, host = [], []
    for i, N in enumerate(Ns):
        W = weight_np(N, K, 62 + i)
        img = emb.quantize(fmt, torch.from_numpy(W).cuda())
        Y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        specs.append((fmt, img, N, K, X, Y))
        host.append(W)
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    first = [sp[5].clone() for sp in specs]
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    for a, sp in zip(first, specs):
        assert torch.equal(a.view(torch.int32), sp[5].view(torch.int32))
    for (f, img, N, _, _, Y), W in zip(specs, host):
        Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
        check_close(Y.cpu().numpy(), Yref, B, f"fused many-tile N={N}")


# Wide layers at 280..561 tokens where one CTA computes two token tiles from each
# dequantised weight tile: several waves, ragged N, the last token tile partly past M
# (420 = 2 x 224 - 28 with the widest pair tiles, 561 = 4 x 144 - 15), K not a multiple
# of the 256-k raw stage.
PAIR_SHAPES = [(420, 30000, 1024), (561, 19000, 1056), (300, 40000, 1024), (280, 23000, 2080)]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("M,N,K", PAIR_SHAPES)
def test_token_pair_gemm_parity(cuda_device, fmt, M, N, K):
    Y, Yref, B, _, _ = run_case(fmt, M, N, K, seed=M * 13 + N + K)
    check_close(Y, Yref, B, f"token-pair gemm fmt={fmt} M={M} N={N} K={K}")


# 5..64 tokens with K >= 1024 (the action-chunk range): ragged token tails, ragged N, K
# that is not a multiple of the 64-k step or the 256-k raw stage, and long rows.
ACTION_CHUNK_SHAPES = [(5, 136, 1024), (8, 200, 1056), (9, 77, 2048), (16, 300, 1024), (17, 129, 1056),
                   (33, 64, 4128), (50, 1000, 1024), (50, 130, 4096), (64, 257, 2080)]


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("M,N,K", ACTION_CHUNK_SHAPES)
def test_action_chunk_parity(cuda_device, fmt, M, N, K):
    Y, Yref, B, _, _ = run_case(fmt, M, N, K, seed=M * 11 + N + K)
    check_close(Y, Yref, B, f"action-chunk fmt={fmt} M={M} N={N} K={K}")


@pytest.mark.parametrize("fmt", FMTS)
def test_action_chunk_fused_group_and_determinism(cuda_device, fmt):
    M, K, Ns = 50, 1024, (1024, 128, 128)
    Xb = activation_bits_np(M, K, 71)
    X = to_dev_bf16(Xb)
    specs, host = [], []
    for i, N in enumerate(Ns):
        W = weight_np(N, K, 72 + i)
        img = emb.quantize(fmt, torch.from_numpy(W).cuda())
        Y = torch.full((M, N), float("nan"), dtype=torch.float32, device="cuda")
        specs.append((fmt, img, N, K, X, Y))
        host.append(W)
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    first = [sp[5].clone() for sp in specs]
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    for a, sp in zip(first, specs):
        assert torch.equal(a.view(torch.int32), sp[5].view(torch.int32))
    for (f, img, N, _, _, Y), W in zip(specs, host):
        Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
        check_close(Y.cpu().numpy(), Yref, B, f"fused action-chunk N={N}")


def test_precise_operand_flag_few_dominant_terms(cuda_device):
    """The tensor-core GEMM at K >= 1024 stages bf16(w') (relative error <= 2^-8 per
    weight, bf16's unit roundoff): with activations where a single term dominates sum|w x|
    (one-hot rows), the output error reaches that rounding and so exceeds the 1e-3 * S
    bound for some outputs; the documented (2^-8 + 2^-12) * S + 1e-6 bound holds. With EMB_PRECISE_OPERAND the same layer runs
    with the two-operand weights and meets 1e-3 * S + 1e-6 everywhere."""
    fmt, M, N, K = emb.EMB_Q8_0, 64, 256, 2048
    W = weight_np(N, K, 95)
    img = emb.quantize(fmt, torch.from_numpy(W).cuda())
    ks = (np.arange(M) * 37) % K
    Xb = np.zeros((M, K), dtype=np.uint16)
    Xb[np.arange(M), ks] = 0x3F80                       # e_k: one term per output
    Xb[:, (ks + 1) % K] = 0x3380                        # plus one 2^-24 term (negligible)
    X = to_dev_bf16(Xb)
    Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
    S = (B - 1e-6) / 1e-3
    Yd = torch.empty(M, N, device="cuda")
    Yp = torch.empty(M, N, device="cuda")
    emb.emb_qlayer_seq([(fmt, img, N, K, X, Yd)], M)
    emb.emb_qlayer_seq([(fmt, img, N, K, X, Yp, emb.EMB_EPI_F32 | emb.EMB_PRECISE_OPERAND)], M)
    torch.cuda.synchronize()
    err_d = np.abs(Yd.cpu().numpy().astype(np.float64) - Yref)
    assert (err_d <= (2.0 ** -8 + 2.0 ** -12) * S + 1e-6).all()
    assert (err_d > B).any()            # the single-operand form is not within 1e-3 here
    check_close(Yp.cpu().numpy(), Yref, B, "EMB_PRECISE_OPERAND")
