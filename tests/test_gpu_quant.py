"""GPU packing and dequantisation are bit-exact against the oracle (whole packed
image, padding included; fp32 and bf16 dequantised values)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
from tests.golden_io import read_blocks
from tests.gpu_util import gpu_quantize
from workloads import weight_np

pytestmark = pytest.mark.gpu

SHAPES = [(1, 32), (3, 96), (7, 160), (128, 1024), (136, 1152), (256, 2048), (5, 4608),
          (33, 11008)]


def _adversarial(N, K, seed):
    W = weight_np(N, K, seed)
    rng = np.random.default_rng(seed)
    blocks = W.reshape(N, K // 32, 32)
    # ties at half-codes, equal +-max, zero blocks, tiny (fp16-subnormal) scales
    blocks[0, 0, :] = 0.0
    if K >= 64:
        blocks[0, 1, :] = np.float32(rng.standard_normal(32) * 1e-6)
    if N > 1:
        blocks[1, 0, 3] = 0.5
        blocks[1, 0, 7] = -0.5
    if N > 2:
        blocks[2, 0, :] = np.arange(32, dtype=np.float32) * np.float32(0.5) - 8
    return W


@pytest.mark.parametrize("fmt", [emb.EMB_Q8_0, emb.EMB_Q4_0, emb.EMB_Q6_0])
@pytest.mark.parametrize("N,K", SHAPES)
def test_pack_bit_exact(cuda_device, fmt, N, K):
    W = _adversarial(N, K, 100 + N + K)
    img = gpu_quantize(fmt, W).cpu().numpy()
    ref = oracle.quantize(fmt, W)
    assert img.shape == ref.shape
    diff = np.nonzero(img != ref)[0]
    assert diff.size == 0, f"{diff.size} bytes differ, first at {diff[:8]}"


@pytest.mark.parametrize("fmt,fname,dflt", [(emb.EMB_Q8_0, "q8_0_blocks.txt", 0),
                                            (emb.EMB_Q4_0, "q4_0_blocks.txt", 8),
                                            (emb.EMB_Q6_0, "q6_0_blocks.txt", 32)])
def test_pack_golden_blocks(cuda_device, fmt, fname, dflt):
    blocks = read_blocks(fname, dflt)
    W = np.stack([b["w"] for b in blocks]).astype(np.float32)   # one row per block
    img = gpu_quantize(fmt, W).cpu().numpy()
    codes, scales = oracle.split_image(fmt, img, len(blocks), 32)
    for i, b in enumerate(blocks):
        assert scales[i, 0] == b["scale"], b["name"]
        if fmt == emb.EMB_Q8_0:
            assert np.array_equal(codes[32 * i:32 * i + 32].view(np.int8), b["codes"]), b["name"]
        elif fmt == emb.EMB_Q4_0:
            assert np.array_equal(codes[16 * i:16 * i + 16], b["bytes"]), b["name"]
        else:   # low plane (16 bytes per block), then the high plane (8 bytes per block)
            n = len(blocks)
            assert np.array_equal(codes[16 * i:16 * i + 16], b["low"]), b["name"]
            assert np.array_equal(codes[16 * n + 8 * i:16 * n + 8 * i + 8], b["high"]), b["name"]


@pytest.mark.parametrize("fmt", [emb.EMB_Q8_0, emb.EMB_Q4_0, emb.EMB_Q6_0])
@pytest.mark.parametrize("N,K", [(3, 96), (136, 1152), (64, 4096)])
def test_dequant_bit_exact(cuda_device, fmt, N, K):
    W = _adversarial(N, K, 7 + K)
    img_ref = oracle.quantize(fmt, W)
    img = torch.from_numpy(img_ref).cuda()   # the oracle's own image: tests dequant alone
    out32 = torch.empty(N, K, dtype=torch.float32, device="cuda")
    out16 = torch.empty(N, K, dtype=torch.int16, device="cuda")
    emb.emb_dequantize_f32(fmt, img, N, K, out32)
    emb.emb_dequantize_bf16(fmt, img, N, K, out16)
    torch.cuda.synchronize()
    assert np.array_equal(out32.cpu().numpy().view(np.uint32),
                          oracle.dequant_f32(fmt, img_ref, N, K).view(np.uint32))
    assert np.array_equal(out16.cpu().numpy().view(np.uint16),
                          oracle.dequant_bf16(fmt, img_ref, N, K))


def test_quantize_is_stream_ordered(cuda_device):
    """Quantise on a side stream, consume on it, without host syncs in between."""
    s = torch.cuda.Stream()
    W = weight_np(256, 2048, 5)
    with torch.cuda.stream(s):
        Wd = torch.from_numpy(W).cuda(non_blocking=False)
        img = emb.quantize(emb.EMB_Q8_0, Wd, stream=s)
    s.synchronize()
    assert np.array_equal(img.cpu().numpy(), oracle.quantize(emb.EMB_Q8_0, W))
