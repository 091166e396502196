"""The dequantised weights that the timed kernels themselves compute, compared with the
oracle value by value.

emb_dequantize_f32/bf16 run a separate export kernel; the GEMV and GEMM kernels each
dequantise in their own way (byte-permute magic numbers and FFMA2 in the GEMV, LOP3 nibble
to bf16 conversion in the Q4_0 mma.sync GEMV, an FFMA2 on a byte-permuted 2^15 + code and
a bf16 pack in the tcgen05 GEMM). Here they are observed directly through emb_qmatmul: an
activation row that is the unit vector e_k turns output m into column k of the dequantised
matrix, because every product but one is zero and the one left is w' * 1.

  * GEMV (M <= 4): the products are exact in fp32 and every sum adds zeros to one term,
    so Y[m][n] must equal the oracle's w'[n][k_m] (Table 3's 8-, 6- and 4-bit weights as
    dequantised by the oracle: w' = d*q, d*(q-32), d*(q-8), exact in fp32).
  * tcgen05 GEMM at K >= 1024: the MMA operand is bf16(w'), one round-to-nearest-even of
    the exact w', so Y[m][n] must equal the oracle's bf16 dequantisation widened to fp32.
  * tcgen05 GEMM at K < 1024: the kernel adds a second operand lo = bf16(w' - bf16(w'))
    (see the kernel's precision note), so Y must equal hi + lo, which is exact in fp32
    (at most 17 significant bits).

Zeros are compared by value: a dequantised zero is -0 when its scale is negative, while a
sum that starts from +0 gives +0; the sign of a zero output is not part of the contract.

The packed images are written here byte by byte in the documented layout (codes plane,
Q6_0 high-bits plane, fp16 scales plane), so that every code value occurs at every
position of a block (all 256 Q8_0 bytes including -128, all 16 Q4_0 nibbles in both
halves of a byte, all 64 Q6_0 codes in both planes), with normal, subnormal, zero,
negative and largest finite fp16 scales.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb

ONE_BF16 = 0x3F80


def _r256(v: int) -> int:
    return (v + 255) // 256 * 256


def _scales(N: int, K: int, seed: int) -> np.ndarray:
    """fp16 scale bit patterns [N][K/32]: mostly random normals of either sign, plus every
    kind of special finite value (zeros of both signs, subnormals, the smallest normal,
    the largest finite) spread over rows and block positions."""
    rng = np.random.default_rng(seed)
    nb = K // 32
    mag = rng.uniform(2.0 ** -14, 4.0, size=(N, nb)).astype(np.float16).view(np.uint16)
    sign = (rng.random((N, nb)) < 0.5).astype(np.uint16) << 15
    s = mag | sign
    special = np.array([0x0000, 0x8000, 0x0001, 0x8001, 0x03FF, 0x83FF, 0x0200, 0x0400,
                        0x8400, 0x7BFF, 0xFBFF, 0x3C00, 0xBC00], dtype=np.uint16)
    idx = (np.arange(N)[:, None] * 3 + np.arange(nb)[None, :] * 5) % 29
    pick = idx < special.size
    s[pick] = special[idx[pick]]
    return s


def crafted_image(fmt: int, N: int, K: int, seed: int) -> np.ndarray:
    """A packed image whose codes run through every value at every position: the code of
    (row n, column k) is (a n + b k) mod 2^bits with a odd, so any 2^bits consecutive rows
    hold every code at every column."""
    n = np.arange(N, dtype=np.int64)[:, None]
    k = np.arange(K, dtype=np.int64)[None, :]
    total = oracle.packed_bytes(fmt, N, K)
    img = np.zeros(total, dtype=np.uint8)
    ldS = (K // 32 + 7) // 8 * 8
    if fmt == emb.EMB_Q8_0:
        q = ((37 * n + 11 * k) & 255).astype(np.uint8)
        img[:N * K] = q.reshape(-1)
        soff = _r256(N * K)
    else:
        bits = 4 if fmt == emb.EMB_Q4_0 else 6
        q = (((5 if bits == 4 else 7) * n + 3 * k + 1) & ((1 << bits) - 1)).astype(np.uint8)
        blk = q.reshape(N, K // 32, 32)
        lo = (blk[:, :, :16] & 15) | ((blk[:, :, 16:] & 15) << 4)
        img[:N * K // 2] = lo.reshape(-1)
        soff = _r256(N * K // 2)
        if bits == 6:
            h = blk >> 4
            hi = (h[:, :, 0:8] | (h[:, :, 8:16] << 2) | (h[:, :, 16:24] << 4) | (h[:, :, 24:32] << 6))
            hoff = soff
            img[hoff:hoff + N * K // 4] = hi.astype(np.uint8).reshape(-1)
            soff = _r256(hoff + N * K // 4)
    sc = np.zeros((N, ldS), dtype=np.uint16)
    sc[:, :K // 32] = _scales(N, K, seed)
    img[soff:soff + N * ldS * 2] = sc.view(np.uint8).reshape(-1)
    assert soff + N * ldS * 2 == total
    return img


def onehot_rows(ks, K: int) -> torch.Tensor:
    """bf16 device rows e_{k} for each k in ks (bit patterns: 1.0 = 0x3F80)."""
    x = np.zeros((len(ks), K), dtype=np.uint16)
    x[np.arange(len(ks)), np.asarray(ks)] = ONE_BF16
    return torch.from_numpy(x.view(np.int16)).cuda().view(torch.bfloat16)


def run_onehot(fmt: int, img_dev: torch.Tensor, N: int, K: int, M: int, ks) -> np.ndarray:
    """Y rows for the given k positions, M rows per emb_qmatmul call (the last call takes
    what is left); row p of the result is the call's output for activation e_{ks[p]}."""
    X = onehot_rows(ks, K)
    P = len(ks)
    # one-token calls write one row each: a row pitch of a multiple of four floats keeps
    # every call's output 16-byte aligned whatever N is
    pitch = (N + 3) // 4 * 4 if M == 1 else N
    Y = torch.full((P, pitch), float("nan"), dtype=torch.float32, device="cuda")
    for j in range(0, P, M):
        m = min(M, P - j)
        emb.emb_qmatmul(fmt, img_dev, X[j].data_ptr(), Y[j].data_ptr(), m, N, K)
    torch.cuda.synchronize()
    assert emb.emb_device_status() == emb.EMB_OK
    return Y[:, :N].cpu().numpy()


def _assert_columns_equal(Y: np.ndarray, W: np.ndarray, ks, what: str) -> None:
    """Y[p][n] == W[n][ks[p]] for every p, n (values; zeros of either sign are equal)."""
    expect = np.ascontiguousarray(W[:, np.asarray(ks)].T)
    assert np.isfinite(Y).all(), f"{what}: non-finite output"
    bad = Y != expect
    if bad.any():
        p, n = np.argwhere(bad)[0]
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} values differ; first at "
                             f"k={ks[p]} n={n}: got {Y[p, n]!r} want {expect[p, n]!r}")


def _bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << 16).view(np.float32)


def _hi_lo(fmt: int, img: np.ndarray, N: int, K: int) -> np.ndarray:
    """hi + lo of the split operand: hi = bf16(w'), lo = bf16(w' - hi), both nearest-even,
    summed exactly (fp64, then fp32: at most 17 significant bits)."""
    w = oracle.dequant_f32(fmt, img, N, K).astype(np.float64)
    hi = _bf16_to_f32(oracle.dequant_bf16(fmt, img, N, K)).astype(np.float64)
    lo = oracle.bf16_round((w - hi).astype(np.float32))  # w - hi is exact in fp32
    s = hi + lo
    assert np.array_equal(s.astype(np.float32).astype(np.float64), s)
    return s.astype(np.float32)


def _all_k(K: int):
    return list(range(K))


def _spread_k(K: int, count: int, seed: int):
    """Every position of the first two 32-blocks, every residue mod 256 (the tensor-core
    GEMM's raw-stage period), and random others; at most `count` more, distinct."""
    ks = list(range(min(64, K)))
    ks += [(257 * m + 64) % K for m in range(min(256, K))]
    rng = np.random.default_rng(seed)
    ks += rng.integers(0, K, size=count).tolist()
    seen, out = set(), []
    for k in ks:
        if k not in seen:
            seen.add(k)
            out.append(int(k))
    return out


# ---------------------------------------------------------------- GEMV (M <= 4)
# (fmt, N, K, M, which kernel the shape routes to, k positions)
GEMV_CASES = [
    # register kernel, one row per CTA (small layer), every k; M = 1, 2 (two tokens per
    # CTA), 3 and 4 (four-token tiles)
    (emb.EMB_Q8_0, 256, 2048, 1, "register R=1", "all"),
    (emb.EMB_Q8_0, 256, 2048, 2, "register R=1 MT=2", "all"),
    (emb.EMB_Q8_0, 256, 2048, 3, "register R=1 MT=4", "all"),
    (emb.EMB_Q4_0, 256, 2048, 1, "register R=1", "all"),
    (emb.EMB_Q4_0, 256, 2048, 4, "register R=1 MT=4", "all"),
    (emb.EMB_Q6_0, 256, 2048, 1, "register R=1", "all"),
    (emb.EMB_Q6_0, 256, 2048, 4, "register R=1 MT=4", "all"),
    # Q6_0 with K % 64 != 0 (no staged or tensor-map path)
    (emb.EMB_Q6_0, 256, 1056, 2, "register R=1", "all"),
    # four rows per CTA (2048 rows, 16-byte units per row < 320)
    (emb.EMB_Q4_0, 2048, 2048, 1, "register R=4", "all"),
    (emb.EMB_Q8_0, 2048, 2048, 2, "register R=4 MT=2", "all"),
    # long Q8_0 rows below 12 MB: a thread's whole row share loaded before the wait (PF = 4)
    (emb.EMB_Q8_0, 256, 16384, 1, "register PF=4 R=1", "spread"),
    (emb.EMB_Q6_0, 1024, 8192, 1, "register R=2 long rows (< 12 MB)", "spread"),
    (emb.EMB_Q6_0, 2048, 16384, 1, "ring, Q6_0 high plane in the stage", "spread"),
    # ring kernel (rows > 6 KB, >= 12 MB, M = 1: X in registers, rows through a shared-memory
    # ring): the Gemma-2B down projection shape, 2..4 units per thread, ragged last CTAs
    (emb.EMB_Q8_0, 2048, 16384, 1, "ring PF=4", "spread"),
    (emb.EMB_Q8_0, 2048, 8192, 1, "ring PF=2", "spread"),
    (emb.EMB_Q8_0, 1027, 12288, 1, "ring PF=3, ragged last CTA", "spread"),
    (emb.EMB_Q4_0, 2048, 16384, 1, "ring PF=2", "spread"),
    (emb.EMB_Q4_0, 1024, 24576, 1, "ring PF=3", "spread"),
    (emb.EMB_Q4_0, 1538, 16384, 1, "ring, ragged last CTA", "spread"),
    (emb.EMB_Q4_0, 1539, 16384, 1, "ring, ragged last CTA", "spread"),
    # staged kernel: >= 12 MB of codes with rows <= 6 KB at M = 1; any rows at M = 2..4
    (emb.EMB_Q8_0, 6144, 2048, 1, "staged", "all"),
    (emb.EMB_Q8_0, 6144, 2048, 4, "staged MT=4", "all"),
    (emb.EMB_Q4_0, 12288, 2048, 1, "staged", "all"),
    (emb.EMB_Q4_0, 4096, 12288, 1, "staged, 6 KB rows", "spread"),
    (emb.EMB_Q6_0, 8192, 2048, 1, "staged", "all"),
    (emb.EMB_Q6_0, 8192, 2048, 2, "staged MT=2", "all"),
    # Q4_0 mma.sync kernel: >= 12 MB, rows <= 2 KB, M = 2..4
    (emb.EMB_Q4_0, 12288, 2048, 2, "q4 mma.sync", "all"),
    (emb.EMB_Q4_0, 12288, 2048, 3, "q4 mma.sync", "all"),
    (emb.EMB_Q4_0, 12288, 4096, 4, "q4 mma.sync", "spread"),
]


@pytest.mark.gpu
@pytest.mark.parametrize("fmt,N,K,M,path,which", GEMV_CASES,
                         ids=[f"{emb_fmt}-{N}x{K}-M{M}-{path.replace(' ', '_')}"
                              for emb_fmt, N, K, M, path, _ in GEMV_CASES])
def test_gemv_dequant_exact(cuda_device, fmt, N, K, M, path, which):
    img = crafted_image(fmt, N, K, seed=N + K + fmt)
    ks = _all_k(K) if which == "all" else _spread_k(K, 256, seed=K + M)
    Y = run_onehot(fmt, torch.from_numpy(img).cuda(), N, K, M, ks)
    W = oracle.dequant_f32(fmt, img, N, K)
    _assert_columns_equal(Y, W, ks, f"GEMV {path} fmt={fmt} {N}x{K} M={M}")


# ---------------------------------------------------------------- GEMM (M > 4)
# (fmt, N, K, M, which kernel variant the shape takes, k positions)
GEMM_CASES = [
    # X = the identity (M = K): Y is the whole dequantised matrix, transposed
    (emb.EMB_Q8_0, 384, 1024, 1024, "identity, bf16 operand", "identity"),
    (emb.EMB_Q4_0, 384, 1024, 1024, "identity, bf16 operand", "identity"),
    (emb.EMB_Q6_0, 384, 1024, 1024, "identity, bf16 operand", "identity"),
    (emb.EMB_Q8_0, 256, 512, 512, "identity, hi + lo operand", "identity"),
    (emb.EMB_Q4_0, 256, 512, 512, "identity, hi + lo operand", "identity"),
    (emb.EMB_Q6_0, 256, 512, 512, "identity, hi + lo operand", "identity"),
    # the action chunk (50 tokens): one tile per CTA, K split over a cluster
    (emb.EMB_Q8_0, 1024, 4096, 50, "M=50 split-K cluster", "spread"),
    (emb.EMB_Q6_0, 1024, 4096, 50, "M=50 split-K cluster", "spread"),
    (emb.EMB_Q4_0, 256, 640, 50, "M=50 hi + lo operand", "spread"),
    # prefill: two token tiles per CTA sharing each A tile (Llama-style q/k/v at M = 280)
    (emb.EMB_Q4_0, 12288, 4096, 280, "M=280 two token tiles per CTA", "spread"),
    # prefill: one 208-token tile per CTA (M = 816)
    (emb.EMB_Q8_0, 2048, 2048, 816, "M=816 one tile per CTA", "spread"),
    (emb.EMB_Q6_0, 2048, 2048, 816, "M=816 one tile per CTA", "spread"),
    # prefill with more tiles than SMs: persistent CTAs looping over (weight, token) tiles
    (emb.EMB_Q8_0, 10240, 1024, 816, "M=816 persistent CTAs", "spread"),
    (emb.EMB_Q4_0, 10240, 1024, 816, "M=816 persistent CTAs", "spread"),
]


@pytest.mark.gpu
@pytest.mark.parametrize("fmt,N,K,M,path,which", GEMM_CASES,
                         ids=[f"{emb_fmt}-{N}x{K}-M{M}" for emb_fmt, N, K, M, _, _ in GEMM_CASES])
def test_gemm_dequant_exact(cuda_device, fmt, N, K, M, path, which):
    img = crafted_image(fmt, N, K, seed=3 * N + K + fmt)
    ks = _all_k(K) if which == "identity" else _spread_k(K, 2 * M, seed=K + M)
    Y = run_onehot(fmt, torch.from_numpy(img).cuda(), N, K, M, ks)
    if K >= 1024:
        W = _bf16_to_f32(oracle.dequant_bf16(fmt, img, N, K))
    else:
        W = _hi_lo(fmt, img, N, K)
    _assert_columns_equal(Y, W, ks, f"GEMM {path} fmt={fmt} {N}x{K} M={M}")


def test_crafted_image_covers_every_code():
    """CPU check of the test input itself: the crafted images hold every code value at
    every block position, and every special scale value somewhere."""
    for fmt, bits, N in ((emb.EMB_Q8_0, 8, 256), (emb.EMB_Q4_0, 4, 16), (emb.EMB_Q6_0, 6, 64)):
        K = 1056
        img = crafted_image(fmt, N, K, seed=1)
        if fmt == emb.EMB_Q8_0:
            q = img[:N * K].reshape(N, K)
        elif fmt == emb.EMB_Q4_0:
            lo = img[:N * K // 2].reshape(N, K // 32, 16)
            q = np.concatenate([lo & 15, lo >> 4], axis=2).reshape(N, K)
        else:
            q = oracle.q6_codes(img, N, K)
        for k in range(K):
            assert len(np.unique(q[:, k])) == 1 << bits, (fmt, k)
        _, sc = oracle.split_image(fmt, img, N, K)
        want = {0x0000, 0x8000, 0x0001, 0x8001, 0x03FF, 0x0400, 0x7BFF, 0xFBFF}
        assert want <= set(np.unique(sc[:, :K // 32]).tolist()), fmt
        # finite scales only (NaN / Inf scales are outside the contract)
        assert ((sc & 0x7C00) != 0x7C00).all()
