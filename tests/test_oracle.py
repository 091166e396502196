"""Pins for the CPU oracle: each test checks it against something other than itself
(library conversions, hand-worked blocks, closed forms, exact rational arithmetic,
invariants of the block formats).  CPU only."""
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle
from oracle import Q4_0, Q6_0, Q8_0
from tests.golden_io import read_blocks
from workloads import activation_bits_np, bf16_bits_np, weight_np


# ------------------------------------------------------------------ number conversions

def _stratified_f32_bits():
    """Every exponent and sign, with mantissas that straddle each fp16/bf16 rounding point."""
    rng = np.random.default_rng(7)
    exps = np.arange(256, dtype=np.uint32)
    special_lo = np.array([0, 1, 0xFFF, 0x1000, 0x1001, 0x1FFF, 0x2000, 0x2001, 0x3000,
                           0x7FFF, 0x8000, 0x8001, 0xFFFF, 0x10000, 0x17FFF, 0x18000],
                          dtype=np.uint32)
    hi = rng.integers(0, 1 << 23, size=600, dtype=np.uint32)
    mants = np.unique(np.concatenate([
        (hi[:, None] & ~np.uint32(0x1FFF)) | (special_lo[None, :] & 0x1FFF),
        (hi[:, None] & ~np.uint32(0xFFFF)) | special_lo[None, :],
        rng.integers(0, 1 << 23, size=4000, dtype=np.uint32)[:, None],
        np.array([0, 1, 0x7FFFFF], dtype=np.uint32)[:, None],
    ], axis=None))
    bits = (exps[:, None] << 23) | mants[None, :]
    bits = np.concatenate([bits.ravel(), bits.ravel() | np.uint32(0x80000000)])
    return bits


def test_f16_rounding_matches_numpy():
    bits = _stratified_f32_bits()
    x = bits.view(np.float32)
    finite = ~np.isnan(x)
    with np.errstate(over="ignore"):
        expect = x[finite].astype(np.float16).view(np.uint16)
    got = oracle.f32_to_f16_bits(x[finite])
    bad = np.nonzero(got != expect)[0]
    assert bad.size == 0, f"{bad.size} mismatches, first {x[finite][bad[:5]]}"
    # NaN stays NaN
    nan = oracle.f32_to_f16_bits(np.array([np.nan], dtype=np.float32))[0]
    assert (nan & 0x7C00) == 0x7C00 and (nan & 0x3FF) != 0


def test_f16_to_f32_all_patterns():
    h = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    got = oracle.f16_bits_to_f32(h)
    expect = h.view(np.float16).astype(np.float32)
    same = (got.view(np.uint32) == expect.view(np.uint32)) | (np.isnan(got) & np.isnan(expect))
    assert same.all()


def test_bf16_rounding_matches_torch():
    bits = _stratified_f32_bits()
    x = bits.view(np.float32)
    finite = ~np.isnan(x)
    expect = torch.from_numpy(x[finite].copy()).to(torch.bfloat16).view(torch.int16).numpy()
    got = oracle.f32_to_bf16_bits(x[finite])
    assert np.array_equal(got, expect.view(np.uint16))


# ------------------------------------------------------------------------- layout size

@pytest.mark.parametrize("fmt,N,K,expect", [
    # Q8_0 2048x2048: codes 4194304 B (already 256-aligned) + 2048 rows * 64 halves * 2 B
    (Q8_0, 2048, 2048, 4194304 + 2048 * 64 * 2),
    # Q4_0 3x96: codes 144 B -> scales at 256; K/32 = 3 blocks -> pitch 8 halves
    (Q4_0, 3, 96, 256 + 3 * 8 * 2),
    # Q8_0 1x32: codes 32 -> 256; pitch 8 halves
    (Q8_0, 1, 32, 256 + 16),
    # Q8_0 5x1152: 36 blocks -> pitch 40 halves; codes 5760 -> 5888
    (Q8_0, 5, 1152, 5888 + 5 * 40 * 2),
    # Q6_0 3x96: low plane 144 B -> high plane at 256 (72 B, ends at 328) -> scales at 512
    (Q6_0, 3, 96, 512 + 3 * 8 * 2),
    # Q6_0 2048x2048: low 2097152 B, high 1048576 B (both 256-aligned), scales 2048 * 64 * 2
    (Q6_0, 2048, 2048, 2097152 + 1048576 + 2048 * 64 * 2),
])
def test_packed_bytes(fmt, N, K, expect):
    assert oracle.packed_bytes(fmt, N, K) == expect


@pytest.mark.parametrize("fmt,N,K", [(3, 4, 32), (-1, 4, 32), (Q8_0, 0, 32), (Q8_0, 4, 48),
                                     (Q4_0, 4, 0), (Q6_0, 4, 48), (Q6_0, 0, 64)])
def test_packed_bytes_rejects(fmt, N, K):
    assert oracle.packed_bytes(fmt, N, K) == 0


# ----------------------------------------------------------------- hand-worked blocks

def _image_of_block(fmt, w):
    img = oracle.quantize(fmt, w.reshape(1, 32))
    codes, scales = oracle.split_image(fmt, img, 1, 32)
    return img, codes, scales


@pytest.mark.parametrize("blk", read_blocks("q8_0_blocks.txt", 0), ids=lambda b: b["name"])
def test_q8_0_golden(blk):
    img, codes, scales = _image_of_block(Q8_0, blk["w"])
    assert scales[0, 0] == blk["scale"], hex(scales[0, 0])
    assert np.array_equal(codes.view(np.int8).astype(np.int64), blk["codes"])
    # padding (rest of the scale row, the gap before the scales plane) is zero
    assert not scales[0, 1:].any()
    assert not img[32:256].any()


@pytest.mark.parametrize("blk", read_blocks("q4_0_blocks.txt", 8), ids=lambda b: b["name"])
def test_q4_0_golden(blk):
    img, codes, scales = _image_of_block(Q4_0, blk["w"])
    assert scales[0, 0] == blk["scale"], hex(scales[0, 0])
    assert np.array_equal(codes, blk["bytes"]), codes
    # the listed codes agree with the listed bytes (fixture self-consistency)
    c = blk["codes"]
    assert np.array_equal((c[:16] | (c[16:] << 4)).astype(np.uint8), blk["bytes"])


@pytest.mark.parametrize("blk", read_blocks("q6_0_blocks.txt", 32), ids=lambda b: b["name"])
def test_q6_0_golden(blk):
    img = oracle.quantize(Q6_0, blk["w"].reshape(1, 32))
    _, scales = oracle.split_image(Q6_0, img, 1, 32)
    assert scales[0, 0] == blk["scale"], hex(scales[0, 0])
    assert np.array_equal(img[:16], blk["low"]), img[:16]
    assert np.array_equal(img[256:264], blk["high"]), img[256:264]
    assert np.array_equal(oracle.q6_codes(img, 1, 32)[0], blk["codes"])
    # padding (between the planes, before the scales, rest of the scale row) is zero
    assert not img[16:256].any() and not img[264:512].any() and not scales[0, 1:].any()
    # the listed codes agree with the listed bytes (fixture self-consistency)
    c = blk["codes"]
    assert np.array_equal(((c[:16] & 15) | ((c[16:] & 15) << 4)).astype(np.uint8), blk["low"])
    h = (c[0:8] >> 4) | ((c[8:16] >> 4) << 2) | ((c[16:24] >> 4) << 4) | ((c[24:32] >> 4) << 6)
    assert np.array_equal(h.astype(np.uint8), blk["high"])


def test_golden_dequant_values():
    """Dequantised values of the hand-worked blocks: d*q, d*(q-8), d*(q-32) in exact
    arithmetic."""
    for fmt, fname, dflt in ((Q8_0, "q8_0_blocks.txt", 0), (Q4_0, "q4_0_blocks.txt", 8),
                             (Q6_0, "q6_0_blocks.txt", 32)):
        for blk in read_blocks(fname, dflt):
            img = oracle.quantize(fmt, blk["w"].reshape(1, 32))
            deq = oracle.dequant_f32(fmt, img, 1, 32)[0].astype(np.float64)
            d = float(np.array([blk["scale"]], dtype=np.uint16).view(np.float16)[0])
            q = blk["codes"].astype(np.float64) - {Q8_0: 0, Q4_0: 8, Q6_0: 32}[fmt]
            assert np.array_equal(deq, d * q), blk["name"]


# ------------------------------------------------------------ lossless exact grids

def _grid_weights(fmt, N, K, rng):
    """Weights that each format represents exactly: per block k_i * 2^e with a scale
    that the quantiser recovers exactly (Q8_0: one |k|=127; Q4_0 / Q6_0: the first
    maximum is -8 / -32)."""
    e = rng.integers(-12, 3, size=(N, K // 32))
    if fmt == Q8_0:
        k = rng.integers(-127, 128, size=(N, K))
        k[:, ::32] = np.where(rng.random((N, K // 32)) < 0.5, 127, -127)
    else:
        half = 8 if fmt == Q4_0 else 32
        k = rng.integers(-half + 1, half, size=(N, K))
        k[:, ::32] = -half
    w = k * np.exp2(np.repeat(e, 32, axis=1))
    return w.astype(np.float32), k


@pytest.mark.parametrize("fmt", [Q8_0, Q4_0, Q6_0])
def test_exact_grid_roundtrip(fmt):
    rng = np.random.default_rng(11)
    W, _ = _grid_weights(fmt, 9, 256, rng)
    img = oracle.quantize(fmt, W)
    assert np.array_equal(oracle.dequant_f32(fmt, img, 9, 256), W)
    bf = oracle.dequant_bf16(fmt, img, 9, 256)
    # values with at most 8 significant bits are exact in bf16
    assert np.array_equal(bf, bf16_bits_np(W))


# ------------------------------------------------------------------ round-trip bounds

def _random_blocks(nblocks, rng, lo=1e-2, hi=1e3):
    scale = np.exp(rng.uniform(np.log(lo), np.log(hi), size=(nblocks, 1)))
    w = rng.standard_normal((nblocks, 32)) * scale
    # adversarial rows: single spikes, equal magnitudes of both signs, constant rows
    w[::7, 1:] *= 1e-3
    w[1::7, 5] = -np.abs(w[1::7, 2])
    w[1::7, 2] = np.abs(w[1::7, 2])
    w[2::7] = w[2::7, :1]
    return w.astype(np.float32)


@pytest.mark.parametrize("fmt", [Q8_0, Q4_0, Q6_0])
def test_roundtrip_invariant(fmt):
    rng = np.random.default_rng(3 + fmt)
    nb = 200_000
    W = _random_blocks(nb, rng).reshape(-1, 32 * 50)        # 4000 rows x 50 blocks
    N, K = W.shape
    img = oracle.quantize(fmt, W)
    deq = oracle.dequant_f32(fmt, img, N, K).astype(np.float64)
    _, scales = oracle.split_image(fmt, img, N, K)
    d = np.abs(scales[:, :K // 32].view(np.float16).astype(np.float64))
    d = np.repeat(d, 32, axis=1)
    w = W.astype(np.float64)
    err = np.abs(w - deq)
    slack = np.abs(w) * 2.0 ** -24                           # one binary32 division rounding
    normal = d >= 2.0 ** -14
    assert normal.mean() > 0.98
    if fmt == Q8_0:
        assert (err[normal] <= d[normal] / 2 + slack[normal]).all()
    else:
        t = w / np.where(d == 0, 1, d)
        # sign of d is -sign(m): codes are w/d with d signed; in range means
        # w/d in [-half - 0.5, half - 0.5] (half = 8 for Q4_0, 32 for Q6_0)
        half = 8 if fmt == Q4_0 else 32
        dsigned = np.repeat(scales[:, :K // 32].view(np.float16).astype(np.float64), 32, axis=1)
        t = w / dsigned
        inrange = normal & (t >= -half - 0.5) & (t <= half - 0.5)
        assert inrange.mean() > 0.9
        assert (err[inrange] <= d[inrange] / 2 + slack[inrange]).all()
        # out of range only on the side opposite to m (|d| >= |m|/half (1 - 2^-11)), by less
        # than |d| (1 + half 2^-11)
        assert (t[normal] <= half * (1 + 2.0 ** -10)).all() and (t[normal] >= -half - 0.5).all()
        assert (err[normal] <= d[normal] * (1 + half * 2.0 ** -11) + slack[normal]).all()


@pytest.mark.parametrize("fmt", [Q8_0, Q4_0, Q6_0])
def test_roundtrip_subnormal_scales(fmt):
    """Tiny blocks whose scale is an fp16 subnormal (or rounds to 0): the scale carries an
    absolute rounding error of at most 2^-25, so the bound gains 127*2^-25 (Q8_0),
    8*2^-25 (Q4_0) or 32*2^-25 (Q6_0) on top of the normal-scale bounds."""
    rng = np.random.default_rng(13 + fmt)
    W = _random_blocks(50_000, rng, lo=1e-9, hi=1e-4).reshape(-1, 32 * 50)
    N, K = W.shape
    img = oracle.quantize(fmt, W)
    deq = oracle.dequant_f32(fmt, img, N, K).astype(np.float64)
    _, scales = oracle.split_image(fmt, img, N, K)
    d = np.repeat(np.abs(scales[:, :K // 32].view(np.float16).astype(np.float64)), 32, axis=1)
    w = W.astype(np.float64)
    err = np.abs(w - deq)
    slack = np.abs(w) * 2.0 ** -24
    sub = d < 2.0 ** -14
    assert sub.mean() > 0.5
    if fmt == Q8_0:
        assert (err <= np.maximum(d / 2, 127 * 2.0 ** -25) + slack).all()
    else:
        half = 8 if fmt == Q4_0 else 32
        assert (err <= d * (1 + half * 2.0 ** -11) + half * 2.0 ** -25 + slack).all()


@pytest.mark.parametrize("fmt", [Q8_0, Q4_0, Q6_0])
def test_scale_is_rounded_block_extreme(fmt):
    """d is the fp16 rounding of max|w|/127 (Q8_0) or m/-8 (Q4_0) or m/-32 (Q6_0),
    computed independently."""
    rng = np.random.default_rng(5)
    W = _random_blocks(20_000, rng).reshape(-1, 32 * 40)
    N, K = W.shape
    img = oracle.quantize(fmt, W)
    _, scales = oracle.split_image(fmt, img, N, K)
    blocks = W.reshape(N, K // 32, 32)
    if fmt == Q8_0:
        d32 = np.abs(blocks).max(axis=2) / np.float32(127)
    else:
        idx = np.abs(blocks).argmax(axis=2)                  # first index of the maximum
        m = np.take_along_axis(blocks, idx[..., None], axis=2)[..., 0]
        d32 = m / np.float32(-8 if fmt == Q4_0 else -32)
    with np.errstate(over="ignore"):
        expect = d32.astype(np.float32).astype(np.float16).view(np.uint16)
    assert np.array_equal(scales[:, :K // 32], expect)


def test_codes_round_half_away_vs_numpy():
    """Codes equal numpy's round-half-away of w/d on random blocks (independent decode)."""
    rng = np.random.default_rng(9)
    W = _random_blocks(10_000, rng).reshape(-1, 32 * 25)
    N, K = W.shape
    for fmt in (Q8_0, Q4_0, Q6_0):
        img = oracle.quantize(fmt, W)
        codes, scales = oracle.split_image(fmt, img, N, K)
        d = np.repeat(scales[:, :K // 32].view(np.float16).astype(np.float32), 32, axis=1)
        with np.errstate(divide="ignore", invalid="ignore"):
            t = (W / d).astype(np.float32)
        r = np.sign(t) * np.floor(np.abs(t) + np.float32(0.5))
        if fmt == Q8_0:
            expect = np.where(d == 0, 0, np.clip(r, -127, 127)).astype(np.int64)
            got = codes.view(np.int8).reshape(N, K).astype(np.int64)
        elif fmt == Q4_0:
            expect = np.where(d == 0, 8, np.clip(r, -8, 7) + 8).astype(np.int64)
            b = codes.reshape(N, K // 32, 16)
            got = np.concatenate([b & 0xF, b >> 4], axis=2).reshape(N, K).astype(np.int64)
        else:
            expect = np.where(d == 0, 32, np.clip(r, -32, 31) + 32).astype(np.int64)
            got = oracle.q6_codes(img, N, K)
        assert np.array_equal(got, expect)


# ----------------------------------------------------------------------------- matmul

def _exact_Y(W, Xf):
    """Exact rational Y[m][n] = sum_k W[n][k] X[m][k] and sum |.| from the raw inputs."""
    M, K = Xf.shape
    N = W.shape[0]
    Y = [[Fraction(0)] * N for _ in range(M)]
    A = [[Fraction(0)] * N for _ in range(M)]
    for m in range(M):
        for n in range(N):
            s = Fraction(0)
            a = Fraction(0)
            for k in range(K):
                p = Fraction(float(W[n, k])) * Fraction(float(Xf[m, k]))
                s += p
                a += abs(p)
            Y[m][n] = s
            A[m][n] = a
    return Y, A


@pytest.mark.parametrize("fmt", [Q8_0, Q4_0, Q6_0])
@pytest.mark.parametrize("M,N,K", [(1, 1, 32), (3, 4, 64), (4, 3, 32), (2, 2, 96)])
def test_matmul_brute_force_exact(fmt, M, N, K):
    rng = np.random.default_rng(100 + M * 10 + N + K)
    W, _ = _grid_weights(fmt, N, K, rng)                     # quantised without loss
    # dyadic activations with 7-bit numerators: every product and every partial sum is
    # exact in fp64, so the oracle must reproduce the rational result bit for bit.
    Xf = (rng.integers(-127, 128, size=(M, K)) * np.exp2(rng.integers(-6, 2, size=(M, K))))
    Xf = Xf.astype(np.float32)
    X = bf16_bits_np(Xf)
    assert np.array_equal(X.astype(np.uint32) << 16, Xf.view(np.uint32))
    img = oracle.quantize(fmt, W)
    Y, B = oracle.qmatmul(fmt, img, X, N, K, nthreads=1)
    Ye, Ae = _exact_Y(W, Xf)
    for m in range(M):
        for n in range(N):
            assert Fraction(Y[m, n]) == Ye[m][n]
            assert B[m, n] == pytest.approx(float(Ae[m][n]) * 1e-3 + 1e-6, rel=1e-15)


def test_matmul_constant_weights_give_row_sums():
    """W = c everywhere (Q8_0): every code is 127 and w' = 127*d, so Y[m][n] = w' * sum_k x."""
    M, N, K = 3, 5, 128
    c = np.float32(0.3)
    W = np.full((N, K), c, dtype=np.float32)
    X = activation_bits_np(M, K, 21)
    img = oracle.quantize(Q8_0, W)
    codes, scales = oracle.split_image(Q8_0, img, N, K)
    assert (codes.view(np.int8) == 127).all()
    wq = Fraction(float(np.float16(c / np.float32(127)))) * 127
    Y, _ = oracle.qmatmul(Q8_0, img, X, N, K)
    xs = (X.astype(np.uint32) << 16).view(np.float32)
    for m in range(M):
        expect = wq * sum(Fraction(float(v)) for v in xs[m])
        assert np.allclose(Y[m], float(expect), rtol=1e-15, atol=0)


def test_matmul_orientation_identity():
    """W = s*I (32x32): Y[m][n] = w'_nn * x[m][n] -- catches a transposed operand."""
    K = N = 32
    M = 4
    s = np.float32(0.75)
    W = np.eye(N, K, dtype=np.float32) * s
    W[3, 3] = -s
    X = activation_bits_np(M, K, 4)
    xs = (X.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
    for fmt in (Q8_0, Q4_0, Q6_0):
        img = oracle.quantize(fmt, W)
        diag = np.diag(oracle.dequant_f32(fmt, img, N, K)).astype(np.float64)
        Y, _ = oracle.qmatmul(fmt, img, X, N, K)
        assert np.array_equal(Y, xs * diag[None, :])
        # and the diagonal itself is the closed-form quantisation of +-s
        if fmt == Q8_0:
            d = float(np.float16(s / np.float32(127)))
            assert np.all(np.abs(diag) == 127 * d)
        else:
            assert np.all(np.abs(diag) == s)            # s/8, s/32 are exact in fp16


def test_matmul_matches_numpy_fp64():
    """Random shapes: the oracle's sequential fp64 sum vs numpy's fp64 matmul (BLAS)."""
    for fmt in (Q8_0, Q4_0, Q6_0):
        M, N, K = 5, 70, 320
        W = weight_np(N, K, 30 + fmt)
        X = activation_bits_np(M, K, 31 + fmt)
        img = oracle.quantize(fmt, W)
        deq = oracle.dequant_f32(fmt, img, N, K).astype(np.float64)
        xs = (X.astype(np.uint32) << 16).view(np.float32).astype(np.float64)
        Y, B = oracle.qmatmul(fmt, img, X, N, K)
        Yn = xs @ deq.T
        mag = np.abs(xs) @ np.abs(deq).T
        assert np.all(np.abs(Y - Yn) <= 1e-13 * mag)
        assert np.allclose(B, 1e-3 * mag + 1e-6, rtol=1e-12, atol=0)


def test_threaded_and_sampled_agree():
    N, K, M = 37, 96, 3
    W = weight_np(N, K, 41)
    X = activation_bits_np(M, K, 42)
    for fmt in (Q8_0, Q4_0, Q6_0):
        img = oracle.quantize(fmt, W)
        Y1, B1 = oracle.qmatmul(fmt, img, X, N, K, nthreads=1)
        Y4, B4 = oracle.qmatmul(fmt, img, X, N, K, nthreads=4)
        assert np.array_equal(Y1, Y4) and np.array_equal(B1, B4)
        ms = np.array([0, 2, 1, 2])
        ns = np.array([0, 36, 17, 5])
        Ys, Bs = oracle.qmatmul_sampled(fmt, img, X, N, K, ms, ns)
        assert np.array_equal(Ys, Y1[ms, ns]) and np.array_equal(Bs, B1[ms, ns])


def test_quantize_rows_are_independent():
    """Quantising a subset of rows gives exactly those rows of the full image
    (what the sampled full-size parity checks rely on)."""
    N, K = 12, 160
    W = weight_np(N, K, 51)
    for fmt in (Q8_0, Q4_0, Q6_0):
        full = oracle.quantize(fmt, W)
        cf, sf = oracle.split_image(fmt, full, N, K)
        rows = [0, 5, 11]
        sub = oracle.quantize(fmt, W[rows])
        cs, ss = oracle.split_image(fmt, sub, len(rows), K)
        planes = [(0, K)] if fmt == Q8_0 else [(0, K // 2)] if fmt == Q4_0 else \
            [(0, K // 2), (N * K // 2, K // 4)]       # (plane start in cf, bytes per row)
        for i, r in enumerate(rows):
            so = 0
            for start, rb in planes:
                sub_start = start * len(rows) // N
                assert np.array_equal(cs[sub_start + i * rb:sub_start + (i + 1) * rb],
                                      cf[start + r * rb:start + (r + 1) * rb])
            assert np.array_equal(ss[i], sf[r])
