"""CPU oracle for the block-quantised matmul (TEST INFRASTRUCTURE ONLY).

A plain, slow, obviously-correct restatement of the computation in C++
(``emb_oracle.cpp``), wrapped here with ctypes + numpy.  Only ``tests/``,
``__graft_entry__.smoke()`` and ``bench.py``'s cpu_baseline / reference leg may
import this package.  It shares no code with the CUDA library
(``paper_2607_02501_gb300``) and neither imports the other.

What it computes follows the paper's 8-, 6- and 4-bit weight configurations
(Section 4 "Evaluation", Table 3); the block formats themselves are not given in
the paper and are the readings stated in ``emb_oracle.cpp``'s header.
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "emb_oracle.cpp")
_OUT_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_OUT_DIR, "liboracle.so")

Q8_0 = 0
Q4_0 = 1
Q6_0 = 2

_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle with the host g++ (portable C++17, no -march flags)."""
    os.makedirs(_OUT_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    # -ffp-contract=off: no fused multiply-add contraction, so results match across hosts.
    cmd = ["g++", "-O2", "-std=c++17", "-fPIC", "-shared", "-pthread",
           "-ffp-contract=off", "-fno-fast-math", _SRC, "-o", tmp]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    if _lib is not None:
        return _lib
    lib = ctypes.CDLL(build())
    i64, i32, vp = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p
    lib.ref_f32_to_f16.argtypes = [ctypes.c_float]
    lib.ref_f32_to_f16.restype = ctypes.c_uint16
    lib.ref_f16_to_f32.argtypes = [ctypes.c_uint16]
    lib.ref_f16_to_f32.restype = ctypes.c_float
    lib.ref_f32_to_bf16.argtypes = [ctypes.c_float]
    lib.ref_f32_to_bf16.restype = ctypes.c_uint16
    lib.ref_bf16_to_f32.argtypes = [ctypes.c_uint16]
    lib.ref_bf16_to_f32.restype = ctypes.c_float
    lib.ref_packed_bytes.argtypes = [i32, i64, i64]
    lib.ref_packed_bytes.restype = i64
    lib.ref_quantize.argtypes = [i32, vp, i64, i64, vp]
    lib.ref_quantize.restype = i32
    lib.ref_dequant_f32.argtypes = [i32, vp, i64, i64, vp]
    lib.ref_dequant_f32.restype = i32
    lib.ref_dequant_bf16.argtypes = [i32, vp, i64, i64, vp]
    lib.ref_dequant_bf16.restype = i32
    lib.ref_qmatmul.argtypes = [i32, vp, vp, i64, i64, i64, vp, vp, i32]
    lib.ref_qmatmul.restype = i32
    lib.ref_qmatmul_sampled.argtypes = [i32, vp, vp, i64, i64, i64, vp, vp, i64, vp, vp]
    lib.ref_qmatmul_sampled.restype = i32
    for name in ("ref_f32_to_f16_n", "ref_f16_to_f32_n", "ref_f32_to_bf16_n"):
        getattr(lib, name).argtypes = [vp, vp, i64]
        getattr(lib, name).restype = None
    lib.ref_host_threads.argtypes = []
    lib.ref_host_threads.restype = i32
    _lib = lib
    return lib


def _ptr(a: np.ndarray) -> int:
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data


def host_threads() -> int:
    """Threads in this process's CPU affinity mask."""
    return int(_load().ref_host_threads())


def f32_to_f16_bits(x) -> np.ndarray:
    """binary32 -> binary16 bit patterns, round to nearest even."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    _load().ref_f32_to_f16_n(_ptr(x), _ptr(out), x.size)
    return out


def f16_bits_to_f32(h) -> np.ndarray:
    h = np.ascontiguousarray(h, dtype=np.uint16)
    out = np.empty(h.shape, dtype=np.float32)
    _load().ref_f16_to_f32_n(_ptr(h), _ptr(out), h.size)
    return out


def f32_to_bf16_bits(x) -> np.ndarray:
    """binary32 -> bfloat16 bit patterns, round to nearest even."""
    x = np.ascontiguousarray(x, dtype=np.float32)
    out = np.empty(x.shape, dtype=np.uint16)
    _load().ref_f32_to_bf16_n(_ptr(x), _ptr(out), x.size)
    return out


def packed_bytes(fmt: int, N: int, K: int) -> int:
    return int(_load().ref_packed_bytes(fmt, N, K))


def quantize(fmt: int, W: np.ndarray) -> np.ndarray:
    """fp32 W [N][K] -> packed image (uint8, whole buffer including zero padding)."""
    W = np.ascontiguousarray(W, dtype=np.float32)
    N, K = W.shape
    nbytes = packed_bytes(fmt, N, K)
    if nbytes == 0:
        raise ValueError(f"invalid shape for the oracle: fmt={fmt} N={N} K={K}")
    out = np.zeros(nbytes, dtype=np.uint8)
    rc = _load().ref_quantize(fmt, _ptr(W), N, K, _ptr(out))
    if rc:
        raise ValueError("ref_quantize failed")
    return out


def dequant_f32(fmt: int, img: np.ndarray, N: int, K: int) -> np.ndarray:
    out = np.empty((N, K), dtype=np.float32)
    img = np.ascontiguousarray(img, dtype=np.uint8)
    if _load().ref_dequant_f32(fmt, _ptr(img), N, K, _ptr(out)):
        raise ValueError("ref_dequant_f32 failed")
    return out


def dequant_bf16(fmt: int, img: np.ndarray, N: int, K: int) -> np.ndarray:
    """bf16 bit patterns (uint16) of the once-rounded dequantised weights."""
    out = np.empty((N, K), dtype=np.uint16)
    img = np.ascontiguousarray(img, dtype=np.uint8)
    if _load().ref_dequant_bf16(fmt, _ptr(img), N, K, _ptr(out)):
        raise ValueError("ref_dequant_bf16 failed")
    return out


def qmatmul(fmt: int, img: np.ndarray, X_bf16_bits: np.ndarray, N: int, K: int,
            nthreads: int = 0):
    """Y [M][N] fp64 and its per-element tolerance bound, from bf16 X bits [M][K]."""
    X = np.ascontiguousarray(X_bf16_bits, dtype=np.uint16)
    M = X.shape[0]
    assert X.shape == (M, K)
    img = np.ascontiguousarray(img, dtype=np.uint8)
    Y = np.empty((M, N), dtype=np.float64)
    B = np.empty((M, N), dtype=np.float64)
    if _load().ref_qmatmul(fmt, _ptr(img), _ptr(X), M, N, K, _ptr(Y), _ptr(B), nthreads):
        raise ValueError("ref_qmatmul failed")
    return Y, B


def qmatmul_sampled(fmt: int, img: np.ndarray, X_bf16_bits: np.ndarray, N: int, K: int,
                    ms, ns):
    """Y and bound at the listed (m, n) pairs only."""
    X = np.ascontiguousarray(X_bf16_bits, dtype=np.uint16)
    M = X.shape[0]
    ms = np.ascontiguousarray(ms, dtype=np.int64)
    ns = np.ascontiguousarray(ns, dtype=np.int64)
    assert ms.shape == ns.shape
    img = np.ascontiguousarray(img, dtype=np.uint8)
    Y = np.empty(ms.shape, dtype=np.float64)
    B = np.empty(ms.shape, dtype=np.float64)
    if _load().ref_qmatmul_sampled(fmt, _ptr(img), _ptr(X), M, N, K, _ptr(ms), _ptr(ns),
                                   ms.size, _ptr(Y), _ptr(B)):
        raise ValueError("ref_qmatmul_sampled failed")
    return Y, B


def split_image(fmt: int, img: np.ndarray, N: int, K: int):
    """Views of the codes plane and the scales plane (fp16 bits, [N][ldS]) of an image.
    For Q6_0 the codes "plane" is the low-nibble plane followed by the high-bits plane
    (concatenated, without the padding between them)."""
    ldS = (K // 32 + 7) // 8 * 8
    if fmt == Q6_0:
        lo = N * K // 2
        hoff = (lo + 255) // 256 * 256
        off = (hoff + N * K // 4 + 255) // 256 * 256
        codes = np.concatenate([img[:lo], img[hoff:hoff + N * K // 4]])
    else:
        codes_bytes = N * K if fmt == Q8_0 else N * K // 2
        off = (codes_bytes + 255) // 256 * 256
        codes = img[:codes_bytes]
    scales = img[off:off + N * ldS * 2].view(np.uint16).reshape(N, ldS)
    return codes, scales


def q6_codes(img: np.ndarray, N: int, K: int) -> np.ndarray:
    """The 6-bit codes [N][K] of a Q6_0 image, read back from its two planes."""
    lo = N * K // 2
    hoff = (lo + 255) // 256 * 256
    L = img[:lo].reshape(N, K // 32, 16).astype(np.int64)
    H = img[hoff:hoff + N * K // 4].reshape(N, K // 32, 8).astype(np.int64)
    q = np.empty((N, K // 32, 32), dtype=np.int64)
    q[:, :, :16] = L & 15
    q[:, :, 16:] = L >> 4
    for t in range(4):
        q[:, :, 8 * t:8 * t + 8] |= ((H >> (2 * t)) & 3) << 4
    return q.reshape(N, K)


# ---------------------------------------------------------------------- epilogues
# Per-layer output transforms of a layer chain (this build's fused epilogues; the paper
# describes fused execution in Section 3.2, principle 2, without fixing any). Plain fp64
# definitions on top of the fp64 matmul reference Y and its bound B.

EPI_F32, EPI_BF16, EPI_ADD, EPI_GEGLU, EPI_SWIGLU = 0, 1, 2, 3, 4


def gelu_tanh(g):
    """GELU in its tanh form: 0.5 g (1 + tanh(sqrt(2/pi) (g + 0.044715 g^3))), fp64."""
    g = np.asarray(g, dtype=np.float64)
    return 0.5 * g * (1.0 + np.tanh(np.sqrt(2.0 / np.pi) * (g + 0.044715 * g ** 3)))


def silu(g):
    """SiLU: g * sigmoid(g) = g / (1 + exp(-g)), fp64."""
    g = np.asarray(g, dtype=np.float64)
    with np.errstate(over="ignore"):
        return g / (1.0 + np.exp(-g))


def bf16_round(y):
    """fp64 values rounded to bfloat16 (via binary32, nearest even) and back, fp64."""
    b = f32_to_bf16_bits(np.asarray(y, dtype=np.float32))
    return (b.astype(np.uint32) << 16).view(np.float32).astype(np.float64)


def epilogue_reference(kind: int, Y, B, R=None):
    """Reference output and per-element bound of one layer with epilogue `kind`.

    Y, B: the fp64 matmul reference and its bound ([M][N]); R: the fp32 values already
    in the output buffer (EPI_ADD only). Gated kinds take the rows of W interleaved as
    (gate_0, up_0, gate_1, up_1, ...) and give [M][N/2]: act(gate) * up.
    Bounds (the fp32 result acc satisfies |acc - Y| <= B):
      EPI_F32:   B
      EPI_BF16:  B + 2^-8 (|Y| + B)                     one bf16 rounding of acc
      EPI_ADD:   B + 2^-23 (|R| + |Y| + B)              one fp32 rounding of R + acc
      gated:     |act(g)| B_u + (|u| + B_u) (1.2 B_g + 2^-20 (|g| + B_g + 1))
                 + 2^-8 |h| + 1e-6                      act' <= 1.2 for both activations;
                 fp32 evaluation of act within 2^-20 (|g| + 1); one bf16 rounding of h
    """
    Y = np.asarray(Y, dtype=np.float64)
    B = np.asarray(B, dtype=np.float64)
    if kind == EPI_F32:
        return Y, B
    if kind == EPI_BF16:
        return Y, B + 2.0 ** -8 * (np.abs(Y) + B)
    if kind == EPI_ADD:
        R = np.asarray(R, dtype=np.float64)
        return R + Y, B + 2.0 ** -23 * (np.abs(R) + np.abs(Y) + B)
    g, u = Y[:, 0::2], Y[:, 1::2]
    Bg, Bu = B[:, 0::2], B[:, 1::2]
    act = gelu_tanh(g) if kind == EPI_GEGLU else silu(g)
    h = act * u
    bound = (np.abs(act) * Bu + (np.abs(u) + Bu) * (1.2 * Bg + 2.0 ** -20 * (np.abs(g) + Bg + 1.0))
             + 2.0 ** -8 * np.abs(h) + 1e-6)
    return h, bound


# The non-matmul steps of a backbone / action-expert layer (RMSNorm, rotary embedding,
# attention): oracle/layer.py.
from .layer import attention_reference, rmsnorm_reference, rope_reference  # noqa: E402,F401
