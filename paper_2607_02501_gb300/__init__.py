"""Python binding of libembqmm.so (the C ABI declared in include/emb_qmm.h).

Argument marshalling only: every step of the computation runs in the library's
CUDA kernels. Functions keep the C names and take either torch tensors (their
data_ptr() is passed) or raw device addresses; `stream` defaults to torch's
current CUDA stream. A non-OK status raises EmbError. There is no fallback: if
the library is not built, importing works but every call raises.

Paper: arXiv 2607.02501 (Embodied.cpp) -- the block-quantised linear layers of
the 8-bit / 4-bit configurations (Section 4, Table 3) executed latency-first at
batch 1 (Section 3.1 challenge 2; Section 3.2 design principle 2).
"""
from __future__ import annotations

import ctypes
import os
import re
from typing import Iterable, Optional, Sequence

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libembqmm.so")
HEADER_PATH = os.path.join(_HERE, "..", "include", "emb_qmm.h")

EMB_Q8_0 = 0
EMB_Q4_0 = 1
EMB_Q6_0 = 2

EMB_OK = 0
EMB_EINVAL = 1
EMB_EALIGN = 2
EMB_ENOSPC = 3
EMB_ECUDA = 4
EMB_ETIMEOUT = 5
EMB_EUNSUPPORTED = 6
EMB_MAX_LAYERS = 4096
EMB_PRECISE_OPERAND = 0x100   # flag OR-ed into a layer's epilogue (two-operand tensor-core weights)

# layer epilogues (emb_epilogue)
EMB_EPI_F32 = 0
EMB_EPI_BF16 = 1
EMB_EPI_ADD = 2
EMB_EPI_GEGLU = 3
EMB_EPI_SWIGLU = 4

_STATUS_NAMES = {0: "EMB_OK", 1: "EMB_EINVAL", 2: "EMB_EALIGN", 3: "EMB_ENOSPC",
                 4: "EMB_ECUDA", 5: "EMB_ETIMEOUT", 6: "EMB_EUNSUPPORTED"}


class EmbError(RuntimeError):
    def __init__(self, status: int, where: str):
        self.status = status
        super().__init__(f"{where}: {_STATUS_NAMES.get(status, status)}")


class emb_qlayer(ctypes.Structure):
    _fields_ = [("fmt", ctypes.c_int32), ("epilogue", ctypes.c_int32),
                ("W_blocks", ctypes.c_void_p), ("N", ctypes.c_int64), ("K", ctypes.c_int64),
                ("X", ctypes.c_void_p), ("Y", ctypes.c_void_p)]


_lib = None


def build(force: bool = False) -> str:
    from . import buildlib as _b
    return _b.build(force=force)


def lib():
    """The loaded shared library; raises if it has not been built."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: run paper_2607_02501_gb300.build() "
                           "(nvcc, sm_103a) first; there is no non-CUDA implementation")
    L = ctypes.CDLL(LIB_PATH)
    i64, i32, vp, sz = ctypes.c_int64, ctypes.c_int, ctypes.c_void_p, ctypes.c_size_t
    L.emb_qweight_bytes.argtypes = [i32, i64, i64]
    L.emb_qweight_bytes.restype = sz
    for name in ("emb_quantize_q8_0", "emb_quantize_q4_0", "emb_quantize_q6_0"):
        getattr(L, name).argtypes = [vp, i64, i64, vp, vp]
        getattr(L, name).restype = i32
    L.emb_qmatmul.argtypes = [i32, vp, vp, vp, i64, i64, i64, vp]
    L.emb_qmatmul.restype = i32
    L.emb_qlayer_seq_workspace.argtypes = [ctypes.POINTER(emb_qlayer), i32, i64]
    L.emb_qlayer_seq_workspace.restype = sz
    L.emb_qlayer_seq.argtypes = [ctypes.POINTER(emb_qlayer), i32, i64, vp, sz, vp]
    L.emb_qlayer_seq.restype = i32
    L.emb_chain_create.argtypes = [ctypes.POINTER(emb_qlayer), i32, i64, vp, sz, ctypes.POINTER(vp)]
    L.emb_chain_create.restype = i32
    L.emb_chain_launch.argtypes = [vp, vp]
    L.emb_chain_launch.restype = i32
    L.emb_chain_destroy.argtypes = [vp]
    L.emb_chain_destroy.restype = i32
    for name in ("emb_dequantize_f32", "emb_dequantize_bf16"):
        getattr(L, name).argtypes = [i32, vp, i64, i64, vp, vp]
        getattr(L, name).restype = i32
    L.emb_device_status.argtypes = [vp]
    L.emb_device_status.restype = i32
    L.emb_selftest_wait_timeout.argtypes = [i64, vp]
    L.emb_selftest_wait_timeout.restype = i32
    L.emb_status_string.argtypes = [i32]
    L.emb_status_string.restype = ctypes.c_char_p
    L.emb_build_info.argtypes = []
    L.emb_build_info.restype = ctypes.c_char_p
    L.emb_qlayer_seq_chained.argtypes = [ctypes.POINTER(emb_qlayer), i32, i64, vp]
    L.emb_qlayer_seq_chained.restype = i32
    L.emb_qlayer_seq_noalloc.argtypes = [ctypes.POINTER(emb_qlayer), i32, i64, vp]
    L.emb_qlayer_seq_noalloc.restype = i32
    L.emb_chain_record_begin.argtypes = [vp]
    L.emb_chain_record_begin.restype = i32
    L.emb_chain_record_end.argtypes = [vp, ctypes.POINTER(vp)]
    L.emb_chain_record_end.restype = i32
    f32 = ctypes.c_float
    L.emb_rmsnorm.argtypes = [vp, vp, vp, i64, i64, f32, vp]
    L.emb_rmsnorm.restype = i32
    L.emb_rope.argtypes = [vp, i64, i64, i64, i64, f32, vp]
    L.emb_rope.restype = i32
    L.emb_rope_qk.argtypes = [vp, i64, vp, i64, i64, i64, i64, f32, vp]
    L.emb_rope_qk.restype = i32
    L.emb_attention.argtypes = [vp, vp, vp, i64, vp, vp, i64, vp, i64, i64, i64, i64, f32, vp]
    L.emb_attention.restype = i32
    _lib = L
    return L


def declared_symbols() -> list:
    """Names of every entry point declared in include/emb_qmm.h."""
    with open(HEADER_PATH) as fh:
        text = fh.read()
    return re.findall(r"EMB_API\s+[\w\s\*]*?\b(emb_\w+)\s*\(", text)


# ------------------------------------------------------------------ marshalling

def _ptr(x) -> Optional[int]:
    if x is None:
        return None
    if isinstance(x, int):
        return x
    return int(x.data_ptr())


def _stream(stream) -> Optional[int]:
    if stream is None:
        import torch
        return int(torch.cuda.current_stream().cuda_stream)
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


def _check(status: int, where: str) -> None:
    if status != EMB_OK:
        raise EmbError(status, where)


# ------------------------------------------------------------------ entry points

def emb_qweight_bytes(fmt: int, N: int, K: int) -> int:
    return int(lib().emb_qweight_bytes(fmt, N, K))


def emb_quantize_q8_0(W, N: int, K: int, W_blocks, stream=None) -> None:
    _check(lib().emb_quantize_q8_0(_ptr(W), N, K, _ptr(W_blocks), _stream(stream)),
           "emb_quantize_q8_0")


def emb_quantize_q4_0(W, N: int, K: int, W_blocks, stream=None) -> None:
    _check(lib().emb_quantize_q4_0(_ptr(W), N, K, _ptr(W_blocks), _stream(stream)),
           "emb_quantize_q4_0")


def emb_quantize_q6_0(W, N: int, K: int, W_blocks, stream=None) -> None:
    _check(lib().emb_quantize_q6_0(_ptr(W), N, K, _ptr(W_blocks), _stream(stream)),
           "emb_quantize_q6_0")


def emb_qmatmul(fmt: int, W_blocks, X, Y, M: int, N: int, K: int, stream=None) -> None:
    _check(lib().emb_qmatmul(fmt, _ptr(W_blocks), _ptr(X), _ptr(Y), M, N, K, _stream(stream)),
           "emb_qmatmul")


def make_layers(specs: Sequence) -> ctypes.Array:
    """specs: iterable of (fmt, W_blocks, N, K, X, Y[, epilogue]) -> a C array of emb_qlayer."""
    arr = (emb_qlayer * len(specs))()
    for i, sp in enumerate(specs):
        fmt, W, N, K, X, Y = sp[:6]
        epi = sp[6] if len(sp) > 6 else EMB_EPI_F32
        arr[i] = emb_qlayer(fmt, epi, _ptr(W), N, K, _ptr(X), _ptr(Y))
    return arr


def emb_qlayer_seq_workspace(layers, M: int) -> int:
    arr = layers if isinstance(layers, ctypes.Array) else make_layers(layers)
    n = int(lib().emb_qlayer_seq_workspace(arr, len(arr), M))
    if n == ctypes.c_size_t(-1).value:
        raise EmbError(EMB_EINVAL, "emb_qlayer_seq_workspace")
    return n


def chain_workspace(layers, M: int, device=None):
    """A zero-filled device buffer of emb_qlayer_seq_workspace(layers, M) bytes on the
    current (or given) CUDA device, or None when the chain needs none."""
    import torch
    n = emb_qlayer_seq_workspace(layers, M)
    if n == 0:
        return None
    return torch.zeros(n, dtype=torch.uint8, device=device if device is not None else "cuda")


def emb_qlayer_seq(layers, M: int, workspace=None, ws_bytes: int = 0, stream=None) -> None:
    arr = layers if isinstance(layers, ctypes.Array) else make_layers(layers)
    _check(lib().emb_qlayer_seq(arr, len(arr), M, _ptr(workspace), ws_bytes, _stream(stream)),
           "emb_qlayer_seq")


def emb_qlayer_seq_chained(layers, M: int, stream=None) -> None:
    """emb_qlayer_seq whose first launch also overlaps the previous launch on the stream
    (the call's weights must not be written by that launch)."""
    arr = layers if isinstance(layers, ctypes.Array) else make_layers(layers)
    _check(lib().emb_qlayer_seq_chained(arr, len(arr), M, _stream(stream)), "emb_qlayer_seq_chained")


def emb_qlayer_seq_noalloc(layers, M: int, stream=None) -> None:
    """emb_qlayer_seq with the library's own static device workspace (one per device;
    calls on different streams of a device must not overlap)."""
    arr = layers if isinstance(layers, ctypes.Array) else make_layers(layers)
    _check(lib().emb_qlayer_seq_noalloc(arr, len(arr), M, _stream(stream)), "emb_qlayer_seq_noalloc")


def emb_chain_create(layers, M: int, workspace=None, ws_bytes: int = 0) -> int:
    """Record a chain; returns the handle (an address). See RecordedChain for a wrapper
    that also keeps the layers' tensors alive."""
    arr = layers if isinstance(layers, ctypes.Array) else make_layers(layers)
    h = ctypes.c_void_p()
    _check(lib().emb_chain_create(arr, len(arr), M, _ptr(workspace), ws_bytes, ctypes.byref(h)),
           "emb_chain_create")
    return int(h.value)


def emb_chain_launch(chain: int, stream=None) -> None:
    _check(lib().emb_chain_launch(chain, _stream(stream)), "emb_chain_launch")


def emb_chain_destroy(chain: int) -> None:
    _check(lib().emb_chain_destroy(chain), "emb_chain_destroy")


class RecordedChain:
    """emb_qlayer_seq recorded once (emb_chain_create) and replayed with one call per
    step. Holds the specs so that every buffer the recording points at stays alive."""

    def __init__(self, specs, M: int, workspace: bool = True):
        self.specs = list(specs)
        self.layers = make_layers(self.specs)
        self.M = M
        # the workspace the chain's fastest schedule wants (zero-filled; None if none)
        self.workspace = chain_workspace(self.layers, M) if workspace else None
        ws = self.workspace
        self.handle = emb_chain_create(self.layers, M, ws, 0 if ws is None else ws.numel())

    def launch(self, stream=None) -> None:
        emb_chain_launch(self.handle, stream)

    def close(self) -> None:
        if self.handle:
            emb_chain_destroy(self.handle)
            self.handle = 0

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def emb_chain_record_begin(stream) -> None:
    _check(lib().emb_chain_record_begin(_stream(stream)), "emb_chain_record_begin")


def emb_chain_record_end(stream) -> int:
    h = ctypes.c_void_p()
    _check(lib().emb_chain_record_end(_stream(stream), ctypes.byref(h)), "emb_chain_record_end")
    return int(h.value)


class Recording:
    """Record library calls made on `stream` (a torch.cuda.Stream) inside the with-block
    into one chain; `launch()` replays it, `close()` frees it. `keep` holds the buffers the
    recording points at."""

    def __init__(self, stream, keep=()):
        self.stream = stream
        self.keep = list(keep)
        self.handle = 0

    def __enter__(self):
        emb_chain_record_begin(self.stream)
        return self

    def __exit__(self, exc_type, exc, tb):
        h = emb_chain_record_end(self.stream)
        if exc_type is None:
            self.handle = h
        elif h:
            emb_chain_destroy(h)
        return False

    def launch(self, stream=None) -> None:
        emb_chain_launch(self.handle, stream)

    def close(self) -> None:
        if self.handle:
            emb_chain_destroy(self.handle)
            self.handle = 0

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def emb_rmsnorm(x, gamma, y, eps: float = 1e-6, stream=None) -> None:
    """x: fp32 [M][D]; gamma: fp32 [D]; y: bf16 [M][D] (all device tensors)."""
    M, D = x.shape
    _check(lib().emb_rmsnorm(_ptr(x), _ptr(gamma), _ptr(y), M, D, eps, _stream(stream)), "emb_rmsnorm")


def emb_rope(x, n_heads: int, head_dim: int, pos0: int, base: float = 10000.0, stream=None) -> None:
    """In place on bf16 x [M][n_heads * head_dim]; token m at position pos0 + m."""
    _check(lib().emb_rope(_ptr(x), x.shape[0], n_heads, head_dim, pos0, base, _stream(stream)),
           "emb_rope")


def emb_rope_qk(q, n_q_heads: int, k, n_k_heads: int, head_dim: int, pos0: int,
                base: float = 10000.0, stream=None) -> None:
    """emb_rope of q and k (same positions) in one launch."""
    _check(lib().emb_rope_qk(_ptr(q), n_q_heads, _ptr(k), n_k_heads, q.shape[0], head_dim, pos0, base,
                             _stream(stream)), "emb_rope_qk")


def emb_attention(Q, K0, V0, K1, V1, O, n_heads: int, n_kv_heads: int, head_dim: int,
                  scale: float, stream=None) -> None:
    """Q, O: bf16 [M][n_heads * head_dim]; K0/V0 (prefix) and K1/V1 (chunk): bf16
    [n][n_kv_heads * head_dim] or None."""
    n0 = 0 if K0 is None else K0.shape[0]
    n1 = 0 if K1 is None else K1.shape[0]
    _check(lib().emb_attention(_ptr(Q), _ptr(K0), _ptr(V0), n0, _ptr(K1), _ptr(V1), n1, _ptr(O),
                               Q.shape[0], n_heads, n_kv_heads, head_dim, scale, _stream(stream)),
           "emb_attention")


def emb_dequantize_f32(fmt: int, W_blocks, N: int, K: int, out, stream=None) -> None:
    _check(lib().emb_dequantize_f32(fmt, _ptr(W_blocks), N, K, _ptr(out), _stream(stream)),
           "emb_dequantize_f32")


def emb_dequantize_bf16(fmt: int, W_blocks, N: int, K: int, out, stream=None) -> None:
    _check(lib().emb_dequantize_bf16(fmt, _ptr(W_blocks), N, K, _ptr(out), _stream(stream)),
           "emb_dequantize_bf16")


def emb_device_status(stream=None) -> int:
    """Synchronise the stream; return (and clear) the device status code."""
    return int(lib().emb_device_status(_stream(stream)))


def emb_selftest_wait_timeout(timeout_ns: int, stream=None) -> None:
    _check(lib().emb_selftest_wait_timeout(timeout_ns, _stream(stream)),
           "emb_selftest_wait_timeout")


def emb_status_string(status: int) -> str:
    return lib().emb_status_string(status).decode()


def emb_build_info() -> str:
    return lib().emb_build_info().decode()


# ------------------------------------------------------------------ tensor helpers

def empty_qweight(fmt: int, N: int, K: int, device="cuda"):
    """A device byte tensor sized for one packed image (torch allocations are 512-B aligned)."""
    import torch
    n = emb_qweight_bytes(fmt, N, K)
    if n == 0:
        raise EmbError(EMB_EINVAL, "emb_qweight_bytes")
    return torch.empty(n, dtype=torch.uint8, device=device)


def quantize(fmt: int, W, stream=None):
    """Pack fp32 device W [N][K]; returns the packed image as a uint8 device tensor."""
    N, K = W.shape
    out = empty_qweight(fmt, N, K, device=W.device)
    {EMB_Q8_0: emb_quantize_q8_0, EMB_Q4_0: emb_quantize_q4_0,
     EMB_Q6_0: emb_quantize_q6_0}[fmt](W, N, K, out, stream)
    return out


def qmatmul(fmt: int, W_blocks, X, N: int, stream=None, out=None):
    """Y = X @ w'^T for bf16 device X [M][K]; returns fp32 [M][N]."""
    import torch
    M, K = X.shape
    Y = torch.empty(M, N, dtype=torch.float32, device=X.device) if out is None else out
    emb_qmatmul(fmt, W_blocks, X, Y, M, N, K, stream)
    return Y
