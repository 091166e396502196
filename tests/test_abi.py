"""The C-ABI library loads, exports every declared entry point, and rejects invalid
arguments before touching the GPU (CPU only: no call here reaches a launch)."""
import ctypes

import numpy as np
import pytest

import oracle
import paper_2607_02501_gb300 as emb


@pytest.fixture(scope="module")
def L():
    emb.build()
    return emb.lib()


def test_every_declared_symbol_is_exported(L):
    names = emb.declared_symbols()
    assert len(names) == 24
    for n in names:
        assert hasattr(L, n), n


def test_every_declaration_cites_its_passage():
    """Every EMB_API declaration of include/emb_qmm.h is preceded by its own comment that
    names the paper passage (a Section or Table) the entry point serves."""
    import re
    with open(emb.HEADER_PATH) as fh:
        text = fh.read()
    body = text[text.index('extern "C" {'):]
    decls = list(re.finditer(r"EMB_API\s+[\w\s\*]*?\b(emb_\w+)\s*\(", body))
    assert len(decls) == len(emb.declared_symbols())
    prev_end = 0
    for d in decls:
        between = body[prev_end:d.start()]
        comments = re.findall(r"/\*.*?\*/", between, flags=re.S)
        assert comments, f"{d.group(1)} has no comment of its own"
        assert re.search(r"\b(Section|Table)\s+\d", comments[-1]), \
            f"{d.group(1)}: its comment names no Section or Table"
        prev_end = body.index(";", d.end()) + 1


def test_no_undeclared_exports(L):
    import subprocess
    out = subprocess.run(["nm", "-D", "--defined-only", emb.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = {line.split()[-1] for line in out.splitlines() if " T " in line}
    assert exported == set(emb.declared_symbols())


@pytest.mark.parametrize("fmt", [emb.EMB_Q8_0, emb.EMB_Q4_0, emb.EMB_Q6_0])
@pytest.mark.parametrize("N,K", [(1, 32), (3, 96), (2048, 2048), (256, 2048), (2048, 16384),
                                 (5, 1152), (4096, 11008), (129, 4608), (7, 4160)])
def test_qweight_bytes_matches_oracle(L, fmt, N, K):
    assert emb.emb_qweight_bytes(fmt, N, K) == oracle.packed_bytes(fmt, N, K)


@pytest.mark.parametrize("fmt,N,K", [(3, 4, 32), (-1, 4, 32), (0, 0, 32), (0, 4, 0), (0, 4, 48), (2, 4, 48),
                                     (1, -5, 64), (0, 4, 31)])
def test_qweight_bytes_invalid(L, fmt, N, K):
    assert emb.emb_qweight_bytes(fmt, N, K) == 0


def test_status_strings(L):
    for s in range(7):
        assert emb.emb_status_string(s).startswith(emb._STATUS_NAMES[s])
    assert "unknown" in emb.emb_status_string(99)


# Fake device addresses: only ever used in calls that must fail validation.
A = 0x7f0000000000            # 256-aligned
B = A + (1 << 30)
C = A + (2 << 30)


@pytest.mark.parametrize("args,expect", [
    ((0, None, B, C, 1, 128, 64), emb.EMB_EINVAL),          # null W
    ((0, A, None, C, 1, 128, 64), emb.EMB_EINVAL),          # null X
    ((0, A, B, None, 1, 128, 64), emb.EMB_EINVAL),          # null Y
    ((3, A, B, C, 1, 128, 64), emb.EMB_EINVAL),             # unknown format
    ((2, A, B, C, 1, 128, 48), emb.EMB_EINVAL),             # Q6_0, K % 32
    ((0, A, B, C, 0, 128, 64), emb.EMB_EINVAL),             # M < 1
    ((0, A, B, C, 1, 0, 64), emb.EMB_EINVAL),               # N < 1
    ((0, A, B, C, 1, 128, 48), emb.EMB_EINVAL),             # K % 32
    ((1, A, B, C, 1, 128, 0), emb.EMB_EINVAL),              # K < 32
    ((0, A + 16, B, C, 1, 128, 64), emb.EMB_EALIGN),        # W not 256-aligned
    ((0, A, B + 2, C, 1, 128, 64), emb.EMB_EALIGN),         # X not 16-aligned
    ((1, A, B, C + 4, 1, 128, 64), emb.EMB_EALIGN),         # Y not 16-aligned
    ((0, A, B, B + 64, 1, 128, 64), emb.EMB_EINVAL),        # Y overlaps X
    ((0, A, B, A + 256, 1, 128, 64), emb.EMB_EINVAL),       # Y overlaps W
])
def test_qmatmul_rejects_before_launch(L, args, expect):
    fmt, W, X, Y, M, N, K = args
    assert L.emb_qmatmul(fmt, W, X, Y, M, N, K, None) == expect


def test_quantize_rejects(L):
    assert L.emb_quantize_q8_0(None, 4, 32, A, None) == emb.EMB_EINVAL
    assert L.emb_quantize_q4_0(B, 4, 48, A, None) == emb.EMB_EINVAL
    assert L.emb_quantize_q8_0(B + 4, 4, 32, A, None) == emb.EMB_EALIGN
    assert L.emb_quantize_q4_0(B, 4, 32, A + 128, None) == emb.EMB_EALIGN
    assert L.emb_quantize_q8_0(A, 4, 32, A + 256, None) == emb.EMB_EINVAL   # in/out overlap
    assert L.emb_quantize_q6_0(None, 4, 32, A, None) == emb.EMB_EINVAL
    assert L.emb_quantize_q6_0(B, 4, 32, A + 16, None) == emb.EMB_EALIGN
    assert L.emb_quantize_q6_0(A, 4, 64, A + 512, None) == emb.EMB_EINVAL   # in/out overlap


def test_dequantize_rejects(L):
    assert L.emb_dequantize_f32(3, A, 4, 32, B, None) == emb.EMB_EINVAL
    assert L.emb_dequantize_bf16(0, A, 4, 33, B, None) == emb.EMB_EINVAL
    assert L.emb_dequantize_f32(0, A + 1, 4, 32, B, None) == emb.EMB_EALIGN
    assert L.emb_dequantize_bf16(1, A, 4, 32, None, None) == emb.EMB_EINVAL


def test_selftest_rejects_out_of_range_timeouts(L):
    assert L.emb_selftest_wait_timeout(10, None) == emb.EMB_EINVAL
    assert L.emb_selftest_wait_timeout(10 ** 10, None) == emb.EMB_EINVAL


def _layers(specs):
    return emb.make_layers(specs)


def test_seq_rejects(L):
    M = 1
    good = (0, A, 128, 64, B, C)
    arr = _layers([good])
    assert L.emb_qlayer_seq(None, 1, M, None, 0, None) == emb.EMB_EINVAL
    assert L.emb_qlayer_seq(arr, 0, M, None, 0, None) == emb.EMB_EINVAL
    assert L.emb_qlayer_seq(arr, emb.EMB_MAX_LAYERS + 1, M, None, 0, None) == emb.EMB_EINVAL
    assert L.emb_qlayer_seq(arr, 1, 0, None, 0, None) == emb.EMB_EINVAL
    bad = _layers([good])
    bad[0].epilogue = 5                                    # unknown epilogue
    assert L.emb_qlayer_seq(bad, 1, M, None, 0, None) == emb.EMB_EINVAL
    bad[0].epilogue = -1
    assert L.emb_qlayer_seq(bad, 1, M, None, 0, None) == emb.EMB_EINVAL
    odd = _layers([(0, A, 127, 64, B, C, emb.EMB_EPI_GEGLU)])   # gated needs even N
    assert L.emb_qlayer_seq(odd, 1, M, None, 0, None) == emb.EMB_EINVAL
    # layer 1's weights overlap layer 0's output
    chain = _layers([good, (0, C, 128, 64, B, C + (1 << 20))])
    assert L.emb_qlayer_seq(chain, 2, M, None, 0, None) == emb.EMB_EINVAL
    # misaligned member
    chain = _layers([good, (1, A + (64 << 20), 128, 64, B + 8, C + (1 << 20))])
    assert L.emb_qlayer_seq(chain, 2, M, None, 0, None) == emb.EMB_EALIGN
    assert L.emb_qlayer_seq_workspace(chain, 2, M) == ctypes.c_size_t(-1).value


def test_seq_epilogue_overlap_rules(L):
    """A layer may read (as X) an earlier layer's output; weights may not be written;
    Y's extent follows the epilogue (bf16: 2 bytes per element, gated: N/2 columns)."""
    M = 1
    # layer 1 reads layer 0's bf16 output as its X: accepted (no launch on the CPU: the
    # checks pass and the call then needs a GPU, so use the workspace query to validate)
    chain = _layers([(0, A, 128, 64, B, C, emb.EMB_EPI_BF16),
                     (0, A + (64 << 20), 128, 128, C, C + (1 << 20))])
    assert emb.emb_qlayer_seq_workspace(chain, M) == 0
    # layer 1's weights overlap layer 0's output: rejected
    chain = _layers([(0, A, 128, 64, B, C, emb.EMB_EPI_BF16), (0, C, 128, 64, B, C + (1 << 20))])
    assert L.emb_qlayer_seq_workspace(chain, 2, M) == ctypes.c_size_t(-1).value
    # a gated layer writes M x N/2 bf16: 64 x 2 = 128 bytes, so X right behind is fine
    ok = _layers([(0, A, 128, 64, C + 128, C, emb.EMB_EPI_GEGLU)])
    assert emb.emb_qlayer_seq_workspace(ok, M) == 0
    bad = _layers([(0, A, 128, 64, C + 64, C, emb.EMB_EPI_GEGLU)])   # X inside Y
    assert L.emb_qlayer_seq_workspace(bad, 1, M) == ctypes.c_size_t(-1).value


def test_seq_workspace_without_a_device(L):
    """Decode chains never want a workspace; without a GPU no schedule is planned, so a
    prefill chain's answer is 0 too (the call itself would fail)."""
    chain = _layers([(0, A, 128, 64, B, C), (1, A + (64 << 20), 256, 64, B, C + (1 << 20))])
    assert emb.emb_qlayer_seq_workspace(chain, 1) == 0
    assert emb.emb_qlayer_seq_workspace(chain, 816) == 0


def test_seq_rejects_misaligned_workspace(L):
    """A workspace must be 256-byte aligned; checked before anything is enqueued."""
    chain = _layers([(0, A, 128, 64, B, C)])
    assert L.emb_qlayer_seq(chain, 1, 1, ctypes.c_void_p(B + (8 << 20) + 16), 1 << 20, None) == emb.EMB_EALIGN
    h = ctypes.c_void_p()
    assert L.emb_chain_create(chain, 1, 1, ctypes.c_void_p(B + (8 << 20) + 16), 1 << 20,
                              ctypes.byref(h)) == emb.EMB_EALIGN
    assert h.value is None


def test_precise_operand_flag(L):
    """EMB_PRECISE_OPERAND may be OR-ed into any epilogue; other flag bits are rejected."""
    for kind in range(5):
        ok = _layers([(0, A, 128, 64, B, C, kind | emb.EMB_PRECISE_OPERAND)])
        assert emb.emb_qlayer_seq_workspace(ok, 64) == 0
    bad = _layers([(0, A, 128, 64, B, C, 0x200)])
    assert L.emb_qlayer_seq_workspace(bad, 1, 64) == ctypes.c_size_t(-1).value
    bad = _layers([(0, A, 128, 64, B, C, 5 | emb.EMB_PRECISE_OPERAND)])
    assert L.emb_qlayer_seq_workspace(bad, 1, 64) == ctypes.c_size_t(-1).value


def test_chain_create_rejects(L):
    """Recorded chains validate exactly like emb_qlayer_seq, before touching the GPU."""
    M = 1
    good = (0, A, 128, 64, B, C)
    h = ctypes.c_void_p(123)
    arr = _layers([good])
    assert L.emb_chain_create(arr, 1, M, None, 0, None) == emb.EMB_EINVAL
    assert L.emb_chain_create(None, 1, M, None, 0, ctypes.byref(h)) == emb.EMB_EINVAL
    assert h.value is None   # cleared on failure
    assert L.emb_chain_create(arr, 0, M, None, 0, ctypes.byref(h)) == emb.EMB_EINVAL
    chain = _layers([good, (0, C, 128, 64, B, C + (1 << 20))])   # weights are layer 0's Y
    assert L.emb_chain_create(chain, 2, M, None, 0, ctypes.byref(h)) == emb.EMB_EINVAL
    odd = _layers([(0, A, 127, 64, B, C, emb.EMB_EPI_SWIGLU)])      # gated with odd N
    assert L.emb_chain_create(odd, 1, M, None, 0, ctypes.byref(h)) == emb.EMB_EINVAL
    chain = _layers([good, (1, A + (64 << 20), 128, 64, B + 8, C + (1 << 20))])   # misaligned X
    assert L.emb_chain_create(chain, 2, M, None, 0, ctypes.byref(h)) == emb.EMB_EALIGN
    assert L.emb_chain_launch(None, None) == emb.EMB_EINVAL
    assert L.emb_chain_destroy(None) == emb.EMB_OK


def test_library_has_no_torch_dependency():
    import subprocess
    out = subprocess.run(["ldd", emb.LIB_PATH], capture_output=True, text=True).stdout
    assert "torch" not in out and "libcudart" not in out


D_ = C + (1 << 30)
E_ = C + (2 << 30)


def test_recording_rejects_null_stream_and_handle(L):
    h = ctypes.c_void_p()
    assert L.emb_chain_record_begin(None) == emb.EMB_EINVAL
    assert L.emb_chain_record_end(None, ctypes.byref(h)) == emb.EMB_EINVAL
    assert L.emb_chain_record_end(A, None) == emb.EMB_EINVAL


@pytest.mark.parametrize("args,expect", [
    ((None, B, C, 4, 1024, 1e-6), emb.EMB_EINVAL),        # null x
    ((A, B, C, 0, 1024, 1e-6), emb.EMB_EINVAL),           # M = 0
    ((A, B, C, 4, 1028, 1e-6), emb.EMB_EINVAL),           # D % 8 != 0
    ((A, B, C, 4, 1024, -1.0), emb.EMB_EINVAL),           # eps < 0
    ((A, B, C, 4, 1024, float("nan")), emb.EMB_EINVAL),   # eps NaN
    ((A + 4, B, C, 4, 1024, 1e-6), emb.EMB_EALIGN),       # x misaligned
    ((A, B, C + 2, 4, 1024, 1e-6), emb.EMB_EALIGN),       # y misaligned
    ((A, B, A + 4096, 4, 1024, 1e-6), emb.EMB_EINVAL),    # y inside x
    ((A, B, B, 4, 1024, 1e-6), emb.EMB_EINVAL),           # y over gamma
])
def test_rmsnorm_validation(L, args, expect):
    assert L.emb_rmsnorm(*args, None) == expect


@pytest.mark.parametrize("args,expect", [
    ((None, 50, 8, 128, 816, 1e4), emb.EMB_EINVAL),       # null x
    ((A, 50, 8, 127, 816, 1e4), emb.EMB_EINVAL),          # odd head_dim
    ((A, 50, 0, 128, 816, 1e4), emb.EMB_EINVAL),          # no heads
    ((A, 50, 8, 128, -1, 1e4), emb.EMB_EINVAL),           # negative position
    ((A, 50, 8, 128, 816, 0.0), emb.EMB_EINVAL),          # base <= 0
    ((A, 50, 8, 1024, 816, 1e4), emb.EMB_EINVAL),         # head_dim > 512
    ((A, 50, 8, 128, (1 << 24) - 10, 1e4), emb.EMB_EINVAL),  # positions past 2^24
    ((A + 2, 50, 8, 128, 816, 1e4), emb.EMB_EALIGN),      # misaligned
])
def test_rope_validation(L, args, expect):
    assert L.emb_rope(*args, None) == expect


# Q, K0, V0, n0, K1, V1, n1, O, M, H, Hk, d, scale
@pytest.mark.parametrize("args,expect", [
    ((A, B, C, 816, D_, E_, 50, A + (3 << 20), 50, 8, 1, 96, 0.1), emb.EMB_EUNSUPPORTED),  # head_dim 96
    ((A, B, C, 816, D_, E_, 50, A + (3 << 20), 50, 8, 3, 128, 0.1), emb.EMB_EINVAL),       # 8 % 3
    ((A, B, C, 0, D_, E_, 0, A + (3 << 20), 50, 8, 1, 128, 0.1), emb.EMB_EINVAL),          # no keys
    ((A, None, C, 816, D_, E_, 50, A + (3 << 20), 50, 8, 1, 128, 0.1), emb.EMB_EINVAL),    # K0 missing
    ((A, B, C, 816, None, E_, 50, A + (3 << 20), 50, 8, 1, 128, 0.1), emb.EMB_EINVAL),     # K1 missing
    ((A, B, C, 816, D_, E_, 50, A + 1024, 50, 8, 1, 128, 0.1), emb.EMB_EINVAL),            # O inside Q
    ((A, B, C, 816, D_, E_, 50, B + 4096, 50, 8, 1, 128, 0.1), emb.EMB_EINVAL),            # O inside K0
    ((A, B, C, 816, D_, E_, 50, A + (3 << 20), 50, 8, 1, 128, float("inf")), emb.EMB_EINVAL),
    ((A, B + 8, C, 816, D_, E_, 50, A + (3 << 20), 50, 8, 1, 128, 0.1), emb.EMB_EALIGN),   # K0 misaligned
])
def test_attention_validation(L, args, expect):
    assert L.emb_attention(*args, None) == expect



def test_rope_qk_validation(L):
    assert L.emb_rope_qk(A, 8, None, 1, 50, 128, 816, 1e4, None) == emb.EMB_EINVAL      # k missing
    assert L.emb_rope_qk(A, 8, A + 4096, 1, 50, 128, 816, 1e4, None) == emb.EMB_EINVAL  # k inside q
    assert L.emb_rope_qk(A, 8, B + 2, 1, 50, 128, 816, 1e4, None) == emb.EMB_EALIGN     # k misaligned
    assert L.emb_rope_qk(A, 8, B, -1, 50, 128, 816, 1e4, None) == emb.EMB_EINVAL        # negative heads
