"""emb_qlayer_seq_noalloc: a chain run with the library's own static device workspace
(no caller allocation). Its results must be bitwise those of emb_qlayer_seq with a caller
workspace (the same schedules), meet the oracle's bound, stay the same from call to call
(the flags are handed back, and re-zeroed by every call), and replay inside a recorded
chain. Collected last: it leaves the library's static array in use on the device."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
from tests.gpu_util import check_close, to_dev_bf16
from workloads import activation_bits_np, weight_np

pytestmark = pytest.mark.gpu
Q8, Q4 = emb.EMB_Q8_0, emb.EMB_Q4_0


def _layer(fmt, M, N, K, seed, kind=emb.EMB_EPI_F32):
    W = weight_np(N, K, seed)
    Xb = activation_bits_np(M, K, seed + 1)
    img = emb.quantize(fmt, torch.from_numpy(W).cuda())
    return W, Xb, img, to_dev_bf16(Xb)


@pytest.mark.parametrize("fmt,M,N,K", [(Q4, 280, 5000, 4096), (Q8, 256, 20000, 2048)])
def test_noalloc_matches_a_caller_workspace(cuda_device, fmt, M, N, K):
    W, Xb, img, X = _layer(fmt, M, N, K, 21)
    Y1 = torch.full((M, N), float("nan"), device="cuda")
    layers = [(fmt, img, N, K, X, Y1)]
    ws = emb.chain_workspace(layers, M)
    assert ws is not None, "this shape should take the stream-K schedule"
    emb.emb_qlayer_seq(layers, M, ws, ws.numel())
    Y2 = torch.full_like(Y1, float("nan"))
    emb.emb_qlayer_seq_noalloc([(fmt, img, N, K, X, Y2)], M)
    Y3 = torch.full_like(Y1, float("nan"))
    emb.emb_qlayer_seq_noalloc([(fmt, img, N, K, X, Y3)], M)
    torch.cuda.synchronize()
    assert emb.emb_device_status() == emb.EMB_OK
    assert torch.equal(Y1.view(torch.int32), Y2.view(torch.int32))
    assert torch.equal(Y2.view(torch.int32), Y3.view(torch.int32))
    Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
    check_close(Y2.cpu().numpy(), Yref, B, f"noalloc fmt={fmt} M={M} N={N} K={K}")


def test_noalloc_decode_and_recorded_chain(cuda_device):
    """A decode chain (no workspace wanted) gives emb_qlayer_seq's bits; a prefill call
    recorded into a chain replays with the same bits as the eager call."""
    W, Xb, img, X = _layer(Q8, 1, 4096, 2048, 5)
    Ya = torch.empty(1, 4096, device="cuda")
    Yb = torch.empty(1, 4096, device="cuda")
    emb.emb_qlayer_seq([(Q8, img, 4096, 2048, X, Ya)], 1)
    emb.emb_qlayer_seq_noalloc([(Q8, img, 4096, 2048, X, Yb)], 1)
    torch.cuda.synchronize()
    assert torch.equal(Ya.view(torch.int32), Yb.view(torch.int32))

    fmt, M, N, K = Q4, 280, 5000, 4096
    W, Xb, img, X = _layer(fmt, M, N, K, 8)
    Ye = torch.full((M, N), float("nan"), device="cuda")
    emb.emb_qlayer_seq_noalloc([(fmt, img, N, K, X, Ye)], M)
    Yr = torch.full_like(Ye, float("nan"))
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        emb.emb_chain_record_begin(s)
        emb.emb_qlayer_seq_noalloc([(fmt, img, N, K, X, Yr)], M, stream=s)
        chain = emb.emb_chain_record_end(s)
        emb.emb_chain_launch(chain, s)
        emb.emb_chain_launch(chain, s)
    torch.cuda.synchronize()
    emb.emb_chain_destroy(chain)
    assert emb.emb_device_status() == emb.EMB_OK
    assert torch.equal(Ye.view(torch.int32), Yr.view(torch.int32))
