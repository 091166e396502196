"""emb_qlayer_seq: fused groups + programmatic dependent launch give the same bits as
separate emb_qmatmul calls, match the oracle, and survive CUDA-graph capture/replay."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
from tests.gpu_util import check_close, to_dev_bf16
from workloads import activation_bits_np, weight_np

pytestmark = pytest.mark.gpu


def _decoder(fmt, M, hidden, kv, ffn, layers, seed):
    """A small decoder chain: groups (q,k,v) (o) (gate,up) (down) sharing X per group."""
    specs, host = [], []
    s = seed
    for _ in range(layers):
        for group in ([(hidden, hidden), (kv, hidden), (kv, hidden)], [(hidden, hidden)],
                      [(ffn, hidden), (ffn, hidden)], [(hidden, ffn)]):
            K = group[0][1]
            Xb = activation_bits_np(M, K, s)
            X = to_dev_bf16(Xb)
            for (N, K_) in group:
                s += 1
                W = weight_np(N, K_, s)
                img = emb.quantize(fmt, torch.from_numpy(W).cuda())
                Y = torch.empty(M, N, dtype=torch.float32, device="cuda")
                specs.append((fmt, img, N, K_, X, Y))
                host.append((W, Xb))
            s += 1
    return specs, host


@pytest.mark.parametrize("fmt", [emb.EMB_Q8_0, emb.EMB_Q4_0])
@pytest.mark.parametrize("M", [1, 4, 50, 136])
def test_seq_equals_single_calls_and_oracle(cuda_device, fmt, M):
    specs, host = _decoder(fmt, M, 512, 128, 1536, 2, 1000 + M)
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    seq_out = [sp[5].clone() for sp in specs]
    for sp in specs:
        sp[5].fill_(float("nan"))
        emb.emb_qmatmul(sp[0], sp[1], sp[4], sp[5], M, sp[2], sp[3])
    torch.cuda.synchronize()
    for i, sp in enumerate(specs):
        assert torch.equal(seq_out[i].view(torch.int32), sp[5].view(torch.int32)), i
    for i in (0, 1, 4, 6, 7):   # q, k, gate, down of layer 0, q of layer 1
        W, Xb = host[i]
        Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, specs[i][2], specs[i][3])
        check_close(seq_out[i].cpu().numpy(), Yref, B, f"layer {i}")


@pytest.mark.parametrize("fmt", [emb.EMB_Q8_0, emb.EMB_Q4_0])
def test_long_rows_group_across_matrices(cuda_device, fmt):
    """Two long-row matrices sharing X at M = 1 form one launch of the ring kernel, whose
    CTAs own runs of rows that cross from the first matrix into the second: bitwise the
    separate calls, within the oracle's bound."""
    K, Ns, M = 16384, (1000, 1030), 1
    Xb = activation_bits_np(M, K, 77)
    X = to_dev_bf16(Xb)
    Ws = [weight_np(N, K, 78 + i) for i, N in enumerate(Ns)]
    imgs = [emb.quantize(fmt, torch.from_numpy(W).cuda()) for W in Ws]
    Ys = [torch.full((M, N), float("nan"), device="cuda") for N in Ns]
    emb.emb_qlayer_seq([(fmt, img, N, K, X, Y) for img, N, Y in zip(imgs, Ns, Ys)], M)
    torch.cuda.synchronize()
    for img, N, Y, W in zip(imgs, Ns, Ys, Ws):
        Y1 = torch.full_like(Y, float("nan"))
        emb.emb_qmatmul(fmt, img, X, Y1, M, N, K)
        torch.cuda.synchronize()
        assert torch.equal(Y.view(torch.int32), Y1.view(torch.int32)), N
        Yref, B = oracle.qmatmul(fmt, oracle.quantize(fmt, W), Xb, N, K)
        check_close(Y.cpu().numpy(), Yref, B, f"fmt={fmt} N={N}")
    assert emb.emb_device_status() == emb.EMB_OK


@pytest.mark.parametrize("M", [1, 50])
def test_seq_graph_replay(cuda_device, M):
    fmt = emb.EMB_Q8_0
    specs, _ = _decoder(fmt, M, 1024, 128, 2048, 2, 7)
    layers = emb.make_layers(specs)
    emb.emb_qlayer_seq(layers, M)
    torch.cuda.synchronize()
    expect = [sp[5].clone() for sp in specs]
    for sp in specs:
        sp[5].zero_()
    s = torch.cuda.Stream()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        emb.emb_qlayer_seq(layers, M)
    for _ in range(3):
        for sp in specs:
            sp[5].fill_(float("nan"))
        g.replay()
        torch.cuda.synchronize()
        for i, sp in enumerate(specs):
            assert torch.equal(expect[i].view(torch.int32), sp[5].view(torch.int32)), i


def test_seq_waw_same_output_buffer(cuda_device):
    """Two consecutive layers writing the same Y: the later one wins (stream order kept
    under programmatic dependent launch)."""
    M, N, K = 1, 2048, 2048
    X1 = to_dev_bf16(activation_bits_np(M, K, 1))
    X2 = to_dev_bf16(activation_bits_np(M, K, 2))
    W1 = emb.quantize(emb.EMB_Q8_0, torch.from_numpy(weight_np(N, K, 3)).cuda())
    W2 = emb.quantize(emb.EMB_Q8_0, torch.from_numpy(weight_np(N, K, 4)).cuda())
    Y = torch.empty(M, N, device="cuda")
    for _ in range(5):
        emb.emb_qlayer_seq([(0, W1, N, K, X1, Y), (0, W2, N, K, X2, Y)], M)
    ref = emb.qmatmul(emb.EMB_Q8_0, W2, X2, N)
    torch.cuda.synchronize()
    assert torch.equal(Y, ref)


def test_timeout_path_reports_status(cuda_device):
    """A bounded wait that nothing completes returns EMB_ETIMEOUT through the status
    word; the context stays usable afterwards."""
    assert emb.emb_device_status() == emb.EMB_OK
    emb.emb_selftest_wait_timeout(2_000_000)   # 2 ms
    assert emb.emb_device_status() == emb.EMB_ETIMEOUT
    assert emb.emb_device_status() == emb.EMB_OK   # cleared
    y = torch.ones(4, device="cuda") * 2
    assert y.sum().item() == 8.0


@pytest.mark.parametrize("fmt,M", [(emb.EMB_Q8_0, 1), (emb.EMB_Q4_0, 1), (emb.EMB_Q8_0, 50),
                                   (emb.EMB_Q4_0, 280)])
def test_recorded_chain_replays(cuda_device, fmt, M):
    """emb_chain_create records the chain's launches once; every replay reads the X
    buffers as they are at launch time and gives the bits of emb_qlayer_seq."""
    specs, _ = _decoder(fmt, M, 512, 128, 1536, 2, 3000 + M)
    rec = emb.RecordedChain(specs, M)
    xs = {sp[4].data_ptr(): sp[4] for sp in specs}
    for it in range(3):
        for j, x in enumerate(xs.values()):   # new activations in the same buffers
            x.copy_(to_dev_bf16(activation_bits_np(M, x.shape[1], 50 * it + j)))
        for sp in specs:
            sp[5].fill_(float("nan"))
        rec.launch()
        torch.cuda.synchronize()
        got = [sp[5].clone() for sp in specs]
        emb.emb_qlayer_seq(specs, M)
        torch.cuda.synchronize()
        for i, sp in enumerate(specs):
            assert torch.equal(got[i].view(torch.int32), sp[5].view(torch.int32)), (it, i)
    assert emb.emb_device_status() == emb.EMB_OK
    rec.close()
    rec.close()   # idempotent
