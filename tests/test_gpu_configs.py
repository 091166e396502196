"""Parity at the full sizes of every workload (one closed-loop step of the paper's
batch-1 setting: decode M=1, action chunk M=50, prefill M=280/768/816), run through
emb_qlayer_seq exactly as the bench launches it (with the workspace its recorded chains
get, so prefill layers take the stream-K schedule where it pays). Every linear is checked on sampled
output rows (the oracle quantises those rows of W itself and computes them one by
one); layer 0 of each distinct shape is also compared in full."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
import workloads as wl
from tests.gpu_util import bits_of, check_close, layout_rows, sample_rows

pytestmark = pytest.mark.gpu


def _run_workload(w: wl.Workload, rows_per_linear=12, full_first=True, layers=None,
                  token_sample=None):
    dev = "cuda"
    groups = w.groups if layers is None else w.groups[:4 * layers]
    specs, checks = [], []
    seen_shapes = set()
    for gi, group in enumerate(groups):
        K = group[0].K
        X = wl.activation_torch(w.M, K, wl.activation_seed(group[0]), device=dev)
        Xb = bits_of(X)
        for lin in group:
            W = wl.weight_torch(lin, device=dev)
            img = emb.quantize(w.fmt, W)
            Y = torch.empty(w.M, lin.N, dtype=torch.float32, device=dev)
            full = full_first and (lin.N, lin.K) not in seen_shapes
            seen_shapes.add((lin.N, lin.K))
            rows = np.arange(lin.N) if full else sample_rows(lin.N, rows_per_linear, lin.seed)
            Wrows = W[torch.as_tensor(rows, device=dev)].cpu().numpy()
            checks.append((lin, rows, Wrows, Xb, img, Y, full))
            specs.append((w.fmt, img, lin.N, lin.K, X, Y))
            del W
    # with the workspace the bench's recorded chains take (stream-K prefill launches)
    ws = emb.chain_workspace(specs, w.M)
    emb.emb_qlayer_seq(specs, w.M, ws, 0 if ws is None else ws.numel())
    assert emb.emb_device_status() == emb.EMB_OK
    if ws is not None:
        assert int(ws[:4096].count_nonzero()) == 0, "stream-K flags left set"
    worst = 0.0
    toks = np.arange(w.M) if token_sample is None else token_sample
    for lin, rows, Wrows, Xb, img, Y, full in checks:
        ref_img = oracle.quantize(w.fmt, Wrows)
        got_img = img.cpu().numpy() if full else layout_rows(w.fmt, img, lin.N, lin.K, rows)
        assert np.array_equal(got_img, ref_img), f"{lin.name}: packed bytes differ"
        Yref, B = oracle.qmatmul(w.fmt, ref_img, Xb[toks], len(rows), lin.K)
        Yg = Y.cpu().numpy()[np.ix_(toks, rows)]
        worst = max(worst, check_close(Yg, Yref, B, f"{w.name} {lin.name}"))
    return worst


def test_single_linear():
    print("max err/sum|wx|:", _run_workload(wl.single_linear()))


@pytest.mark.parametrize("fmt", [wl.Q8_0, wl.Q4_0, wl.Q6_0])
def test_gemma2b_decode(fmt):
    print("max err/sum|wx|:", _run_workload(wl.gemma2b_decode(fmt)))


def test_action_expert_denoise():
    print("max err/sum|wx|:", _run_workload(wl.action_expert_denoise()))


@pytest.mark.parametrize("fmt", [wl.Q8_0, wl.Q4_0, wl.Q6_0])
def test_gemma2b_prefill(fmt):
    toks = np.unique(np.r_[0, 255, 256, 767, 768, 815, np.random.default_rng(1).choice(816, 10)])
    print("max err/sum|wx|:", _run_workload(wl.gemma2b_prefill(fmt), layers=4, token_sample=toks))


@pytest.mark.parametrize("fmt", [wl.Q8_0, wl.Q4_0])
def test_vit_tower(fmt):
    toks = np.unique(np.r_[0, 255, 256, 767, np.random.default_rng(2).choice(768, 10)])
    print("max err/sum|wx|:", _run_workload(wl.vit_tower(fmt), layers=6, token_sample=toks))


@pytest.mark.parametrize("M", [1, 280])
def test_llama7b(M):
    toks = None if M == 1 else np.unique(np.r_[0, 143, 144, 279, np.random.default_rng(3).choice(280, 8)])
    print("max err/sum|wx|:", _run_workload(wl.llama7b(M), layers=4 if M > 1 else None,
                                            token_sample=toks))
