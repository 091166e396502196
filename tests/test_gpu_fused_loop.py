"""The action expert's fused flow-matching loop at its full size (10 denoising steps x 18
layers, M = 50, Q8_0), launched as one chain exactly as the bench builds it: every layer
of the loop keeps one weight image, one activation buffer and one output buffer across
the steps; q/k/v write bf16, gate/up (interleaved rows) writes the GeGLU product in bf16
that down reads as its X, and o and down add into one fp32 residual stream.

Checked against the oracle on sampled outputs: q/k/v and the gated product element by
element, and the residual stream after all 360 adds, with the bound carried add by add
(each add's own matmul bound, its fp32 rounding, and the bound inherited so far)."""
import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
import workloads as wl
from tests.gpu_util import bits_of, sample_rows

pytestmark = pytest.mark.gpu


def _check(out, ref, bound, what):
    out = np.asarray(out, dtype=np.float64)
    assert np.isfinite(out).all(), f"{what}: non-finite output"
    bad = np.abs(out - ref) > bound
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} outside, first "
                           f"{np.argwhere(bad)[:4].tolist()}")


def test_action_expert_fused_loop(cuda_device):
    w = wl.action_expert_fused()
    M, dev = w.M, "cuda"
    resid_n = {lin.N for g in w.groups for lin in g if lin.epilogue == wl.EPI_ADD}
    assert len(resid_n) == 1
    D = resid_n.pop()
    R0 = (np.random.default_rng(11).standard_normal((M, D)) * 2).astype(np.float32)
    R = torch.from_numpy(R0.copy()).to(dev)
    lins, imgs, xs, ys, specs, outs = {}, {}, {}, {}, [], []
    x_of = {}     # layer name -> the buffer it reads
    order = []    # residual-add layers in chain order
    for group in w.groups:
        g0 = group[0]
        if g0.x_from:
            X = outs[-g0.x_from]
        else:
            if g0.name not in xs:
                xs[g0.name] = wl.activation_torch(M, g0.K, wl.activation_seed(g0), device=dev)
            X = xs[g0.name]
        for lin in group:
            if lin.name not in imgs:
                lins[lin.name] = lin
                imgs[lin.name] = emb.quantize(w.fmt, wl.weight_torch(lin, device=dev))
            if lin.epilogue == wl.EPI_ADD:
                Y = R
                order.append(lin.name)
            else:
                if lin.name not in ys:
                    cols = lin.N // 2 if lin.epilogue == wl.EPI_GEGLU else lin.N
                    ys[lin.name] = torch.full((M, cols), float("nan"), dtype=torch.bfloat16,
                                              device=dev)
                Y = ys[lin.name]
            x_of[lin.name] = X
            specs.append((w.fmt, imgs[lin.name], lin.N, lin.K, X, Y, lin.epilogue))
        outs.append(Y)
    assert len(order) == 2 * 18 * 10
    emb.emb_qlayer_seq(specs, M)
    torch.cuda.synchronize()
    assert emb.emb_device_status() == emb.EMB_OK

    def ref_rows(name, rows):
        """Oracle matmul of rows of layer `name` against the bits its X held."""
        lin = lins[name]
        W = wl.weight_torch(lin, device=dev)[torch.as_tensor(rows, device=dev)].cpu().numpy()
        return oracle.qmatmul(w.fmt, oracle.quantize(w.fmt, W), bits_of(x_of[name]), len(rows),
                              lin.K)

    # bf16 outputs and the gated product (identical in every step: same X, same W)
    for name, lin in lins.items():
        if lin.epilogue == wl.EPI_BF16:
            rows = sample_rows(lin.N, 12, lin.seed)
            Yr, B = ref_rows(name, rows)
            ref, bound = oracle.epilogue_reference(wl.EPI_BF16, Yr, B)
            _check(ys[name].float().cpu().numpy()[:, rows], ref, bound, name)
        elif lin.epilogue == wl.EPI_GEGLU:
            cols = sample_rows(lin.N // 2, 12, lin.seed)
            rows = np.stack([2 * cols, 2 * cols + 1], axis=1).reshape(-1)
            Yr, B = ref_rows(name, rows)
            ref, bound = oracle.epilogue_reference(wl.EPI_GEGLU, Yr, B)
            _check(ys[name].float().cpu().numpy()[:, cols], ref, bound, name)

    # the residual stream: R0 plus every o and down output, added in chain order
    cols = sample_rows(D, 16, 5)
    per_layer = {name: ref_rows(name, cols) for name in set(order)}
    ref = R0[:, cols].astype(np.float64)
    bound = np.zeros_like(ref)
    for name in order:
        Yr, B = per_layer[name]
        new_ref, b = oracle.epilogue_reference(wl.EPI_ADD, Yr, B, ref)
        bound = bound * (1.0 + 2.0 ** -23) + b
        ref = new_ref
    _check(R.cpu().numpy()[:, cols], ref, bound, "residual stream after 360 adds")
