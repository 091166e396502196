"""The layer steps around the linears against the oracle: RMSNorm, rotary embedding and
grouped-head attention over a prefix cache plus the chunk's own keys, element by element on
seeded inputs (ragged and maximum sizes, grouped, multi-query and per-head key/value heads,
one or many key splits); then one whole action-expert layer (norm, q/k/v, rotary, attention,
o + residual, norm, GeGLU gate/up, down + residual) recorded as one chain and replayed, each
step checked against the oracle from the bits the GPU produced before it."""
import math

import numpy as np
import pytest
import torch

import oracle
import paper_2607_02501_gb300 as emb
from tests.gpu_util import bits_of
from workloads import activation_bits_np, weight_np

pytestmark = pytest.mark.gpu


def _bf16_dev(a):
    return torch.from_numpy(np.asarray(a, dtype=np.float32)).to(torch.bfloat16).cuda()


def _vals(t):
    return t.float().cpu().numpy().astype(np.float64)


def _check(out, ref, bound, what):
    assert np.isfinite(out).all(), f"{what}: non-finite output"
    bad = np.abs(out - ref) > bound
    assert not bad.any(), (f"{what}: {int(bad.sum())} of {bad.size} outside, first "
                           f"{np.argwhere(bad)[:4].tolist()} err={np.abs(out - ref)[bad][:4]} "
                           f"bound={bound[bad][:4]}")


@pytest.mark.parametrize("M,D", [(1, 1024), (50, 1024), (816, 2048), (3, 8), (7, 4104), (2, 65536)])
def test_rmsnorm_parity(cuda_device, M, D):
    rng = np.random.default_rng(M * 7 + D)
    x = (rng.standard_normal((M, D)) * 3).astype(np.float32)
    g = (1.0 + 0.1 * rng.standard_normal(D)).astype(np.float32)
    y = torch.full((M, D), float("nan"), dtype=torch.bfloat16, device="cuda")
    emb.emb_rmsnorm(torch.from_numpy(x).cuda(), torch.from_numpy(g).cuda(), y, 1e-6)
    torch.cuda.synchronize()
    ref, bound = oracle.rmsnorm_reference(x, g, 1e-6)
    _check(_vals(y), ref, bound, f"rmsnorm M={M} D={D}")


@pytest.mark.parametrize("M,H,d,pos0,base", [(50, 8, 128, 816, 10000.0), (1, 1, 64, 0, 10000.0),
                                             (816, 8, 256, 0, 10000.0), (3, 5, 2, 7, 500.0),
                                             (50, 1, 128, 816, 10000.0), (9, 3, 64, 100000, 1e6)])
def test_rope_parity(cuda_device, M, H, d, pos0, base):
    rng = np.random.default_rng(M + H * 3 + d)
    xb = oracle.bf16_round(rng.standard_normal((M, H * d)) * 2)
    x = _bf16_dev(xb)
    emb.emb_rope(x, H, d, pos0, base)
    torch.cuda.synchronize()
    ref, bound = oracle.rope_reference(xb, H, d, pos0, base)
    _check(_vals(x), ref, bound, f"rope M={M} H={H} d={d} pos0={pos0}")


@pytest.mark.parametrize("M,H,Hk,d", [(50, 8, 1, 128), (7, 3, 5, 64), (1, 1, 1, 2)])
def test_rope_qk_is_two_ropes_in_one_launch(cuda_device, M, H, Hk, d):
    rng = np.random.default_rng(M + H + Hk + d)
    qb = oracle.bf16_round(rng.standard_normal((M, H * d)))
    kb = oracle.bf16_round(rng.standard_normal((M, Hk * d)))
    q1, k1, q2, k2 = _bf16_dev(qb), _bf16_dev(kb), _bf16_dev(qb), _bf16_dev(kb)
    emb.emb_rope_qk(q1, H, k1, Hk, d, 816, 10000.0)
    emb.emb_rope(q2, H, d, 816, 10000.0)
    emb.emb_rope(k2, Hk, d, 816, 10000.0)
    torch.cuda.synchronize()
    assert torch.equal(q1.view(torch.int16), q2.view(torch.int16))
    assert torch.equal(k1.view(torch.int16), k2.view(torch.int16))
    for t, xb, heads in ((q1, qb, H), (k1, kb, Hk)):
        ref, bound = oracle.rope_reference(xb, heads, d, 816, 10000.0)
        _check(_vals(t), ref, bound, f"rope_qk heads={heads}")


# (M, H, Hk, d, n0, n1): the action expert over the 816-token prefix; grouped heads with
# two kv heads and no cache; 16 heads of one kv head (two CTAs of 8 heads); one kv head per
# query head; a single key; many keys at one query (eight key splits); a ragged last tile
ATTN = [(50, 8, 1, 128, 816, 50), (3, 4, 2, 64, 0, 5), (1, 16, 1, 128, 100, 0),
        (7, 8, 8, 64, 130, 1), (2, 1, 1, 128, 1, 0), (1, 8, 1, 128, 4000, 3),
        (5, 2, 1, 64, 63, 66)]


def _attn_inputs(M, H, Hk, d, n0, n1, seed):
    rng = np.random.default_rng(seed)
    r = lambda *s: oracle.bf16_round(rng.standard_normal(s))
    return r(M, H * d), r(n0, Hk * d), r(n0, Hk * d), r(n1, Hk * d), r(n1, Hk * d)


def _run_attention(Qb, K0b, V0b, K1b, V1b, H, Hk, d, scale):
    dev = lambda a: _bf16_dev(a) if a.shape[0] else None
    Q, K0, V0, K1, V1 = _bf16_dev(Qb), dev(K0b), dev(V0b), dev(K1b), dev(V1b)
    O = torch.full((Qb.shape[0], H * d), float("nan"), dtype=torch.bfloat16, device="cuda")
    emb.emb_attention(Q, K0, V0, K1, V1, O, H, Hk, d, scale)
    torch.cuda.synchronize()
    return O


@pytest.mark.parametrize("M,H,Hk,d,n0,n1", ATTN)
def test_attention_parity(cuda_device, M, H, Hk, d, n0, n1):
    ins = _attn_inputs(M, H, Hk, d, n0, n1, M + H + n0 + n1)
    scale = 1.0 / math.sqrt(d)
    O = _run_attention(*ins, H, Hk, d, scale)
    ref, bound = oracle.attention_reference(*ins, H, Hk, d, scale)
    _check(_vals(O), ref, bound, f"attention M={M} H={H} Hk={Hk} d={d} n={n0}+{n1}")
    assert emb.emb_device_status() == emb.EMB_OK


def test_attention_is_deterministic_and_ignores_the_split_of_cache_and_chunk(cuda_device):
    M, H, Hk, d = 50, 8, 1, 128
    Qb, K0b, V0b, K1b, V1b = _attn_inputs(M, H, Hk, d, 816, 50, 3)
    a = _run_attention(Qb, K0b, V0b, K1b, V1b, H, Hk, d, 0.0883883)
    b = _run_attention(Qb, K0b, V0b, K1b, V1b, H, Hk, d, 0.0883883)
    assert torch.equal(a.view(torch.int16), b.view(torch.int16))
    # the same keys given as one list: the same keys in the same order, same tiles and splits
    c = _run_attention(Qb, np.concatenate([K0b, K1b]), np.concatenate([V0b, V1b]),
                       K1b[:0], V1b[:0], H, Hk, d, 0.0883883)
    assert torch.equal(a.view(torch.int16), c.view(torch.int16))


def test_action_expert_layer_recorded(cuda_device):
    """One action-expert layer at M = 50 over an 816-token prefix cache, as one recorded
    chain: h = norm(r); q, k, v = W_qkv h (bf16); rotary on q, k at positions 816..865;
    a = attention(q | prefix k, v + chunk k, v); r += W_o a; h2 = norm(r);
    g = GeGLU(W_gu h2) (interleaved rows); r += W_d g. Checked step by step."""
    M, D, H, Hk, d, F, P = 50, 1024, 8, 1, 128, 4096, 816
    fmt = emb.EMB_Q8_0
    rng = np.random.default_rng(77)
    Ws = {"q": weight_np(H * d, D, 1), "k": weight_np(Hk * d, D, 2), "v": weight_np(Hk * d, D, 3),
          "o": weight_np(D, H * d, 4), "gu": weight_np(2 * F, D, 5), "d": weight_np(D, F, 6)}
    imgs = {k: emb.quantize(fmt, torch.from_numpy(w).cuda()) for k, w in Ws.items()}
    g1 = (1.0 + 0.1 * rng.standard_normal(D)).astype(np.float32)
    g2 = (1.0 + 0.1 * rng.standard_normal(D)).astype(np.float32)
    R0 = (rng.standard_normal((M, D)) * 2).astype(np.float32)
    K0b = oracle.bf16_round(rng.standard_normal((P, Hk * d)))
    V0b = oracle.bf16_round(rng.standard_normal((P, Hk * d)))
    dev = {"g1": torch.from_numpy(g1).cuda(), "g2": torch.from_numpy(g2).cuda(),
           "R": torch.from_numpy(R0.copy()).cuda(), "K0": _bf16_dev(K0b), "V0": _bf16_dev(V0b)}
    bf = lambda *s: torch.full(s, float("nan"), dtype=torch.bfloat16, device="cuda")
    h, q, k, v, a, h2, gg = bf(M, D), bf(M, H * d), bf(M, Hk * d), bf(M, Hk * d), bf(M, H * d), bf(M, D), bf(M, F)
    scale = 1.0 / math.sqrt(d)
    s = torch.cuda.Stream()

    def part1(stream, seq=emb.emb_qlayer_seq, one_rope=False):
        emb.emb_rmsnorm(dev["R"], dev["g1"], h, 1e-6, stream=stream)
        seq([(fmt, imgs["q"], H * d, D, h, q, emb.EMB_EPI_BF16),
                            (fmt, imgs["k"], Hk * d, D, h, k, emb.EMB_EPI_BF16),
                            (fmt, imgs["v"], Hk * d, D, h, v, emb.EMB_EPI_BF16)], M, stream=stream)
        if one_rope:
            emb.emb_rope_qk(q, H, k, Hk, d, P, 10000.0, stream=stream)
        else:
            emb.emb_rope(q, H, d, P, 10000.0, stream=stream)
            emb.emb_rope(k, Hk, d, P, 10000.0, stream=stream)
        emb.emb_attention(q, dev["K0"], dev["V0"], k, v, a, H, Hk, d, scale, stream=stream)
        seq([(fmt, imgs["o"], D, H * d, a, dev["R"], emb.EMB_EPI_ADD)], M, stream=stream)

    def part2(stream, seq=emb.emb_qlayer_seq):
        emb.emb_rmsnorm(dev["R"], dev["g2"], h2, 1e-6, stream=stream)
        seq([(fmt, imgs["gu"], 2 * F, D, h2, gg, emb.EMB_EPI_GEGLU)], M, stream=stream)
        seq([(fmt, imgs["d"], D, F, gg, dev["R"], emb.EMB_EPI_ADD)], M, stream=stream)

    # eager, with the residual kept between the halves, checked step by step against the
    # oracle, each step from the bits the GPU produced before it
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        part1(s)
        s.synchronize()
        R1 = dev["R"].clone()
        part2(s)
    torch.cuda.synchronize()
    assert emb.emb_device_status() == emb.EMB_OK

    ref, bound = oracle.rmsnorm_reference(R0, g1, 1e-6)
    _check(_vals(h), ref, bound, "norm 1")
    hb = bits_of(h)
    Y, B = oracle.qmatmul(fmt, oracle.quantize(fmt, Ws["v"]), hb, Hk * d, D)
    r_, b_ = oracle.epilogue_reference(oracle.EPI_BF16, Y, B)
    _check(_vals(v), r_, b_, "v projection")
    # q and k were rotated in place: the rotation of the projection's bf16 result, where a
    # bf16 input within pre_b of the reference moves each rotated element by at most the
    # sum of its pair's input errors
    half = d // 2
    for name, buf, heads in (("q", q, H), ("k", k, Hk)):
        Y, B = oracle.qmatmul(fmt, oracle.quantize(fmt, Ws[name]), hb, heads * d, D)
        pre, pre_b = oracle.epilogue_reference(oracle.EPI_BF16, Y, B)
        rot, rot_b = oracle.rope_reference(pre, heads, d, P, 10000.0)
        spread = np.empty_like(pre_b)
        for hh in range(heads):
            e = pre_b[:, hh * d:hh * d + half] + pre_b[:, hh * d + half:(hh + 1) * d]
            spread[:, hh * d:hh * d + half] = e
            spread[:, hh * d + half:(hh + 1) * d] = e
        _check(_vals(buf), rot, rot_b + spread * (1 + 2.0 ** -8), f"{name} projection + rotary")
    ref, bound = oracle.attention_reference(_vals(q), K0b, V0b, _vals(k), _vals(v), H, Hk, d, scale)
    _check(_vals(a), ref, bound, "attention")
    Y, B = oracle.qmatmul(fmt, oracle.quantize(fmt, Ws["o"]), bits_of(a), D, H * d)
    r_, b_ = oracle.epilogue_reference(oracle.EPI_ADD, Y, B, R0)
    R1n = R1.cpu().numpy()
    _check(R1n.astype(np.float64), r_, b_, "o + residual")
    ref, bound = oracle.rmsnorm_reference(R1n, g2, 1e-6)
    _check(_vals(h2), ref, bound, "norm 2")
    Y, B = oracle.qmatmul(fmt, oracle.quantize(fmt, Ws["gu"]), bits_of(h2), 2 * F, D)
    r_, b_ = oracle.epilogue_reference(oracle.EPI_GEGLU, Y, B)
    _check(_vals(gg), r_, b_, "gate/up GeGLU")
    Y, B = oracle.qmatmul(fmt, oracle.quantize(fmt, Ws["d"]), bits_of(gg), D, F)
    r_, b_ = oracle.epilogue_reference(oracle.EPI_ADD, Y, B, R1n)
    _check(dev["R"].cpu().numpy().astype(np.float64), r_, b_, "down + residual")

    # the whole layer recorded as one chain, its linears through emb_qlayer_seq_chained (the
    # first launch of each call overlapping the layer step before it): nothing runs while
    # recording, and a replay gives the eager run's bits
    eager = [t.clone() for t in (h, q, k, v, a, h2, gg, dev["R"])]
    dev["R"].copy_(torch.from_numpy(R0))
    for t in (h, q, k, v, a, h2, gg):
        t.fill_(float("nan"))
    torch.cuda.synchronize()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        rec = emb.Recording(s)
        with rec:
            part1(s, emb.emb_qlayer_seq_chained, one_rope=True)
            part2(s, emb.emb_qlayer_seq_chained)
    torch.cuda.synchronize()
    assert torch.isnan(h.float()).all() and torch.equal(dev["R"].cpu(), torch.from_numpy(R0))
    for _ in range(2):
        dev["R"].copy_(torch.from_numpy(R0))
        torch.cuda.synchronize()
        rec.launch(s)
        torch.cuda.synchronize()
        for t, e in zip((h, q, k, v, a, h2, gg, dev["R"]), eager):
            assert torch.equal(t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32),
                               e.view(torch.int16) if e.dtype == torch.bfloat16 else e.view(torch.int32))
    rec.close()
    assert emb.emb_device_status() == emb.EMB_OK
