"""Pins for the oracle's layer references (RMSNorm, rotary embedding, attention): closed
forms, printed textbook values, invariants of the definitions, brute force on tiny inputs,
and each bound against an fp32 model of the computation it bounds. CPU only."""
import math

import numpy as np
import pytest

import oracle

RNG = np.random.default_rng(20260712)


def _bf16(x):
    return oracle.bf16_round(np.asarray(x, dtype=np.float64))


# ------------------------------------------------------------------ RMSNorm

def test_rmsnorm_one_hot_closed_form():
    # x = 3 e_4 over D = 9: mean(x^2) = 1, so y = 3 e_4 (times gamma_4)
    x = np.zeros((1, 9), dtype=np.float32)
    x[0, 4] = 3.0
    gamma = np.full(9, 0.5, dtype=np.float32)
    y, _ = oracle.rmsnorm_reference(x, gamma, 0.0)
    expect = np.zeros((1, 9))
    expect[0, 4] = 1.5
    assert np.array_equal(y, expect)


def test_rmsnorm_constant_row_gives_sign_times_gamma():
    gamma = RNG.standard_normal(64).astype(np.float32)
    for c in (-2.5, 0.125, 7.0):
        y, _ = oracle.rmsnorm_reference(np.full((1, 64), c, dtype=np.float32), gamma, 0.0)
        assert np.allclose(y[0], np.sign(c) * gamma, rtol=1e-15, atol=0)


def test_rmsnorm_scale_invariance_unit_rms_and_gamma():
    x = RNG.standard_normal((5, 96)).astype(np.float32)
    ones = np.ones(96, dtype=np.float32)
    y1, _ = oracle.rmsnorm_reference(x, ones, 0.0)
    y2, _ = oracle.rmsnorm_reference(x * np.float32(8.0), ones, 0.0)
    assert np.allclose(y1, y2, rtol=1e-14, atol=0)
    assert np.allclose(np.mean(y1 * y1, axis=1), 1.0, rtol=1e-14)
    g = RNG.standard_normal(96).astype(np.float32)
    yg, _ = oracle.rmsnorm_reference(x, g, 0.0)
    assert np.allclose(yg, y1 * g.astype(np.float64)[None, :], rtol=1e-14, atol=1e-300)


def test_rmsnorm_eps_enters_under_the_root():
    # D = 4, x = (1, 1, 1, 1), eps = 3: y = 1 / sqrt(1 + 3) = 0.5
    y, _ = oracle.rmsnorm_reference(np.ones((1, 4), dtype=np.float32), np.ones(4, dtype=np.float32), 3.0)
    assert np.array_equal(y, np.full((1, 4), 0.5))
    z, _ = oracle.rmsnorm_reference(np.zeros((1, 4), dtype=np.float32), np.ones(4, dtype=np.float32), 1e-6)
    assert np.array_equal(z, np.zeros((1, 4)))


def test_rmsnorm_bound_covers_an_fp32_model():
    for D in (64, 1024, 2048):
        x = (RNG.standard_normal((8, D)) * 3).astype(np.float32)
        g = (1.0 + 0.1 * RNG.standard_normal(D)).astype(np.float32)
        ref, bound = oracle.rmsnorm_reference(x, g, 1e-6)
        s = np.float32(0)
        ys = []
        for r in range(8):
            s = np.float32(0)
            for v in x[r]:                      # sequential fp32 sum of squares
                s = np.float32(s + np.float32(v * v))
            inv = np.float32(1.0) / np.sqrt(np.float32(s / np.float32(D) + np.float32(1e-6)))
            ys.append(_bf16((x[r] * inv).astype(np.float32) * g))
        y = np.array(ys)
        assert (np.abs(y - ref) <= bound).all()
        assert (np.abs(y - ref) > 0).any()     # the model does round


# ------------------------------------------------------------------ rotary embedding

def test_rope_hand_example():
    # d = 4: pairs (0, 2) with inverse frequency 1 and (1, 3) with 10000^(-1/2) = 0.01;
    # position 1. cos 1, sin 1, cos 0.01, sin 0.01 as printed in tables.
    y, _ = oracle.rope_reference(np.array([[1.0, 0.0, 0.0, 0.0]]), 1, 4, 1, 10000.0)
    assert np.allclose(y, [[0.5403023058681398, 0.0, 0.8414709848078965, 0.0]], rtol=0, atol=1e-15)
    y, _ = oracle.rope_reference(np.array([[0.0, 1.0, 0.0, 0.0]]), 1, 4, 1, 10000.0)
    assert np.allclose(y, [[0.0, 0.9999500004166653, 0.0, 0.009999833334166664]], rtol=0, atol=1e-15)
    # the second element of a pair rotates the other way into the first
    y, _ = oracle.rope_reference(np.array([[0.0, 0.0, 1.0, 0.0]]), 1, 4, 1, 10000.0)
    assert np.allclose(y, [[-0.8414709848078965, 0.0, 0.5403023058681398, 0.0]], rtol=0, atol=1e-15)


def test_rope_position_zero_is_identity_and_pairs_keep_their_norm():
    x = _bf16(RNG.standard_normal((1, 2 * 64)))
    y, _ = oracle.rope_reference(x, 2, 64, 0, 10000.0)
    assert np.array_equal(y, x)
    x = _bf16(RNG.standard_normal((7, 3 * 128)))
    y, _ = oracle.rope_reference(x, 3, 128, 100, 10000.0)
    for h in range(3):
        a, b = x[:, h * 128:h * 128 + 64], x[:, h * 128 + 64:(h + 1) * 128]
        ya, yb = y[:, h * 128:h * 128 + 64], y[:, h * 128 + 64:(h + 1) * 128]
        assert np.allclose(ya * ya + yb * yb, a * a + b * b, rtol=1e-13, atol=1e-300)


def test_rope_scores_depend_on_relative_position_only():
    q = _bf16(RNG.standard_normal((1, 128)))
    k = _bf16(RNG.standard_normal((1, 128)))
    def score(pq, pk):
        a = oracle.rope_reference(q, 1, 128, pq, 10000.0)[0][0]
        b = oracle.rope_reference(k, 1, 128, pk, 10000.0)[0][0]
        return float(a @ b)
    assert math.isclose(score(5, 2), score(813, 810), rel_tol=1e-11)
    assert not math.isclose(score(5, 2), score(5, 3), rel_tol=1e-6)


def test_rope_rotations_compose_and_heads_are_independent():
    x = _bf16(RNG.standard_normal((1, 64)))
    a, _ = oracle.rope_reference(x, 1, 64, 30, 500.0)
    ab, _ = oracle.rope_reference(a, 1, 64, 12, 500.0)
    direct, _ = oracle.rope_reference(x, 1, 64, 42, 500.0)
    assert np.allclose(ab, direct, rtol=0, atol=1e-12)
    two, _ = oracle.rope_reference(np.concatenate([x, x], axis=1), 2, 64, 9, 500.0)
    one, _ = oracle.rope_reference(x, 1, 64, 9, 500.0)
    assert np.array_equal(two[:, :64], one) and np.array_equal(two[:, 64:], one)
    # row m sits at position pos0 + m
    rows, _ = oracle.rope_reference(np.concatenate([x, x]), 1, 64, 9, 500.0)
    nxt, _ = oracle.rope_reference(x, 1, 64, 10, 500.0)
    assert np.array_equal(rows[1:], nxt)


def test_rope_bound_covers_an_fp32_model():
    H, d, M, pos0 = 8, 128, 50, 816
    x = _bf16(RNG.standard_normal((M, H * d)) * 2)
    ref, bound = oracle.rope_reference(x, H, d, pos0, 10000.0)
    half = d // 2
    inv = 10000.0 ** (-2.0 * np.arange(half) / d)
    ang = (pos0 + np.arange(M))[:, None] * inv
    c, s = np.cos(ang).astype(np.float32), np.sin(ang).astype(np.float32)
    y = np.empty_like(x)
    x32 = x.astype(np.float32)
    for h in range(H):
        a, b = x32[:, h * d:h * d + half], x32[:, h * d + half:(h + 1) * d]
        y[:, h * d:h * d + half] = _bf16((a * c).astype(np.float32) - (b * s).astype(np.float32))
        y[:, h * d + half:(h + 1) * d] = _bf16((b * c).astype(np.float32) + (a * s).astype(np.float32))
    assert (np.abs(y - ref) <= bound).all()


# ------------------------------------------------------------------ attention

def _rand(shape, s=1.0):
    return _bf16(RNG.standard_normal(shape) * s)


def test_attention_one_key_returns_its_value():
    q, k, v = _rand((3, 2 * 8)), _rand((1, 8)), _rand((1, 8))
    o, _ = oracle.attention_reference(q, k, v, np.zeros((0, 8)), np.zeros((0, 8)), 2, 1, 8, 0.3)
    assert np.allclose(o, np.tile(v, (3, 2)), rtol=1e-15, atol=0)


def test_attention_identical_keys_average_the_values():
    k = np.tile(_rand((1, 16)), (5, 1))
    v = _rand((5, 16))
    o, _ = oracle.attention_reference(_rand((2, 16)), k[:3], v[:3], k[3:], v[3:], 1, 1, 16, 0.25)
    assert np.allclose(o, np.tile(v.mean(axis=0), (2, 1)), rtol=1e-14, atol=1e-16)


def test_attention_brute_force_tiny():
    """Python loops and math.exp on 2 queries, 2 heads sharing 1 kv head, d = 4, 2 + 1 keys."""
    H, Hk, d = 2, 1, 4
    Q, K0, V0, K1, V1 = _rand((2, H * d)), _rand((2, d)), _rand((2, d)), _rand((1, d)), _rand((1, d))
    scale = 0.5
    o, _ = oracle.attention_reference(Q, K0, V0, K1, V1, H, Hk, d, scale)
    keys = [list(K0[0]), list(K0[1]), list(K1[0])]
    vals = [list(V0[0]), list(V0[1]), list(V1[0])]
    for m in range(2):
        for h in range(H):
            q = [float(t) for t in Q[m, h * d:(h + 1) * d]]
            sc = [scale * sum(qi * ki for qi, ki in zip(q, kk)) for kk in keys]
            mx = max(sc)
            w = [math.exp(t - mx) for t in sc]
            z = sum(w)
            for i in range(d):
                expect = sum(wj * vv[i] for wj, vv in zip(w, vals)) / z
                assert math.isclose(o[m, h * d + i], expect, rel_tol=1e-13, abs_tol=1e-15)


def test_attention_grouped_heads_read_their_kv_head():
    H, Hk, d, n = 4, 2, 8, 6
    K = _rand((n, Hk * d))
    V = np.concatenate([np.full((n, d), 1.0), np.full((n, d), 2.0)], axis=1)
    o, _ = oracle.attention_reference(_rand((3, H * d)), K, V, np.zeros((0, Hk * d)),
                                      np.zeros((0, Hk * d)), H, Hk, d, 0.4)
    assert np.allclose(o[:, :2 * d], 1.0, rtol=1e-15) and np.allclose(o[:, 2 * d:], 2.0, rtol=1e-15)


def test_attention_prefix_chunk_split_and_key_order_do_not_matter():
    H, Hk, d = 4, 1, 16
    Q, K, V = _rand((5, H * d)), _rand((11, d)), _rand((11, d))
    a, _ = oracle.attention_reference(Q, K[:7], V[:7], K[7:], V[7:], H, Hk, d, 0.25)
    b, _ = oracle.attention_reference(Q, K, V, K[:0], V[:0], H, Hk, d, 0.25)
    perm = RNG.permutation(11)
    c, _ = oracle.attention_reference(Q, K[perm[:4]], V[perm[:4]], K[perm[4:]], V[perm[4:]], H, Hk, d, 0.25)
    assert np.allclose(a, b, rtol=1e-14, atol=1e-16) and np.allclose(a, c, rtol=1e-13, atol=1e-15)


def test_attention_large_gain_selects_the_aligned_key():
    d = 8
    K = np.eye(d)[:5] * 4.0
    V = _rand((5, d))
    q = np.zeros((1, d))
    q[0, 3] = 4.0
    o, _ = oracle.attention_reference(q, K, V, K[:0], V[:0], 1, 1, d, 10.0)
    assert np.allclose(o[0], V[3], rtol=0, atol=1e-60)


def _fp32_attention_model(Q, K, V, H, Hk, d, scale, splits, block):
    """What the kernel does: per split of the keys, blocks of `block` keys with an online
    softmax in fp32; the splits combined at the end; bf16 store."""
    f = np.float32
    M, n = Q.shape[0], K.shape[0]
    out = np.empty((M, H * d))
    group = H // Hk
    for h in range(H):
        g = h // group
        for m in range(M):
            q = Q[m, h * d:(h + 1) * d].astype(f)
            parts = []
            for sp in range(splits):
                lo, hi = sp * n // splits, (sp + 1) * n // splits
                mx, l, o = f(-np.inf), f(0), np.zeros(d, dtype=f)
                for b0 in range(lo, hi, block):
                    kb = K[b0:min(hi, b0 + block), g * d:(g + 1) * d].astype(f)
                    vb = V[b0:min(hi, b0 + block), g * d:(g + 1) * d].astype(f)
                    s = (kb @ q).astype(f) * f(scale)
                    new = max(mx, s.max())
                    r = np.exp(f(mx - new)) if np.isfinite(mx) else f(0)
                    p = np.exp((s - new).astype(f)).astype(f)
                    l = f(l * r + p.sum(dtype=f))
                    o = (o * r + (p[:, None] * vb).sum(axis=0, dtype=f)).astype(f)
                    mx = new
                parts.append((mx, l, o))
            M_ = max(pm for pm, _, _ in parts if np.isfinite(pm))
            L = f(0)
            O = np.zeros(d, dtype=f)
            for pm, pl, po in parts:
                if np.isfinite(pm):
                    w = np.exp(f(pm - M_))
                    L = f(L + pl * w)
                    O = (O + po * w).astype(f)
            out[m, h * d:(h + 1) * d] = _bf16((O / L).astype(f))
    return out


@pytest.mark.parametrize("n0,n1,splits,block", [(816, 50, 8, 64), (816, 50, 1, 1), (816, 50, 16, 7),
                                                (100, 7, 2, 64), (100, 7, 3, 1), (5, 0, 1, 64)])
def test_attention_bound_covers_an_fp32_model(n0, n1, splits, block):
    """The bound holds for an fp32 online softmax whatever its key splits and key blocks
    (down to a rescale after every key): it depends on the sizes and inputs only."""
    H, Hk, d = 8, 1, 128
    M = 3
    Q, K0, V0, K1, V1 = (_rand((M, H * d)), _rand((n0, Hk * d)), _rand((n0, Hk * d)),
                         _rand((n1, Hk * d)), _rand((n1, Hk * d)))
    scale = 1.0 / math.sqrt(d)
    ref, bound = oracle.attention_reference(Q, K0, V0, K1, V1, H, Hk, d, scale)
    model = _fp32_attention_model(Q, np.concatenate([K0, K1]), np.concatenate([V0, V1]),
                                  H, Hk, d, scale, splits, block)
    assert (np.abs(model - ref) <= bound).all()
