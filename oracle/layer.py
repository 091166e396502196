"""Oracle for the non-matmul steps of one transformer layer of the shared backbone and the
action expert (TEST INFRASTRUCTURE ONLY; same import rules as the rest of ``oracle``).

The paper runs every model family through one shared backbone execution path (Section 3.2)
but defines none of its operators; these are the standard published definitions, written
out plainly in fp64 (numpy; a matrix product is used as a step):

* RMSNorm (Zhang and Sennrich, 2019): y = x / sqrt(mean(x^2) + eps) * gamma, per token.
* Rotary position embedding (Su et al., RoFormer, 2021), rotate-half pairing: in every head,
  element i and element i + d/2 (i < d/2) form a pair rotated by the angle
  pos * base^(-2i/d); the first output is x_i cos - x_(i+d/2) sin, the second
  x_(i+d/2) cos + x_i sin.
* Scaled dot-product attention (Vaswani et al., 2017) with grouped key/value heads: query
  head h reads key/value head h // (H / Hk); the keys are the prefix cache followed by the
  chunk's own keys, all visible to every query (no mask); weights softmax(scale * q.k).

Every function returns the fp64 reference and a per-element bound on |GPU - reference|
that any correct fp32 implementation with a final bf16 rounding meets, whatever its order
of summation, tiling or key splitting: the bounds depend on the operation's sizes and
inputs only. The derivations are in each function's docstring.
"""
from __future__ import annotations

import numpy as np

U32 = 2.0 ** -24   # fp32 unit roundoff
U_BF16 = 2.0 ** -8  # bf16 unit roundoff (8 significant bits)


def rmsnorm_reference(x, gamma, eps: float):
    """x: fp32 [M][D] (the residual stream); gamma: fp32 [D]. Returns (ref, bound), [M][D].

    Bound (any summation order): the D squares summed in fp32 in any order have relative
    error <= (D - 1) u (non-negative terms); the division by D, eps, a correctly rounded
    square root and reciprocal, and the products with x and gamma add a few roundings, so
    the fp32 value v has relative error below (D + 16) u; the bf16 store adds at most
    2^-8 |v|."""
    x = np.asarray(x, dtype=np.float64)
    gamma = np.asarray(gamma, dtype=np.float64)
    D = x.shape[1]
    inv = 1.0 / np.sqrt(np.mean(x * x, axis=1, keepdims=True) + float(np.float32(eps)))
    ref = x * inv * gamma[None, :]
    e = (D + 16) * U32
    bound = (e + U_BF16 * (1.0 + e)) * np.abs(ref) + 1e-38
    return ref, bound


def rope_reference(x, n_heads: int, head_dim: int, pos0: int, base: float):
    """x: bf16 values as floats [M][n_heads * head_dim], token m at position pos0 + m.
    Returns (ref, bound) of the same shape.

    Bound: cosine and sine within 2^-21 of the exact values of the exact angle (an
    implementation must carry the angle to better than fp32, since positions times
    frequencies reach 2^24 radians; this one uses a two-float angle and fp32 sincosf), then
    x_a cos - x_b sin (or x_b cos + x_a sin) in fp32, two products and one add, at most
    4 u (|x_a| + |x_b|) more; the bf16 store adds 2^-8 of the value."""
    x = np.asarray(x, dtype=np.float64)
    M = x.shape[0]
    half = head_dim // 2
    i = np.arange(half, dtype=np.float64)
    inv_freq = float(base) ** (-2.0 * i / head_dim)                     # [half]
    pos = (pos0 + np.arange(M, dtype=np.float64))[:, None]              # [M][1]
    c, s = np.cos(pos * inv_freq), np.sin(pos * inv_freq)               # [M][half]
    ref = np.empty_like(x)
    mag = np.empty_like(x)
    for h in range(n_heads):
        a = x[:, h * head_dim:h * head_dim + half]
        b = x[:, h * head_dim + half:(h + 1) * head_dim]
        ref[:, h * head_dim:h * head_dim + half] = a * c - b * s
        ref[:, h * head_dim + half:(h + 1) * head_dim] = b * c + a * s
        m = np.abs(a) + np.abs(b)
        mag[:, h * head_dim:h * head_dim + half] = m
        mag[:, h * head_dim + half:(h + 1) * head_dim] = m
    e = (2.0 ** -21 + 4 * U32) * mag
    bound = e + U_BF16 * (np.abs(ref) + e) + 1e-38
    return ref, bound


def attention_reference(Q, K0, V0, K1, V1, n_heads: int, n_kv_heads: int, head_dim: int,
                        scale: float):
    """Q: [M][H*d]; K0, V0: [n0][Hk*d] (prefix cache); K1, V1: [n1][Hk*d] (the chunk's own
    keys and values); all bf16 values as floats. Returns (ref, bound), [M][H*d].

    Bound, per query m and head h with n = n0 + n1 keys, for any fp32 implementation whatever
    its key tiles, key splits and order of summation (fp32 additions are taken as errors of
    up to 2 u, since tensor-core accumulation need not round to nearest):
      * each score s_j = scale q.k_j (exact bf16 products, d - 1 additions, the scale) is
        within Delta = 2 (d + 2) u scale max_j sum_i |q_i k_ji| of exact;
      * each unnormalised weight exp(s_j - s_max), with its rescalings by the running
        maximum and its representation in the value product, is within a relative
        2^-10 of exp of the computed score (an allowance that covers expf within a few
        ulp applied up to a few hundred times, and weights carried at bf16 hi + lo or
        better);
      so every unnormalised weight carries a relative perturbation rho = Delta + 2^-10,
    which moves the normalised output by at most 2.2 rho sum_j p_j |v_j|; the sums of the
    weights and of the weighted values add 4 (n + 8) u sum_j p_j |v_j|; the bf16 store adds
    2^-8 |o|."""
    Q = np.asarray(Q, dtype=np.float64)
    K = np.concatenate([np.asarray(K0, dtype=np.float64).reshape(-1, n_kv_heads * head_dim),
                        np.asarray(K1, dtype=np.float64).reshape(-1, n_kv_heads * head_dim)])
    V = np.concatenate([np.asarray(V0, dtype=np.float64).reshape(-1, n_kv_heads * head_dim),
                        np.asarray(V1, dtype=np.float64).reshape(-1, n_kv_heads * head_dim)])
    M, n = Q.shape[0], K.shape[0]
    group = n_heads // n_kv_heads
    ref = np.empty((M, n_heads * head_dim))
    bound = np.empty_like(ref)
    for h in range(n_heads):
        g = h // group
        q = Q[:, h * head_dim:(h + 1) * head_dim]                # [M][d]
        k = K[:, g * head_dim:(g + 1) * head_dim]                # [n][d]
        v = V[:, g * head_dim:(g + 1) * head_dim]                # [n][d]
        s = scale * (q @ k.T)                                    # [M][n]
        smax = s.max(axis=1, keepdims=True)
        w = np.exp(s - smax)
        p = w / w.sum(axis=1, keepdims=True)
        o = p @ v                                                # [M][d]
        ref[:, h * head_dim:(h + 1) * head_dim] = o
        delta = 2 * (head_dim + 2) * U32 * abs(scale) * (np.abs(q) @ np.abs(k).T).max(axis=1, keepdims=True)
        rho = delta + 2.0 ** -10
        spread = p @ np.abs(v)                                   # sum_j p_j |v_j|, [M][d]
        b = (2.2 * rho + 4.0 * (n + 8) * U32) * spread
        bound[:, h * head_dim:(h + 1) * head_dim] = b + U_BF16 * (np.abs(o) + b) + 1e-38
    return ref, bound
