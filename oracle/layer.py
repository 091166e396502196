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
derived from the fp32 arithmetic the kernels use and their final bf16 rounding; the
derivations are in each function's docstring.
"""
from __future__ import annotations

import numpy as np

U32 = 2.0 ** -24   # fp32 unit roundoff
U_BF16 = 2.0 ** -8  # bf16 unit roundoff (8 significant bits)


def rmsnorm_reference(x, gamma, eps: float):
    """x: fp32 [M][D] (the residual stream); gamma: fp32 [D]. Returns (ref, bound), [M][D].

    Bound: the kernel sums the D squares in fp32 in any order (relative error <= (D - 1) u),
    divides by D, adds eps, takes a correctly rounded square root and reciprocal, and
    multiplies by x then gamma (four more roundings), so its fp32 value v has relative error
    below (D + 16) u; the bf16 store adds at most 2^-8 |v|."""
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

    Bound: the kernel forms each angle as an exact two-float product of the position and
    a two-float inverse frequency (error ~|angle| 2^-46), takes its cosine and sine with
    fp32 sincosf (within 2 ulp) corrected to first order by the angle's low part, so each
    is within 2^-21 of the exact value; then x_a cos - x_b sin (or x_b cos + x_a sin) in
    fp32, two products and one add, at most 3 u (|x_a| + |x_b|) more; the bf16 store adds
    2^-8 of the value."""
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

    Bound, per query m and head h with n = n0 + n1 keys. The kernel computes the scores and
    the weighted values on tensor cores, whose fp32 accumulation need not round to nearest:
    each addition is taken as an error of up to 2 u. So each score carries an error
    Delta <= 2 (d + 2) u scale sum_i |q_i k_i| (exact bf16 products, d - 1 adds, the scale);
    each exponential an error E <= 2^-21 + u |s_j - s_max| (expf within 2 ulp, plus its
    argument's rounding), applied once per key block and once per rescale of the running
    sums (at most n / 32 + 4 times); each weight enters the value product as a bf16 hi + lo
    pair, within 2^-16 of it. A relative perturbation rho = Delta + E (n / 32 + 4) + 2^-16
    of every unnormalised weight moves the normalised output by at most
    2.2 rho sum_j p_j |v_j|; the sums of the weights and of the weighted values add
    4 (n + 8) u sum_j p_j |v_j|; the bf16 store adds 2^-8 |o|."""
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
        E = 2.0 ** -21 + U32 * (smax - s).max(axis=1, keepdims=True)
        rho = delta + E * (n / 32.0 + 4.0) + 2.0 ** -16
        spread = p @ np.abs(v)                                   # sum_j p_j |v_j|, [M][d]
        b = (2.2 * rho + 4.0 * (n + 8) * U32) * spread
        bound[:, h * head_dim:(h + 1) * head_dim] = b + U_BF16 * (np.abs(o) + b) + 1e-38
    return ref, bound
