"""Helpers shared by the GPU parity tests: feed one seeded input to both the CUDA
path (through the C ABI) and the CPU oracle, and compare."""
import numpy as np
import torch

import oracle
import paper_2607_02501_gb300 as emb
from workloads import activation_bits_np, weight_np


def to_dev_bf16(bits: np.ndarray) -> torch.Tensor:
    """bf16 device tensor holding exactly the given bit patterns."""
    t = torch.from_numpy(np.ascontiguousarray(bits).view(np.int16))
    return t.cuda().view(torch.bfloat16)


def bits_of(x: torch.Tensor) -> np.ndarray:
    return x.contiguous().view(torch.int16).cpu().numpy().view(np.uint16)


def gpu_quantize(fmt: int, W_host: np.ndarray) -> torch.Tensor:
    Wd = torch.from_numpy(np.ascontiguousarray(W_host, dtype=np.float32)).cuda()
    return emb.quantize(fmt, Wd)


def check_close(Y: np.ndarray, Yref: np.ndarray, B: np.ndarray, what: str = "") -> float:
    """|Y - Yref| <= B elementwise (B = 1e-3 sum|w x| + 1e-6); returns the largest
    error / sum|w x| ratio seen (for reporting)."""
    Y = np.asarray(Y, dtype=np.float64)
    err = np.abs(Y - Yref)
    assert np.isfinite(Y).all(), f"{what}: non-finite output"
    bad = err > B
    if bad.any():
        idx = np.argwhere(bad)[:5]
        raise AssertionError(f"{what}: {int(bad.sum())} of {bad.size} outside tolerance, "
                             f"first {idx.tolist()} err={err[bad][:5]} bound={B[bad][:5]}")
    mag = (B - 1e-6) / 1e-3
    with np.errstate(divide="ignore", invalid="ignore"):
        r = np.where(mag > 0, err / mag, 0.0)
    return float(r.max()) if r.size else 0.0


def run_case(fmt: int, M: int, N: int, K: int, seed: int):
    """Quantise + matmul on the GPU and in the oracle from the same seeded inputs."""
    W = weight_np(N, K, seed)
    Xb = activation_bits_np(M, K, seed + 1)
    img = gpu_quantize(fmt, W)
    X = to_dev_bf16(Xb)
    Y = emb.qmatmul(fmt, img, X, N)
    torch.cuda.synchronize()
    ref_img = oracle.quantize(fmt, W)
    Yref, B = oracle.qmatmul(fmt, ref_img, Xb, N, K)
    return Y.cpu().numpy(), Yref, B, img, ref_img


def layout_rows(fmt: int, img: torch.Tensor, N: int, K: int, rows) -> np.ndarray:
    """The packed image restricted to the given rows (codes rows, Q6_0 high-bit rows,
    scale rows), laid out as the image of that row subset (what the oracle produces for
    W[rows])."""
    rows = torch.as_tensor(np.asarray(rows), device=img.device, dtype=torch.long)
    n = rows.numel()
    rb = K if fmt == emb.EMB_Q8_0 else K // 2
    hb = K // 4 if fmt == emb.EMB_Q6_0 else 0
    r256 = lambda v: (v + 255) // 256 * 256
    codes = img[:N * rb].view(N, rb)[rows]
    hoff, sub_hoff = r256(N * rb), r256(n * rb)
    off = r256(hoff + N * hb) if hb else r256(N * rb)
    sub_off = r256(sub_hoff + n * hb) if hb else r256(n * rb)
    ldS = (K // 32 + 7) // 8 * 8
    scales = img[off:off + N * ldS * 2].view(N, ldS * 2)[rows]
    out = torch.zeros(sub_off + n * ldS * 2, dtype=torch.uint8, device=img.device)
    out[:n * rb] = codes.reshape(-1)
    if hb:
        out[sub_hoff:sub_hoff + n * hb] = img[hoff:hoff + N * hb].view(N, hb)[rows].reshape(-1)
    out[sub_off:] = scales.reshape(-1)
    return out.cpu().numpy()


def sample_rows(N: int, count: int, seed: int) -> np.ndarray:
    rng = np.random.default_rng(seed)
    rows = set([0, N - 1]) | set(rng.choice(N, size=min(count, N), replace=False).tolist())
    return np.array(sorted(rows), dtype=np.int64)
